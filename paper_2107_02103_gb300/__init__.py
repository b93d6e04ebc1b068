"""GB300 (sm_103a) DP Compress tabulate-fusion library: thin Python binding.

Every function here has the name of a C entry point in include/dp_compress.h
and only marshals arguments: it checks torch tensors (device, dtype,
contiguity, shape), passes their data pointers and the current CUDA stream,
and raises on a non-OK status.  All arithmetic runs in the CUDA kernels of
libdpcompress.so; there is no CPU fallback -- importing this package fails
if the library has not been built (see build.py).

Calls are asynchronous on torch.cuda.current_stream() like any CUDA op.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdpcompress.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'` "
                      "(or paper_2107_02103_gb300/build.py); this package has no CPU fallback")

_lib = ctypes.CDLL(LIB_PATH)

DP_OK, DP_ERR_NULL, DP_ERR_SHAPE, DP_ERR_TABLE_INFO, DP_ERR_CUDA, DP_ERR_UNSUPPORTED = 0, -1, -2, -3, -4, -5
DP_MAX_TYPES, DP_MAX_M1, DP_MAX_WIDTH, DP_MAX_LAYERS = 8, 256, 1024, 8


class dp_table_info(ctypes.Structure):
    """Table range (mirror of the C struct): fine [lower, upper) step stride0, coarse [upper, upper_ext) step stride1."""
    _fields_ = [("lower", ctypes.c_double), ("upper", ctypes.c_double), ("upper_ext", ctypes.c_double),
                ("stride0", ctypes.c_double), ("stride1", ctypes.c_double)]

    def __repr__(self):
        return (f"dp_table_info(lower={self.lower!r}, upper={self.upper!r}, upper_ext={self.upper_ext!r}, "
                f"stride0={self.stride0!r}, stride1={self.stride1!r})")


class dp_tc_plan(ctypes.Structure):
    """Host record of a tensor-core tabulation plan (mirror of the C struct): its device buffer and the
    geometry it was made for."""
    _fields_ = [("data", ctypes.c_void_p), ("bytes", ctypes.c_size_t), ("info", dp_table_info),
                ("nnei", ctypes.c_int32), ("ntypes", ctypes.c_int32), ("M1", ctypes.c_int32)]


DP_TC_REUSE_RUNS = 1


class dp_env_info(ctypes.Structure):
    """Environment-matrix parameters (mirror of the C struct): cutoffs, switch kind, normalisation."""
    _fields_ = [("rcs", ctypes.c_double), ("rc", ctypes.c_double), ("kind", ctypes.c_int32),
                ("mean", ctypes.c_double), ("std", ctypes.c_double), ("std_all", ctypes.c_double)]

    def __repr__(self):
        return (f"dp_env_info(rcs={self.rcs!r}, rc={self.rc!r}, kind={self.kind!r}, mean={self.mean!r}, "
                f"std={self.std!r}, std_all={self.std_all!r})")


def env_info(rcs: float, rc: float, kind: int = 0, norm=None) -> dp_env_info:
    """dp_env_info from cutoffs, switch kind (0 cosine, 1 the paper's quintic) and norm = (mean, std, std_all)."""
    mean, std, std_all = (0.0, 1.0, 1.0) if norm is None else (float(x) for x in norm)
    return dp_env_info(float(rcs), float(rc), int(kind), mean, std, std_all)


class DPError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"[{code}] {msg}")
        self.code = code


_P = ctypes.c_void_p
_I32, _I64, _D = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
_INFO = ctypes.POINTER(dp_table_info)
_ENV = ctypes.POINTER(dp_env_info)
_PLAN = ctypes.POINTER(dp_tc_plan)
_SIGS = {
    "dp_last_error": ([], ctypes.c_char_p),
    "dp_table_info_make": ([_D, _D, _D, _D, _D, _INFO], ctypes.c_int),
    "dp_table_info_sizes": ([_INFO, ctypes.POINTER(_I32), ctypes.POINTER(_I32)], ctypes.c_int),
    "dp_embedding_net_nodes_f64": ([_P, _P, ctypes.c_int, ctypes.c_int, _INFO, _P, _P, _P, _P], ctypes.c_int),
    "dp_table_build_f64": ([_P, _P, _P, ctypes.c_int, ctypes.c_int, _INFO, _P, _P], ctypes.c_int),
    "dp_table_build_f32": ([_P, _P, _P, ctypes.c_int, ctypes.c_int, _INFO, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_f64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, ctypes.c_int,
                                    _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_f32": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, ctypes.c_int,
                                    _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_moments_f64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                            ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_moments_f32": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                            ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_descriptor_f64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                               ctypes.c_int, ctypes.c_int, _P, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_descriptor_f32": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                               ctypes.c_int, ctypes.c_int, _P, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_grad_f64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, ctypes.c_int,
                                     _P, _P, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_grad_f32": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, ctypes.c_int,
                                     _P, _P, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_grad_moments_f64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                             ctypes.c_int, _P, _P, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_grad_moments_f32": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                             ctypes.c_int, _P, _P, _P, _P], ctypes.c_int),
    "dp_profile_begin": ([_P, ctypes.c_int], ctypes.c_int),
    "dp_profile_end": ([], ctypes.c_int),
    "dp_profile_name": ([ctypes.c_int], ctypes.c_char_p),
    "dp_tc_wait_timeouts": ([ctypes.POINTER(ctypes.c_uint)], ctypes.c_int),
    "dp_tabulate_tc_work_bytes": ([_INFO, _I64, ctypes.c_int, ctypes.c_int, ctypes.c_int], ctypes.c_size_t),
    "dp_tabulate_tc_plan_bytes": ([_INFO, ctypes.c_int, ctypes.c_int, ctypes.c_int], ctypes.c_size_t),
    "dp_tabulate_tc_plan_f64": ([_P, _INFO, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P, ctypes.c_size_t, _PLAN,
                                 _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_tc_f64": ([_PLAN, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                       ctypes.c_int, _P, ctypes.c_int, _P, _P, ctypes.c_size_t, _P], ctypes.c_int),
    "dp_tabulate_fusion_grad_tc_f64": ([_PLAN, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                        ctypes.c_int, _P, _P, _P, _P, ctypes.c_size_t, ctypes.c_int, _P],
                                       ctypes.c_int),
    "dp_env_mat_f64": ([_P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, _ENV, _P, _P, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_env_fwd_tc_f64": ([_PLAN, _INFO, _P, _P, _ENV, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                           ctypes.c_int, _P, _P, ctypes.c_int, _P, _P, ctypes.c_size_t, _P],
                                          ctypes.c_int),
    "dp_tabulate_fusion_env_grad_tc_f64": ([_PLAN, _INFO, _P, _P, _ENV, _P, _I64, _I64, ctypes.c_int, ctypes.c_int,
                                            _P, ctypes.c_int, _P, _P, _P, _P, ctypes.c_size_t, ctypes.c_int, _P],
                                           ctypes.c_int),
    "dp_env_mat_f32": ([_P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, _ENV, _P, _P, _P, _P], ctypes.c_int),
    "dp_force_virial_f64": ([_P, _P, _I64, _I64, ctypes.c_int, _ENV, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_force_virial_f32": ([_P, _P, _I64, _I64, ctypes.c_int, _ENV, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_descriptor_contract_f64": ([_P, _I64, ctypes.c_int, ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_descriptor_contract_f32": ([_P, _I64, ctypes.c_int, ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_descriptor_contract_grad_f64": ([_P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_descriptor_contract_grad_f32": ([_P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_table_build_df64": ([_P, _P, _P, ctypes.c_int, ctypes.c_int, _INFO, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_fwd_moments_df64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                             ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_tabulate_fusion_grad_moments_df64": ([_P, _INFO, _P, _P, _P, _P, _I64, ctypes.c_int, ctypes.c_int, _P,
                                              ctypes.c_int, _P, _P, _P, _P], ctypes.c_int),
    "dp_descriptor_contract_df64": ([_P, _I64, ctypes.c_int, ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_descriptor_contract_grad_df64": ([_P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, _P], ctypes.c_int),
    "dp_fitting_fwd_f64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_fwd_f32": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_fwd_df64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_grad_f64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_grad_f32": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_grad_df64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_grad_noalloc_f64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P], ctypes.c_int),
    "dp_fitting_tc_work_bytes": ([_P, ctypes.c_int, _I64], ctypes.c_size_t),
    **{f"dp_{h}_head_{x}": ([_P, _P, _I64, ctypes.c_int, _P, _P], ctypes.c_int)
       for h in ("vector", "tensor") for x in ("f64", "f32")},
    **{f"dp_{h}_head_grad_{x}": ([_P, _P, _P, _I64, ctypes.c_int, _P, _P, ctypes.c_int, _P], ctypes.c_int)
       for h in ("vector", "tensor") for x in ("f64", "f32")},
    "dp_fitting_fwd_tc_f64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P, ctypes.c_size_t, _P],
                              ctypes.c_int),
    "dp_fitting_grad_tc_f64": ([_P, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P, ctypes.c_size_t, _P],
                               ctypes.c_int),
    "dp_env_mat_df64": ([_P, _P, _I64, ctypes.c_int, ctypes.c_int, _P, _ENV, _P, _P, _P, _P], ctypes.c_int),
    "dp_force_virial_df64": ([_P, _P, _I64, _I64, ctypes.c_int, _ENV, _P, _P, _P, _P, _P], ctypes.c_int),
}
for _name, (_args, _res) in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.argtypes = _args
    _fn.restype = _res


def dp_last_error() -> str:
    return _lib.dp_last_error().decode()


def _check(rc: int):
    if rc != DP_OK:
        raise DPError(rc, dp_last_error())


def _stream(t: torch.Tensor):
    return ctypes.c_void_p(torch.cuda.current_stream(t.device).cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dev(t: torch.Tensor, name: str, dtype=None, shape=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t


# Arithmetic "df64": double arrays, double-float arithmetic; its table is float [npair][nint][3][M1][4].
DF64 = "df64"


def _suffix(dtype) -> str:
    if dtype == torch.float64:
        return "f64"
    if dtype == torch.float32:
        return "f32"
    if dtype == DF64:
        return "df64"
    raise TypeError(f"unsupported dtype {dtype}")


def is_df64_table(table: torch.Tensor) -> bool:
    """A table from dp_table_build(..., dtype="df64"): float, (hi, lo) pairs in a last dimension of 4."""
    return table.dtype == torch.float32 and table.dim() == 5 and table.shape[-1] == 4


def dp_table_info_make(s_min: float, s_max: float, stride0: float = 0.01, stride1: float = 0.1,
                       ext: float = 5.0) -> dp_table_info:
    info = dp_table_info()
    _check(_lib.dp_table_info_make(float(s_min), float(s_max), float(stride0), float(stride1), float(ext),
                                   ctypes.byref(info)))
    return info


def dp_table_info_sizes(info: dp_table_info) -> tuple[int, int]:
    n0, n1 = _I32(), _I32()
    _check(_lib.dp_table_info_sizes(ctypes.byref(info), ctypes.byref(n0), ctypes.byref(n1)))
    return int(n0.value), int(n1.value)


def dp_embedding_net_nodes(params: torch.Tensor, widths, info: dp_table_info, out=None):
    """y, dy, d2y [npair][nint+1][M1] (f64) of the embedding net at the table nodes."""
    params = _dev(params, "params", torch.float64)
    w = (ctypes.c_int32 * len(widths))(*[int(x) for x in widths])
    n0, n1 = dp_table_info_sizes(info)
    npair, M1 = int(params.shape[0]), int(widths[-1])
    shape = (npair, n0 + n1 + 1, M1)
    if out is None:
        out = tuple(torch.empty(shape, dtype=torch.float64, device=params.device) for _ in range(3))
    y, dy, d2y = (_dev(o, "out", torch.float64, shape) for o in out)
    _check(_lib.dp_embedding_net_nodes_f64(_ptr(params), w, len(widths) - 1, npair, ctypes.byref(info), _ptr(y),
                                           _ptr(dy), _ptr(d2y), _stream(params)))
    return y, dy, d2y


def dp_table_build(y, dy, d2y, info: dp_table_info, dtype=torch.float64, out=None) -> torch.Tensor:
    """Quintic coefficient table [npair][nint][3][M1][2] (pair-planar a..f) in `dtype` from f64 node values;
    dtype="df64": float [npair][nint][3][M1][4], each coefficient as a (hi, lo) float pair."""
    y = _dev(y, "y", torch.float64)
    npair, nn, M1 = (int(x) for x in y.shape)
    dy = _dev(dy, "dy", torch.float64, y.shape)
    d2y = _dev(d2y, "d2y", torch.float64, y.shape)
    shape = (npair, nn - 1, 3, M1, 4 if dtype == DF64 else 2)
    tdt = torch.float32 if dtype == DF64 else dtype
    table = torch.empty(shape, dtype=tdt, device=y.device) if out is None else _dev(out, "out", tdt, shape)
    fn = getattr(_lib, f"dp_table_build_{_suffix(dtype)}")
    _check(fn(_ptr(y), _ptr(dy), _ptr(d2y), npair, M1, ctypes.byref(info), _ptr(table), _stream(y)))
    return table


def _sel_arr(sel):
    sel = [int(x) for x in sel]
    return (ctypes.c_int32 * len(sel))(*sel), len(sel), sum(sel)


def _fusion_arrays(dtype, s, Rt, nvalid, atype, sel):
    s = _dev(s, "s", dtype)
    nloc, nnei = (int(x) for x in s.shape)
    Rt = _dev(Rt, "Rt", dtype, (nloc, nnei, 4))
    selc, ntypes, nsum = _sel_arr(sel)
    if nsum != nnei:
        raise ValueError(f"sum(sel) = {nsum} != nnei = {nnei}")
    if nvalid is not None:
        nvalid = _dev(nvalid, "nvalid", torch.int32, (nloc, ntypes))
    if atype is not None:
        atype = _dev(atype, "atype", torch.int32, (nloc,))
    return s, Rt, nvalid, atype, selc, ntypes, nloc, nnei


def _fusion_inputs(table, s, Rt, nvalid, atype, sel):
    df = isinstance(table, torch.Tensor) and is_df64_table(table)
    table = _dev(table, "table", None)
    dtype = torch.float64 if df else table.dtype
    s, Rt, nvalid, atype, selc, ntypes, nloc, nnei = _fusion_arrays(dtype, s, Rt, nvalid, atype, sel)
    if table.dim() != 5 or table.shape[-3] != 3 or table.shape[-1] != (4 if df else 2):
        raise ValueError("table must be [npair][nint][3][M1][2] (or [..][4] for df64) from dp_table_build")
    M1 = int(table.shape[-2])
    return dtype, table, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, (DF64 if df else dtype)


def dp_tabulate_fusion_fwd(table, info: dp_table_info, s, Rt, nvalid, atype, sel, out=None) -> torch.Tensor:
    """T [nloc][4][M1] = (1/nnei) R~^T G with G from the table, valid rows only."""
    return _fwd("dp_tabulate_fusion_fwd", table, info, s, Rt, nvalid, atype, sel, out)


def dp_tabulate_fusion_fwd_moments(table, info: dp_table_info, s, Rt, nvalid, atype, sel, out=None) -> torch.Tensor:
    """The same T through interval moments (runs of neighbours sharing a table interval)."""
    return _fwd("dp_tabulate_fusion_fwd_moments", table, info, s, Rt, nvalid, atype, sel, out)


def dp_tabulate_fusion_fwd_moments_df64(table, info: dp_table_info, s, Rt, nvalid, atype, sel, out=None):
    """T of dp_tabulate_fusion_fwd_moments in df64 arithmetic: f64 s, Rt and T, a df64 table."""
    if not is_df64_table(table):
        raise TypeError("table must come from dp_table_build(..., dtype='df64')")
    return _fwd("dp_tabulate_fusion_fwd_moments", table, info, s, Rt, nvalid, atype, sel, out)


def _fwd(name, table, info, s, Rt, nvalid, atype, sel, out):
    dtype, table, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, arith = _fusion_inputs(table, s, Rt, nvalid,
                                                                                             atype, sel)
    if arith == DF64 and not name.endswith("_moments"):
        raise TypeError(f"{name} has no df64 form; use the _moments call")
    shape = (nloc, 4, M1)
    T = torch.empty(shape, dtype=dtype, device=s.device) if out is None else _dev(out, "out", dtype, shape)
    fn = getattr(_lib, f"{name}_{_suffix(arith)}")
    _check(fn(_ptr(table), ctypes.byref(info), _ptr(s), _ptr(Rt), _ptr(nvalid), _ptr(atype), nloc, nnei, ntypes,
              selc, M1, _ptr(T), _stream(s)))
    return T


def dp_tabulate_fusion_fwd_descriptor(table, info: dp_table_info, s, Rt, nvalid, atype, sel, M2: int, out=None):
    """(T [nloc][4][M1], D [nloc][M1][M2]) in one pass: T as dp_tabulate_fusion_fwd, D = S (S^<)^T."""
    dtype, table, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, arith = _fusion_inputs(table, s, Rt, nvalid,
                                                                                             atype, sel)
    if arith == DF64:
        raise TypeError("dp_tabulate_fusion_fwd_descriptor has no df64 form")
    if out is None:
        T = torch.empty((nloc, 4, M1), dtype=dtype, device=s.device)
        D = torch.empty((nloc, M1, int(M2)), dtype=dtype, device=s.device)
    else:
        T = _dev(out[0], "T", dtype, (nloc, 4, M1))
        D = _dev(out[1], "D", dtype, (nloc, M1, int(M2)))
    fn = getattr(_lib, f"dp_tabulate_fusion_fwd_descriptor_{_suffix(dtype)}")
    _check(fn(_ptr(table), ctypes.byref(info), _ptr(s), _ptr(Rt), _ptr(nvalid), _ptr(atype), nloc, nnei, ntypes,
              selc, M1, int(M2), _ptr(T), _ptr(D), _stream(s)))
    return T, D


def dp_tabulate_fusion_grad(table, info: dp_table_info, s, Rt, nvalid, atype, sel, dT, out=None):
    """(ds [nloc][nnei], dRt [nloc][nnei][4]) from dT = dE/dT [nloc][4][M1]."""
    return _grad("dp_tabulate_fusion_grad", table, info, s, Rt, nvalid, atype, sel, dT, out)


def dp_tabulate_fusion_grad_moments(table, info: dp_table_info, s, Rt, nvalid, atype, sel, dT, out=None):
    """The same (ds, dRt) through interval moments (runs of rows sharing a table interval)."""
    return _grad("dp_tabulate_fusion_grad_moments", table, info, s, Rt, nvalid, atype, sel, dT, out)


def dp_tabulate_fusion_grad_moments_df64(table, info: dp_table_info, s, Rt, nvalid, atype, sel, dT, out=None):
    """(ds, dRt) of dp_tabulate_fusion_grad_moments in df64 arithmetic: f64 arrays, a df64 table."""
    if not is_df64_table(table):
        raise TypeError("table must come from dp_table_build(..., dtype='df64')")
    return _grad("dp_tabulate_fusion_grad_moments", table, info, s, Rt, nvalid, atype, sel, dT, out)


def _grad(name, table, info, s, Rt, nvalid, atype, sel, dT, out):
    dtype, table, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, arith = _fusion_inputs(table, s, Rt, nvalid,
                                                                                             atype, sel)
    if arith == DF64 and not name.endswith("_moments"):
        raise TypeError(f"{name} has no df64 form; use the _moments call")
    dT = _dev(dT, "dT", dtype, (nloc, 4, M1))
    if out is None:
        ds = torch.empty((nloc, nnei), dtype=dtype, device=s.device)
        dRt = torch.empty((nloc, nnei, 4), dtype=dtype, device=s.device)
    else:
        ds = _dev(out[0], "ds", dtype, (nloc, nnei))
        dRt = _dev(out[1], "dRt", dtype, (nloc, nnei, 4))
    fn = getattr(_lib, f"{name}_{_suffix(arith)}")
    _check(fn(_ptr(table), ctypes.byref(info), _ptr(s), _ptr(Rt), _ptr(nvalid), _ptr(atype), nloc, nnei, ntypes,
              selc, M1, _ptr(dT), _ptr(ds), _ptr(dRt), _stream(s)))
    return ds, dRt


def dp_profile_begin(events):
    """Kernel timing hook: the multi-kernel calls record these torch.cuda.Event objects (timing enabled)
    after each of their kernels until dp_profile_end(); returns nothing."""
    handles = []
    for ev in events:
        if ev.cuda_event == 0:  # torch creates the CUDA event on its first record
            ev.record()
        handles.append(ev.cuda_event)
    arr = (ctypes.c_void_p * max(len(handles), 1))(*handles)
    _check(_lib.dp_profile_begin(arr, len(handles)))


def dp_profile_end():
    """Names of what each recorded event follows, in recording order; turns the hook off."""
    n = int(_lib.dp_profile_end())
    return [_lib.dp_profile_name(i).decode() for i in range(n)]


def dp_tc_wait_timeouts() -> int:
    """Tensor-core GEMM waits that gave up since the last call (synchronises the device); 0 normally."""
    n = ctypes.c_uint(0)
    _check(_lib.dp_tc_wait_timeouts(ctypes.byref(n)))
    return int(n.value)


def dp_tabulate_tc_work_bytes(info: dp_table_info, nloc, nnei, ntypes, M1) -> int:
    """Bytes of device scratch dp_tabulate_fusion_{fwd,grad}_tc_f64 need (one size for both)."""
    n = int(_lib.dp_tabulate_tc_work_bytes(ctypes.byref(info), int(nloc), int(nnei), int(ntypes), int(M1)))
    if n == 0:
        raise ValueError(_lib.dp_last_error().decode())
    return n


def _tab_tc_work(work, info, nloc, nnei, ntypes, M1, device):
    need = dp_tabulate_tc_work_bytes(info, nloc, nnei, ntypes, M1)
    if work is None:
        return torch.empty((need,), dtype=torch.uint8, device=device)
    if not work.is_cuda or work.dtype != torch.uint8 or not work.is_contiguous() or work.numel() < need:
        raise ValueError(f"work must be a contiguous CUDA uint8 tensor of at least {need} bytes")
    return work


class TcPlan:
    """A tensor-core tabulation plan: the device buffer dp_tabulate_tc_plan_f64 filled (kept alive here)
    and its host record."""

    def __init__(self, buf: torch.Tensor, rec: dp_tc_plan):
        self.buf, self.rec = buf, rec

    @property
    def info(self) -> dp_table_info:
        return self.rec.info


def dp_tabulate_tc_plan_bytes(info: dp_table_info, nnei, ntypes, M1) -> int:
    """Bytes of the device buffer of a tensor-core tabulation plan."""
    n = int(_lib.dp_tabulate_tc_plan_bytes(ctypes.byref(info), int(nnei), int(ntypes), int(M1)))
    if n == 0:
        raise ValueError(_lib.dp_last_error().decode())
    return n


def dp_tabulate_tc_plan_f64(table, info: dp_table_info, nnei, ntypes=None, buf=None) -> TcPlan:
    """The plan of an f64 table [ntypes^2][nint][3][M1][2] for rows of nnei neighbours (setup, once per
    table): its scaled coefficients and their digit planes; buf: a uint8 CUDA tensor or None."""
    table = _dev(table, "table", torch.float64)
    if table.dim() != 5:
        raise ValueError("table must be [ntypes^2][nint][3][M1][2]")
    npair, M1 = int(table.shape[0]), int(table.shape[3])
    ntypes = int(round(npair ** 0.5)) if ntypes is None else int(ntypes)
    if ntypes * ntypes != npair:
        raise ValueError("table must hold ntypes^2 pair tables")
    need = dp_tabulate_tc_plan_bytes(info, nnei, ntypes, M1)
    if buf is None:
        buf = torch.empty((need,), dtype=torch.uint8, device=table.device)
    elif not buf.is_cuda or buf.dtype != torch.uint8 or not buf.is_contiguous() or buf.numel() < need:
        raise ValueError(f"buf must be a contiguous CUDA uint8 tensor of at least {need} bytes")
    rec = dp_tc_plan()
    _check(_lib.dp_tabulate_tc_plan_f64(_ptr(table), ctypes.byref(info), int(nnei), ntypes, M1, _ptr(buf),
                                        buf.numel(), ctypes.byref(rec), _stream(table)))
    return TcPlan(buf, rec)


def _tc_inputs(plan, info, s, Rt, nvalid, atype, sel):
    """The call's checked arrays and its plan: a TcPlan as given, or one made now from an f64 table."""
    if isinstance(plan, TcPlan):
        s, Rt, nvalid, atype, selc, ntypes, nloc, nnei = _fusion_arrays(torch.float64, s, Rt, nvalid, atype, sel)
        M1 = int(plan.rec.M1)
    else:
        dtype, table, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, arith = _fusion_inputs(plan, s, Rt, nvalid,
                                                                                                 atype, sel)
        if arith != torch.float64:
            raise TypeError("the tensor-core calls take an f64 table and f64 arrays")
        plan = dp_tabulate_tc_plan_f64(table, info, nnei, ntypes)
    return plan, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, torch.float64


def dp_tabulate_fusion_fwd_tc_f64(plan, info: dp_table_info, s, Rt, nvalid, atype, sel, out=None, work=None,
                                  M2=None, D=None):
    """T of dp_tabulate_fusion_fwd in f64 with the per-interval contraction on the tensor cores (interval
    moments times the scaled table, an exact digit-split GEMM).  plan: a TcPlan (dp_tabulate_tc_plan_f64)
    or the f64 table itself, planned for this call; work: a uint8 CUDA tensor of
    dp_tabulate_tc_work_bytes(...) bytes, or None to allocate one.  With M2 given, the same call also
    writes the descriptor (dp_descriptor_contract of T) into D [nloc][M1][M2] (allocated when None) and
    returns (T, D)."""
    plan, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, dtype = _tc_inputs(plan, info, s, Rt, nvalid, atype, sel)
    shape = (nloc, 4, M1)
    T = torch.empty(shape, dtype=dtype, device=s.device) if out is None else _dev(out, "out", dtype, shape)
    if M2 is not None:
        if not 1 <= int(M2) <= M1:
            raise ValueError(f"M2 = {M2} not in 1 .. M1 = {M1}")
        dshape = (nloc, M1, int(M2))
        D = torch.empty(dshape, dtype=dtype, device=s.device) if D is None else _dev(D, "D", dtype, dshape)
    if nloc == 0:
        return T if M2 is None else (T, D)
    work = _tab_tc_work(work, info, nloc, nnei, ntypes, M1, s.device)
    _check(_lib.dp_tabulate_fusion_fwd_tc_f64(ctypes.byref(plan.rec), ctypes.byref(info), _ptr(s), _ptr(Rt),
                                              _ptr(nvalid), _ptr(atype), nloc, nnei, ntypes, selc, M1, _ptr(T),
                                              0 if M2 is None else int(M2), None if M2 is None else _ptr(D),
                                              _ptr(work), work.numel(), _stream(s)))
    return T if M2 is None else (T, D)


def dp_tabulate_fusion_grad_tc_f64(plan, info: dp_table_info, s, Rt, nvalid, atype, sel, dT, out=None, work=None,
                                   flags=0):
    """(ds, dRt) of dp_tabulate_fusion_grad in f64 with the per-interval contraction on the tensor cores;
    plan and work as dp_tabulate_fusion_fwd_tc_f64; flags=DP_TC_REUSE_RUNS takes the interval runs the
    forward left in `work` for the same inputs (see include/dp_compress.h)."""
    plan, s, Rt, nvalid, atype, selc, ntypes, nloc, nnei, M1, dtype = _tc_inputs(plan, info, s, Rt, nvalid, atype, sel)
    dT = _dev(dT, "dT", dtype, (nloc, 4, M1))
    if out is None:
        ds = torch.empty((nloc, nnei), dtype=dtype, device=s.device)
        dRt = torch.empty((nloc, nnei, 4), dtype=dtype, device=s.device)
    else:
        ds = _dev(out[0], "ds", dtype, (nloc, nnei))
        dRt = _dev(out[1], "dRt", dtype, (nloc, nnei, 4))
    if nloc == 0:
        return ds, dRt
    if flags and work is None:
        raise ValueError("DP_TC_REUSE_RUNS needs the forward's work buffer")
    work = _tab_tc_work(work, info, nloc, nnei, ntypes, M1, s.device)
    _check(_lib.dp_tabulate_fusion_grad_tc_f64(ctypes.byref(plan.rec), ctypes.byref(info), _ptr(s), _ptr(Rt),
                                               _ptr(nvalid), _ptr(atype), nloc, nnei, ntypes, selc, M1, _ptr(dT),
                                               _ptr(ds), _ptr(dRt), _ptr(work), work.numel(), int(flags),
                                               _stream(s)))
    return ds, dRt


def _env_tc_inputs(plan, info, coord, nlist, sel, atype):
    """The fused calls' checked arrays and plan (a TcPlan, or one made now from an f64 table)."""
    coord = _dev(coord, "coord", torch.float64)
    if coord.dim() != 2 or coord.shape[1] != 3:
        raise ValueError("coord must be [nall][3]")
    nlist = _dev(nlist, "nlist", torch.int32)
    nloc, nnei = (int(x) for x in nlist.shape)
    selc, ntypes, nsum = _sel_arr(sel)
    if nsum != nnei:
        raise ValueError(f"sum(sel) = {nsum} != nnei = {nnei}")
    atype = None if atype is None else _dev(atype, "atype", torch.int32, (nloc,))
    if not isinstance(plan, TcPlan):
        plan = dp_tabulate_tc_plan_f64(_dev(plan, "table", torch.float64), info, nnei, ntypes)
    return plan, coord, nlist, atype, selc, ntypes, nloc, nnei, int(plan.rec.M1)


def dp_tabulate_fusion_env_fwd_tc_f64(plan, info: dp_table_info, coord, nlist, sel, env: dp_env_info, atype=None,
                                      out=None, work=None, M2=None, D=None, nvalid=None):
    """(T, D, nvalid) of dp_env_mat followed by dp_tabulate_fusion_fwd_tc_f64, in one pass that forms the rows
    from coord [nall][3] and nlist [nloc][nnei] itself (s and R~ never reach memory); D is None unless M2 is
    given.  plan and work as dp_tabulate_fusion_fwd_tc_f64."""
    plan, coord, nlist, atype, selc, ntypes, nloc, nnei, M1 = _env_tc_inputs(plan, info, coord, nlist, sel, atype)
    T = torch.empty((nloc, 4, M1), dtype=torch.float64, device=coord.device) if out is None else \
        _dev(out, "out", torch.float64, (nloc, 4, M1))
    if M2 is not None:
        dshape = (nloc, M1, int(M2))
        D = torch.empty(dshape, dtype=torch.float64, device=coord.device) if D is None else \
            _dev(D, "D", torch.float64, dshape)
    nvalid = torch.empty((nloc, ntypes), dtype=torch.int32, device=coord.device) if nvalid is None else \
        _dev(nvalid, "nvalid", torch.int32, (nloc, ntypes))
    if nloc == 0:
        return T, D, nvalid
    work = _tab_tc_work(work, info, nloc, nnei, ntypes, M1, coord.device)
    _check(_lib.dp_tabulate_fusion_env_fwd_tc_f64(ctypes.byref(plan.rec), ctypes.byref(info), _ptr(coord), _ptr(nlist),
                                                  ctypes.byref(env), _ptr(atype), nloc, nnei, ntypes, selc, M1,
                                                  _ptr(nvalid), _ptr(T), 0 if M2 is None else int(M2),
                                                  None if M2 is None else _ptr(D), _ptr(work), work.numel(),
                                                  _stream(coord)))
    return T, D, nvalid


def dp_tabulate_fusion_env_grad_tc_f64(plan, info: dp_table_info, coord, nlist, sel, env: dp_env_info, atype, dT,
                                       out=None, work=None, flags=0):
    """(F [nall][3], virial [3][3]) of dp_tabulate_fusion_grad_tc_f64 followed by dp_force_virial, in one pass
    from coordinates (s, R~, ds and dR~ never reach memory).  plan, work and flags as
    dp_tabulate_fusion_grad_tc_f64 (DP_TC_REUSE_RUNS after dp_tabulate_fusion_env_fwd_tc_f64 on the same
    inputs and work buffer)."""
    plan, coord, nlist, atype, selc, ntypes, nloc, nnei, M1 = _env_tc_inputs(plan, info, coord, nlist, sel, atype)
    nall = int(coord.shape[0])
    dT = _dev(dT, "dT", torch.float64, (nloc, 4, M1))
    if out is None:
        F = torch.empty((nall, 3), dtype=torch.float64, device=coord.device)
        W = torch.empty((3, 3), dtype=torch.float64, device=coord.device)
    else:
        F = _dev(out[0], "F", torch.float64, (nall, 3))
        W = _dev(out[1], "virial", torch.float64, (3, 3))
    work = _tab_tc_work(work, info, max(nloc, 1), nnei, ntypes, M1, coord.device)
    _check(_lib.dp_tabulate_fusion_env_grad_tc_f64(ctypes.byref(plan.rec), ctypes.byref(info), _ptr(coord),
                                                   _ptr(nlist), ctypes.byref(env), _ptr(atype), nloc, nall, nnei,
                                                   ntypes, selc, M1, _ptr(dT), _ptr(F), _ptr(W), _ptr(work),
                                                   work.numel(), int(flags), _stream(coord)))
    return F, W


def dp_env_mat(coord, nlist, sel, env: dp_env_info, out=None, arith=None):
    """(s [nloc][nnei], Rt [nloc][nnei][4], nvalid [nloc][ntypes] int32) from coord [nall][3] and nlist [nloc][nnei]
    (arith="df64": f64 arrays, df64 arithmetic)."""
    coord = _dev(coord, "coord", None)
    if arith == DF64 and coord.dtype != torch.float64:
        raise TypeError("df64 takes f64 arrays")
    dtype = coord.dtype
    if coord.dim() != 2 or coord.shape[1] != 3:
        raise ValueError("coord must be [nall][3]")
    nlist = _dev(nlist, "nlist", torch.int32)
    nloc, nnei = (int(x) for x in nlist.shape)
    selc, ntypes, nsum = _sel_arr(sel)
    if nsum != nnei:
        raise ValueError(f"sum(sel) = {nsum} != nnei = {nnei}")
    if out is None:
        s = torch.empty((nloc, nnei), dtype=dtype, device=coord.device)
        Rt = torch.empty((nloc, nnei, 4), dtype=dtype, device=coord.device)
        nvalid = torch.empty((nloc, ntypes), dtype=torch.int32, device=coord.device)
    else:
        s = _dev(out[0], "s", dtype, (nloc, nnei))
        Rt = _dev(out[1], "Rt", dtype, (nloc, nnei, 4))
        nvalid = _dev(out[2], "nvalid", torch.int32, (nloc, ntypes))
    fn = getattr(_lib, f"dp_env_mat_{_suffix(arith or dtype)}")
    _check(fn(_ptr(coord), _ptr(nlist), nloc, nnei, ntypes, selc, ctypes.byref(env), _ptr(s), _ptr(Rt), _ptr(nvalid),
              _stream(coord)))
    return s, Rt, nvalid


def dp_force_virial(coord, nlist, env: dp_env_info, ds, dRt, out=None, arith=None):
    """(F [nall][3], virial [3][3]) from dE/ds [nloc][nnei] and dE/dRt [nloc][nnei][4] (arith as dp_env_mat)."""
    coord = _dev(coord, "coord", None)
    if arith == DF64 and coord.dtype != torch.float64:
        raise TypeError("df64 takes f64 arrays")
    dtype = coord.dtype
    if coord.dim() != 2 or coord.shape[1] != 3:
        raise ValueError("coord must be [nall][3]")
    nall = int(coord.shape[0])
    nlist = _dev(nlist, "nlist", torch.int32)
    nloc, nnei = (int(x) for x in nlist.shape)
    ds = _dev(ds, "ds", dtype, (nloc, nnei))
    dRt = _dev(dRt, "dRt", dtype, (nloc, nnei, 4))
    if out is None:
        F = torch.empty((nall, 3), dtype=dtype, device=coord.device)
        W = torch.empty((3, 3), dtype=dtype, device=coord.device)
    else:
        F = _dev(out[0], "F", dtype, (nall, 3))
        W = _dev(out[1], "virial", dtype, (3, 3))
    fn = getattr(_lib, f"dp_force_virial_{_suffix(arith or dtype)}")
    _check(fn(_ptr(coord), _ptr(nlist), nloc, nall, nnei, ctypes.byref(env), _ptr(ds), _ptr(dRt), _ptr(F), _ptr(W),
              _stream(coord)))
    return F, W


def dp_descriptor_contract(T, M2: int, out=None, arith=None) -> torch.Tensor:
    """D [nloc][M1][M2] = S (S^<)^T with S = T^T (arith="df64": f64 arrays, df64 arithmetic)."""
    T = _dev(T, "T", None)
    nloc, four, M1 = (int(x) for x in T.shape)
    if four != 4:
        raise ValueError("T must be [nloc][4][M1]")
    shape = (nloc, M1, int(M2))
    D = torch.empty(shape, dtype=T.dtype, device=T.device) if out is None else _dev(out, "out", T.dtype, shape)
    if arith == DF64 and T.dtype != torch.float64:
        raise TypeError("df64 descriptor takes f64 arrays")
    fn = getattr(_lib, f"dp_descriptor_contract_{_suffix(arith or T.dtype)}")
    _check(fn(_ptr(T), nloc, M1, int(M2), _ptr(D), _stream(T)))
    return D


def dp_descriptor_contract_grad(T, dD, out=None, arith=None) -> torch.Tensor:
    """dT [nloc][4][M1] = dE/dT from dD = dE/dD [nloc][M1][M2] through D = S (S^<)^T (arith as above)."""
    T = _dev(T, "T", None)
    nloc, four, M1 = (int(x) for x in T.shape)
    if four != 4:
        raise ValueError("T must be [nloc][4][M1]")
    dD = _dev(dD, "dD", T.dtype)
    if dD.dim() != 3 or dD.shape[0] != nloc or dD.shape[1] != M1:
        raise ValueError("dD must be [nloc][M1][M2]")
    M2 = int(dD.shape[2])
    dT = torch.empty_like(T) if out is None else _dev(out, "out", T.dtype, T.shape)
    if arith == DF64 and T.dtype != torch.float64:
        raise TypeError("df64 descriptor backward takes f64 arrays")
    fn = getattr(_lib, f"dp_descriptor_contract_grad_{_suffix(arith or T.dtype)}")
    _check(fn(_ptr(T), _ptr(dD), nloc, M1, M2, _ptr(dT), _stream(T)))
    return dT


def dp_descriptor_contract_df64(T, M2: int, out=None) -> torch.Tensor:
    """dp_descriptor_contract in df64 arithmetic (f64 T and D)."""
    return dp_descriptor_contract(T, M2, out, arith=DF64)


def dp_descriptor_contract_grad_df64(T, dD, out=None) -> torch.Tensor:
    """dp_descriptor_contract_grad in df64 arithmetic (f64 T, dD and dT)."""
    return dp_descriptor_contract_grad(T, dD, out, arith=DF64)


def dp_env_mat_df64(coord, nlist, sel, env: dp_env_info, out=None):
    """dp_env_mat in df64 arithmetic (f64 arrays)."""
    return dp_env_mat(coord, nlist, sel, env, out, arith=DF64)


def dp_force_virial_df64(coord, nlist, env: dp_env_info, ds, dRt, out=None):
    """dp_force_virial in df64 arithmetic (f64 arrays)."""
    return dp_force_virial(coord, nlist, env, ds, dRt, out, arith=DF64)


def dp_table_build_df64(y, dy, d2y, info: dp_table_info, out=None) -> torch.Tensor:
    """dp_table_build(..., dtype="df64")."""
    return dp_table_build(y, dy, d2y, info, DF64, out)


def _fit_shape(params, widths, type_start):
    widths = [int(x) for x in widths]
    ts = [int(x) for x in type_start]
    ntypes = len(ts) - 1
    P = sum((widths[l - 1] + 1) * widths[l] for l in range(1, len(widths)))
    if params.dim() != 2 or params.shape[0] != ntypes or params.shape[1] != P:
        raise ValueError(f"params must be [ntypes={ntypes}][{P}]")
    H = sum(widths[1:-1])
    return ((ctypes.c_int32 * len(widths))(*widths), len(widths) - 1, ntypes, (ctypes.c_int64 * len(ts))(*ts), ts[-1],
            widths, H)


def _out_shape(nloc, widths):
    """Shape of the fitting net's outputs (and of g): [nloc] for one output, else [nloc][nout]."""
    return (nloc,) if widths[-1] == 1 else (nloc, widths[-1])


def dp_fitting_fwd(params, widths, type_start, D, out=None, arith=None):
    """(E, act [nloc][H]) of the fitting net, E [nloc] (widths[-1] == 1: the atomic energies) or
    [nloc][widths[-1]] (e.g. the M1 weights of dp_vector_head / dp_tensor_head); D [nloc][widths[0]]
    (a [nloc][M1][M2] descriptor is flattened), atoms sorted by centre type with type_start [ntypes+1]
    (host); arith="df64" as elsewhere."""
    params = _dev(params, "params", None)
    dtype = params.dtype
    w, nlayer, ntypes, ts, nloc, widths, H = _fit_shape(params, widths, type_start)
    D = _dev(D, "D", dtype)
    if D.shape[0] != nloc or D.numel() != nloc * widths[0]:
        raise ValueError(f"D must hold [{nloc}][{widths[0]}]")
    if out is None:
        E = torch.empty(_out_shape(nloc, widths), dtype=dtype, device=params.device)
        act = torch.empty((nloc, max(H, 1)), dtype=dtype, device=params.device)
    else:
        E = _dev(out[0], "E", dtype, _out_shape(nloc, widths))
        act = _dev(out[1], "act", dtype, (nloc, max(H, 1)))
    fn = getattr(_lib, f"dp_fitting_fwd_{_suffix(arith or dtype)}")
    _check(fn(_ptr(params), w, nlayer, ntypes, ts, _ptr(D), _ptr(E), _ptr(act), _stream(params)))
    return E, act


def dp_fitting_grad(params, widths, type_start, act, g=None, out=None, work=None, arith=None):
    """dD [nloc][widths[0]] = sum_c g_ic dE_ic/dD_i from the forward's act; g shaped like the forward's
    E, or None (all ones; one output only)."""
    params = _dev(params, "params", None)
    dtype = params.dtype
    w, nlayer, ntypes, ts, nloc, widths, H = _fit_shape(params, widths, type_start)
    act = _dev(act, "act", dtype, (nloc, max(H, 1)))
    if g is not None:
        g = _dev(g, "g", dtype, _out_shape(nloc, widths))
    dD = torch.empty((nloc, widths[0]), dtype=dtype, device=params.device) if out is None else \
        _dev(out, "out", dtype, (nloc, widths[0]))
    maxh = max(widths[1:-1]) if len(widths) > 2 else 1
    if work is None:
        work = torch.empty((2, nloc, maxh), dtype=dtype, device=params.device)
    else:
        work = _dev(work, "work", dtype, (2, nloc, maxh))
    fn = getattr(_lib, f"dp_fitting_grad_{_suffix(arith or dtype)}")
    _check(fn(_ptr(params), w, nlayer, ntypes, ts, _ptr(act), _ptr(g), _ptr(dD), _ptr(work), _stream(params)))
    return dD


def dp_fitting_grad_noalloc_f64(params, widths, type_start, act, g=None, out=None):
    """dp_fitting_grad in f64 with the library's fixed scratch array: no work buffer and no device
    allocation by the library (for callers that cannot allocate; see include/dp_compress.h)."""
    params = _dev(params, "params", torch.float64)
    w, nlayer, ntypes, ts, nloc, widths, H = _fit_shape(params, widths, type_start)
    act = _dev(act, "act", torch.float64, (nloc, max(H, 1)))
    if g is not None:
        g = _dev(g, "g", torch.float64, _out_shape(nloc, widths))
    dD = torch.empty((nloc, widths[0]), dtype=torch.float64, device=params.device) if out is None else \
        _dev(out, "out", torch.float64, (nloc, widths[0]))
    _check(_lib.dp_fitting_grad_noalloc_f64(_ptr(params), w, nlayer, ntypes, ts, _ptr(act), _ptr(g), _ptr(dD),
                                            _stream(params)))
    return dD


def dp_fitting_tc_work_bytes(widths, nloc) -> int:
    """Bytes of device scratch dp_fitting_fwd_tc_f64 / dp_fitting_grad_tc_f64 need for nloc atoms."""
    widths = [int(x) for x in widths]
    w = (ctypes.c_int32 * len(widths))(*widths)
    n = int(_lib.dp_fitting_tc_work_bytes(w, len(widths) - 1, int(nloc)))
    if n == 0 and len(widths) > 2:
        raise ValueError(f"bad fitting-net widths {widths}")
    return n


def _tc_work(work, widths, nloc, device):
    need = dp_fitting_tc_work_bytes(widths, nloc)
    if work is None:
        return torch.empty((max(need, 1),), dtype=torch.uint8, device=device)
    if not work.is_cuda or work.dtype != torch.uint8 or not work.is_contiguous() or work.numel() < need:
        raise ValueError(f"work must be a contiguous CUDA uint8 tensor of at least {need} bytes")
    return work


def dp_fitting_fwd_tc_f64(params, widths, type_start, D, out=None, work=None):
    """dp_fitting_fwd in f64 with the hidden-layer GEMMs on the tensor cores (exact digit splitting);
    work: a uint8 CUDA tensor of dp_fitting_tc_work_bytes(widths, nloc) bytes, or None to allocate one."""
    params = _dev(params, "params", torch.float64)
    w, nlayer, ntypes, ts, nloc, widths, H = _fit_shape(params, widths, type_start)
    D = _dev(D, "D", torch.float64)
    if D.shape[0] != nloc or D.numel() != nloc * widths[0]:
        raise ValueError(f"D must hold [{nloc}][{widths[0]}]")
    if out is None:
        E = torch.empty(_out_shape(nloc, widths), dtype=torch.float64, device=params.device)
        act = torch.empty((nloc, max(H, 1)), dtype=torch.float64, device=params.device)
    else:
        E = _dev(out[0], "E", torch.float64, _out_shape(nloc, widths))
        act = _dev(out[1], "act", torch.float64, (nloc, max(H, 1)))
    work = _tc_work(work, widths, nloc, params.device)
    _check(_lib.dp_fitting_fwd_tc_f64(_ptr(params), w, nlayer, ntypes, ts, _ptr(D), _ptr(E), _ptr(act), _ptr(work),
                                      work.numel(), _stream(params)))
    return E, act


def dp_fitting_grad_tc_f64(params, widths, type_start, act, g=None, out=None, work=None):
    """dp_fitting_grad in f64 with the GEMMs on the tensor cores; work as dp_fitting_fwd_tc_f64."""
    params = _dev(params, "params", torch.float64)
    w, nlayer, ntypes, ts, nloc, widths, H = _fit_shape(params, widths, type_start)
    act = _dev(act, "act", torch.float64, (nloc, max(H, 1)))
    if g is not None:
        g = _dev(g, "g", torch.float64, _out_shape(nloc, widths))
    dD = torch.empty((nloc, widths[0]), dtype=torch.float64, device=params.device) if out is None else \
        _dev(out, "out", torch.float64, (nloc, widths[0]))
    work = _tc_work(work, widths, nloc, params.device)
    _check(_lib.dp_fitting_grad_tc_f64(_ptr(params), w, nlayer, ntypes, ts, _ptr(act), _ptr(g), _ptr(dD),
                                       _ptr(work), work.numel(), _stream(params)))
    return dD


@dataclass
class Model:
    """A compressed embedding: table range and the tables of every type pair, resident on the device."""
    info: dp_table_info
    table: torch.Tensor
    ntypes: int
    M1: int

    @classmethod
    def compress(cls, params: torch.Tensor, widths, info: dp_table_info, dtype=torch.float64) -> "Model":
        """Net nodes (dp_embedding_net_nodes) -> coefficients (dp_table_build), all on the GPU."""
        y, dy, d2y = dp_embedding_net_nodes(params, widths, info)
        table = dp_table_build(y, dy, d2y, info, dtype)
        npair = int(params.shape[0])
        ntypes = int(round(npair ** 0.5))
        if ntypes * ntypes != npair:
            raise ValueError("params must hold ntypes^2 pair rows")
        return cls(info=info, table=table, ntypes=ntypes, M1=int(widths[-1]))


def table_rows(table: torch.Tensor) -> torch.Tensor:
    """View a pair-planar table [npair][nint][3][M1][2] as [npair][nint][M1][6] rows (a, b, c, d, e, f)."""
    return table.permute(0, 1, 3, 2, 4).reshape(table.shape[0], table.shape[1], table.shape[3], 6)


EXPORTS = tuple(_SIGS)


def _head_inputs(T, a):
    T = _dev(T, "T", None)
    if T.dtype not in (torch.float64, torch.float32) or T.dim() != 3 or T.shape[1] != 4:
        raise ValueError("T must be an f64 or f32 [nloc][4][M1] tensor")
    nloc, M1 = int(T.shape[0]), int(T.shape[2])
    a = _dev(a, "a", T.dtype, (nloc, M1))
    return T, a, nloc, M1


def dp_vector_head(T, a, out=None):
    """v [nloc][3] = sum_m a[m] T[1:4, m] per atom (a vector DP model's head on the compressed T)."""
    T, a, nloc, M1 = _head_inputs(T, a)
    v = torch.empty((nloc, 3), dtype=T.dtype, device=T.device) if out is None else _dev(out, "v", T.dtype, (nloc, 3))
    _check(getattr(_lib, f"dp_vector_head_{_suffix(T.dtype)}")(_ptr(T), _ptr(a), nloc, M1, _ptr(v), _stream(T)))
    return v


def dp_tensor_head(T, a, out=None):
    """A [nloc][3][3] = sum_m a[m] t_m t_m^T, t_m = T[1:4, m] (a tensor DP model's head)."""
    T, a, nloc, M1 = _head_inputs(T, a)
    A = torch.empty((nloc, 3, 3), dtype=T.dtype, device=T.device) if out is None else \
        _dev(out, "A", T.dtype, (nloc, 3, 3))
    _check(getattr(_lib, f"dp_tensor_head_{_suffix(T.dtype)}")(_ptr(T), _ptr(a), nloc, M1, _ptr(A), _stream(T)))
    return A


def _head_grad(kind, T, a, dout, shape, dT, da, accumulate, want):
    T, a, nloc, M1 = _head_inputs(T, a)
    dout = _dev(dout, "dout", T.dtype, (nloc,) + shape)
    if not want or set(want) - {"dT", "da"}:
        raise ValueError("want names dT, da or both")
    if "dT" not in want:
        dT = None
    elif dT is None:
        if accumulate:
            raise ValueError("accumulate needs the dT to add to")
        dT = torch.empty((nloc, 4, M1), dtype=T.dtype, device=T.device)
    else:
        dT = _dev(dT, "dT", T.dtype, (nloc, 4, M1))
    if "da" not in want:
        da = None
    else:
        da = torch.empty((nloc, M1), dtype=T.dtype, device=T.device) if da is None else \
            _dev(da, "da", T.dtype, (nloc, M1))
    fn = getattr(_lib, f"dp_{kind}_head_grad_{_suffix(T.dtype)}")
    _check(fn(_ptr(T), _ptr(a), _ptr(dout), nloc, M1, _ptr(dT), _ptr(da), int(bool(accumulate)), _stream(T)))
    return dT, da


def dp_vector_head_grad(T, a, dv, dT=None, da=None, accumulate=False, want=("dT", "da")):
    """(dT [nloc][4][M1], da [nloc][M1]) from dE/dv [nloc][3]; accumulate adds the head's dT to dT;
    want: the outputs to compute (the other is returned as None)."""
    return _head_grad("vector", T, a, dv, (3,), dT, da, accumulate, want)


def dp_tensor_head_grad(T, a, dA, dT=None, da=None, accumulate=False, want=("dT", "da")):
    """(dT [nloc][4][M1], da [nloc][M1]) from dE/dA [nloc][3][3]; accumulate adds the head's dT to dT;
    want: the outputs to compute (the other is returned as None)."""
    return _head_grad("tensor", T, a, dA, (3, 3), dT, da, accumulate, want)
