"""Plain CPU oracle of the DP Compress tabulate-fusion path (arXiv 2107.02103, Sec. II).

TEST INFRASTRUCTURE.  Only `tests/`, `__graft_entry__.smoke()` and the
CPU-baseline leg of `bench.py` may import this package.  It shares no code
with the CUDA library (`paper_2107_02103_gb300`) and never imports it.

The arithmetic lives in `dp_oracle.c` (plain C, long double for the net and
the table, double for the path); this module only moves numpy arrays in and
out of it.  Every function there cites the passage it follows.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dp_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile the oracle with gcc (no contraction of a*b+c into fma)."""
    if (not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src)):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=os.path.dirname(out))
    os.close(fd)
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fno-fast-math", "-std=c11", "-shared", "-fPIC",
           "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


class Info(ctypes.Structure):
    """Table range: fine [lower, upper) step stride0 (n0 intervals), coarse [upper, upper_ext) step stride1."""
    _fields_ = [("lower", ctypes.c_double), ("upper", ctypes.c_double), ("upper_ext", ctypes.c_double),
                ("stride0", ctypes.c_double), ("stride1", ctypes.c_double), ("n0", ctypes.c_int32),
                ("n1", ctypes.c_int32)]

    @property
    def nint(self) -> int:
        return int(self.n0 + self.n1)

    def as_tuple(self):
        return (self.lower, self.upper, self.upper_ext, self.stride0, self.stride1)

    def __repr__(self):
        return (f"Info(lower={self.lower!r}, upper={self.upper!r}, upper_ext={self.upper_ext!r}, "
                f"stride0={self.stride0!r}, stride1={self.stride1!r}, n0={self.n0}, n1={self.n1})")


def load(path: str | None = None):
    """Load the oracle library (building it first if needed); `path` loads another build."""
    global _lib
    if path is None and _lib is not None:
        return _lib
    lib = ctypes.CDLL(path or build())
    P = ctypes.c_void_p
    i32, i64, dbl = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    lib.or_net_eval.argtypes = [P, P, ctypes.c_int, dbl, P, P, P]
    lib.or_net_eval.restype = ctypes.c_int
    lib.or_net_rows.argtypes = [P, i64, P, ctypes.c_int, P, P, i64, P, P, ctypes.c_int]
    lib.or_net_rows.restype = ctypes.c_int
    lib.or_table_info.argtypes = [dbl, dbl, dbl, dbl, dbl, ctypes.POINTER(Info)]
    lib.or_table_info.restype = ctypes.c_int
    lib.or_node_x.argtypes = [ctypes.POINTER(Info), i32]
    lib.or_node_x.restype = dbl
    lib.or_nodes.argtypes = [P, P, ctypes.c_int, ctypes.POINTER(Info), P, P, P]
    lib.or_nodes.restype = ctypes.c_int
    lib.or_table_build.argtypes = [P, P, P, ctypes.c_int, ctypes.POINTER(Info), P]
    lib.or_table_build.restype = None
    lib.or_poly_eval.argtypes = [P, ctypes.c_int, i32, dbl, ctypes.c_int, P]
    lib.or_poly_eval.restype = None
    lib.or_locate.argtypes = [ctypes.POINTER(Info), dbl, ctypes.POINTER(i32), ctypes.POINTER(dbl)]
    lib.or_locate.restype = ctypes.c_int
    lib.or_fwd.argtypes = [P, ctypes.POINTER(Info), P, P, P, P, i64, ctypes.c_int, ctypes.c_int, P, ctypes.c_int,
                           P, i64, P, ctypes.c_int]
    lib.or_fwd.restype = ctypes.c_int
    lib.or_grad.argtypes = [P, ctypes.POINTER(Info), P, P, P, P, i64, ctypes.c_int, ctypes.c_int, P, ctypes.c_int,
                            P, P, i64, P, P, ctypes.c_int]
    lib.or_grad.restype = ctypes.c_int
    lib.or_descriptor.argtypes = [P, i64, ctypes.c_int, ctypes.c_int, P]
    lib.or_descriptor.restype = None
    lib.or_descriptor_grad.argtypes = [P, P, i64, ctypes.c_int, ctypes.c_int, P]
    lib.or_descriptor_grad.restype = None
    lib.or_fitting.argtypes = [P, i64, P, ctypes.c_int, P, P, i64, P, P, P, ctypes.c_int]
    lib.or_fitting.restype = ctypes.c_int
    for f in ("or_vector_head", "or_tensor_head"):
        getattr(lib, f).argtypes = [P, P, i64, ctypes.c_int, P]
        getattr(lib, f).restype = None
    for f in ("or_vector_head_grad", "or_tensor_head_grad"):
        getattr(lib, f).argtypes = [P, P, P, i64, ctypes.c_int, P, P]
        getattr(lib, f).restype = None
    lib.or_embed_rows.argtypes = [P, ctypes.POINTER(Info), P, P, ctypes.c_int, ctypes.c_int, P, ctypes.c_int, P,
                                  i64, P, P]
    lib.or_embed_rows.restype = None
    lib.or_switch.argtypes = [dbl, dbl, dbl, ctypes.c_int, P]
    lib.or_switch.restype = dbl
    lib.or_env_mat.argtypes = [i64, P, P, ctypes.c_int, dbl, dbl, ctypes.c_int, P, P, P]
    lib.or_env_mat.restype = None
    lib.or_force_virial.argtypes = [i64, i64, P, P, ctypes.c_int, dbl, dbl, ctypes.c_int, P, P, P, P, P]
    lib.or_force_virial.restype = None
    if path is None:
        _lib = lib
    return lib


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


class Oracle:
    """Numpy front end of one loaded oracle build (the default build, or a test's variant)."""

    def __init__(self, path: str | None = None):
        self.lib = load(path)

    # -- embedding net ------------------------------------------------------
    def net_eval(self, params, widths, x):
        params = _c(params, np.float64)
        w = _c(widths, np.int32)
        M = int(w[-1])
        y, dy, d2y = (np.empty(M) for _ in range(3))
        r = self.lib.or_net_eval(_p(params), _p(w), len(w) - 1, float(x), _p(y), _p(dy), _p(d2y))
        if r:
            raise ValueError("or_net_eval failed")
        return y, dy, d2y

    def net_rows(self, params, widths, xs, pair, nthreads=0, deriv=True):
        params = _c(np.atleast_2d(params), np.float64)
        w = _c(widths, np.int32)
        xs = _c(xs, np.float64).ravel()
        pair = _c(np.broadcast_to(pair, xs.shape), np.int32)
        M = int(w[-1])
        G = np.empty((xs.size, M))
        dG = np.empty((xs.size, M)) if deriv else None
        r = self.lib.or_net_rows(_p(params), params.shape[1], _p(w), len(w) - 1, _p(xs), _p(pair), xs.size, _p(G),
                                 _p(dG), nthreads)
        if r:
            raise ValueError("or_net_rows failed")
        return (G, dG) if deriv else G

    # -- table --------------------------------------------------------------
    def table_info(self, s_min, s_max, stride0=0.01, stride1=0.1, ext=5.0) -> Info:
        info = Info()
        r = self.lib.or_table_info(float(s_min), float(s_max), float(stride0), float(stride1), float(ext),
                                   ctypes.byref(info))
        if r:
            raise ValueError("empty table range")
        return info

    def node_x(self, info: Info, l: int) -> float:
        return self.lib.or_node_x(ctypes.byref(info), int(l))

    def nodes(self, params, widths, info: Info):
        """y, y', y'' at every node for one parameter row: [nint+1][M] each."""
        params = _c(params, np.float64)
        w = _c(widths, np.int32)
        M = int(w[-1])
        shape = (info.nint + 1, M)
        y, dy, d2y = (np.empty(shape) for _ in range(3))
        r = self.lib.or_nodes(_p(params), _p(w), len(w) - 1, ctypes.byref(info), _p(y), _p(dy), _p(d2y))
        if r:
            raise ValueError("or_nodes failed")
        return y, dy, d2y

    def table_build(self, y, dy, d2y, info: Info):
        y, dy, d2y = (_c(a, np.float64) for a in (y, dy, d2y))
        M = y.shape[-1]
        assert y.shape == (info.nint + 1, M)
        table = np.empty((info.nint, M, 6))
        self.lib.or_table_build(_p(y), _p(dy), _p(d2y), M, ctypes.byref(info), _p(table))
        return table

    def tables(self, params, widths, info: Info):
        """Tables of every parameter row: [npair][nint][M][6]."""
        params = np.atleast_2d(params)
        return np.stack([self.table_build(*self.nodes(params[p], widths, info), info)
                         for p in range(params.shape[0])])

    def poly_eval(self, table, l, t, order=0):
        table = _c(table, np.float64)
        M = table.shape[-2]
        out = np.empty(M)
        self.lib.or_poly_eval(_p(table), M, int(l), float(t), int(order), _p(out))
        return out

    def locate(self, info: Info, x):
        l = ctypes.c_int32()
        t = ctypes.c_double()
        clamped = self.lib.or_locate(ctypes.byref(info), float(x), ctypes.byref(l), ctypes.byref(t))
        return int(l.value), float(t.value), bool(clamped)

    # -- path -----------------------------------------------------------------
    @staticmethod
    def _atoms(atoms, nloc):
        if atoms is None:
            return None, nloc
        a = _c(atoms, np.int64)
        return a, a.size

    def fwd(self, table, info, s, Rt, nvalid, atype, sel, atoms=None, nthreads=0):
        table, s, Rt = (_c(a, np.float64) for a in (table, s, Rt))
        nvalid = _c(nvalid, np.int32)
        sel = _c(sel, np.int32)
        atype_a = None if atype is None else _c(atype, np.int32)
        nloc, nnei = s.shape
        M = table.shape[-2]
        at, n = self._atoms(atoms, nloc)
        T = np.empty((n, 4, M))
        r = self.lib.or_fwd(_p(table), ctypes.byref(info), _p(s), _p(Rt), _p(nvalid), _p(atype_a), nloc, nnei,
                            sel.size, _p(sel), M, _p(at), n, _p(T), nthreads)
        if r:
            raise ValueError("or_fwd: a valid count lies outside [0, sel]")
        return T

    def grad(self, table, info, s, Rt, nvalid, atype, sel, dT, atoms=None, nthreads=0):
        table, s, Rt, dT = (_c(a, np.float64) for a in (table, s, Rt, dT))
        nvalid = _c(nvalid, np.int32)
        sel = _c(sel, np.int32)
        atype_a = None if atype is None else _c(atype, np.int32)
        nloc, nnei = s.shape
        M = table.shape[-2]
        at, n = self._atoms(atoms, nloc)
        ds = np.empty((n, nnei))
        dRt = np.empty((n, nnei, 4))
        r = self.lib.or_grad(_p(table), ctypes.byref(info), _p(s), _p(Rt), _p(nvalid), _p(atype_a), nloc, nnei,
                             sel.size, _p(sel), M, _p(dT), _p(at), n, _p(ds), _p(dRt), nthreads)
        if r:
            raise ValueError("or_grad: a valid count lies outside [0, sel]")
        return ds, dRt

    def descriptor(self, T, M2):
        T = _c(T, np.float64)
        n, four, M = T.shape
        D = np.empty((n, M, M2))
        self.lib.or_descriptor(_p(T), n, M, int(M2), _p(D))
        return D

    def descriptor_grad(self, T, dD):
        T, dD = _c(T, np.float64), _c(dD, np.float64)
        n, four, M = T.shape
        M2 = dD.shape[-1]
        assert dD.shape == (n, M, M2)
        dT = np.empty_like(T)
        self.lib.or_descriptor_grad(_p(T), _p(dD), n, M, int(M2), _p(dT))
        return dT

    def fitting(self, params, widths, D, atype=None, g=None, grad=True, nthreads=0):
        """Outputs of the fitting net, E [n] (widths[-1] == 1: the atomic energies) or [n][widths[-1]],
        and, with grad, sum_c g_c dE_c/dD_i [n][widths[0]] (g shaped like E; None: all ones)."""
        params = _c(np.atleast_2d(params), np.float64)
        w = _c(widths, np.int32)
        D = _c(D.reshape(D.shape[0], -1), np.float64)
        n = D.shape[0]
        assert D.shape[1] == w[0]
        nout = int(w[-1])
        at = None if atype is None else _c(atype, np.int32)
        gg = None if g is None else _c(np.reshape(g, (n, nout)), np.float64)
        E = np.empty((n, nout))
        dD = np.empty((n, int(w[0]))) if grad else None
        if self.lib.or_fitting(_p(params), params.shape[1], _p(w), len(w) - 1, _p(D), _p(at), n, _p(gg), _p(E),
                               _p(dD), nthreads):
            raise ValueError("or_fitting failed")
        E = E[:, 0] if nout == 1 else E
        return (E, dD) if grad else E

    # -- vector and tensor heads ------------------------------------------------
    def vector_head(self, T, a):
        """v [n][3] = sum_m a[m] T[1:4, m] per atom."""
        T, a = _c(T, np.float64), _c(a, np.float64)
        n, four, M = T.shape
        assert a.shape == (n, M)
        v = np.empty((n, 3))
        self.lib.or_vector_head(_p(T), _p(a), n, M, _p(v))
        return v

    def vector_head_grad(self, T, a, dv):
        """(dT [n][4][M], da [n][M]) from dE/dv [n][3]."""
        T, a, dv = _c(T, np.float64), _c(a, np.float64), _c(dv, np.float64)
        n, four, M = T.shape
        dT, da = np.empty_like(T), np.empty((n, M))
        self.lib.or_vector_head_grad(_p(T), _p(a), _p(dv), n, M, _p(dT), _p(da))
        return dT, da

    def tensor_head(self, T, a):
        """A [n][3][3] = sum_m a[m] T[1:4, m] T[1:4, m]^T per atom."""
        T, a = _c(T, np.float64), _c(a, np.float64)
        n, four, M = T.shape
        assert a.shape == (n, M)
        A = np.empty((n, 3, 3))
        self.lib.or_tensor_head(_p(T), _p(a), n, M, _p(A))
        return A

    def tensor_head_grad(self, T, a, dA):
        """(dT [n][4][M], da [n][M]) from dE/dA [n][3][3]."""
        T, a, dA = _c(T, np.float64), _c(a, np.float64), _c(dA, np.float64)
        n, four, M = T.shape
        dT, da = np.empty_like(T), np.empty((n, M))
        self.lib.or_tensor_head_grad(_p(T), _p(a), _p(dA), n, M, _p(dT), _p(da))
        return dT, da

    def embed_rows(self, table, info, s, atype, sel, atoms=None, deriv=False):
        table, s = (_c(a, np.float64) for a in (table, s))
        sel = _c(sel, np.int32)
        atype_a = None if atype is None else _c(atype, np.int32)
        nloc, nnei = s.shape
        M = table.shape[-2]
        at, n = self._atoms(atoms, nloc)
        G = np.empty((n, nnei, M))
        dG = np.empty((n, nnei, M)) if deriv else None
        self.lib.or_embed_rows(_p(table), ctypes.byref(info), _p(s), _p(atype_a), nnei, sel.size, _p(sel), M, _p(at),
                               n, _p(G), _p(dG))
        return (G, dG) if deriv else G


    def switch(self, r, rcs, rc, kind=0):
        """(s(r), s'(r)) of the weighting function (kind 0 cosine, 1 the paper's quintic)."""
        d = ctypes.c_double()
        v = self.lib.or_switch(float(r), float(rcs), float(rc), int(kind), ctypes.byref(d))
        return v, d.value

    def env_mat(self, coord, nlist, rcs, rc, kind=0, norm=None):
        """(s [nloc][nnei], R~ [nloc][nnei][4]) from coordinates [nall][3] and nlist [nloc][nnei] (-1 = padding)."""
        coord, nlist = _c(coord, np.float64), _c(nlist, np.int32)
        nloc, nnei = nlist.shape
        nrm = None if norm is None else _c(np.asarray(norm, dtype=np.float64), np.float64)
        s = np.empty((nloc, nnei))
        Rt = np.empty((nloc, nnei, 4))
        self.lib.or_env_mat(nloc, _p(coord), _p(nlist), nnei, float(rcs), float(rc), int(kind), _p(nrm), _p(s), _p(Rt))
        return s, Rt

    def force_virial(self, coord, nlist, rcs, rc, ds, dRt, kind=0, norm=None):
        """(F [nall][3], W [3][3]) from dE/ds [nloc][nnei] and dE/dR~ [nloc][nnei][4]."""
        coord, nlist = _c(coord, np.float64), _c(nlist, np.int32)
        ds, dRt = _c(ds, np.float64), _c(dRt, np.float64)
        nloc, nnei = nlist.shape
        nall = coord.shape[0]
        nrm = None if norm is None else _c(np.asarray(norm, dtype=np.float64), np.float64)
        F = np.empty((nall, 3))
        W = np.empty((3, 3))
        self.lib.or_force_virial(nloc, nall, _p(coord), _p(nlist), nnei, float(rcs), float(rc), int(kind), _p(nrm),
                                 _p(ds), _p(dRt), _p(F), _p(W))
        return F, W


_default = None


def default() -> Oracle:
    global _default
    if _default is None:
        _default = Oracle()
    return _default
