"""Helpers for the GPU parity tests: run the CUDA path and the oracle on the same seeded inputs."""
from __future__ import annotations

import functools

import numpy as np
import pytest
import torch

import oracle
import workloads as W

TOL = {torch.float64: 1e-11, torch.float32: 2e-5}
NP = {torch.float64: np.float64, torch.float32: np.float32}


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def lib():
    import paper_2107_02103_gb300 as dpc  # fails loudly if the library is not built
    return dpc


def rel(x, ref) -> float:
    """Max-norm relative error: max |x - ref| / max |ref|."""
    x = np.asarray(x, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    scale = float(np.max(np.abs(ref))) if ref.size else 0.0
    return float(np.max(np.abs(x - ref))) / (scale if scale > 0 else 1.0) if ref.size else 0.0


@functools.lru_cache(maxsize=16)
def workload(name: str, **kw) -> W.Workload:
    return W.make(name, **kw)


def product_model(w: W.Workload, dtype, dev="cuda"):
    dpc = lib()
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    params = torch.from_numpy(w.params).to(dev)
    return dpc.Model.compress(params, w.widths, info, dtype)


def to_dev(w: W.Workload, dtype, dev="cuda"):
    cast = lambda a: torch.from_numpy(np.ascontiguousarray(a.astype(NP[dtype]))).to(dev)  # noqa: E731
    return dict(s=cast(w.s), Rt=cast(w.Rt), dT=cast(w.dT), nvalid=torch.from_numpy(w.nvalid).to(dev),
                atype=torch.from_numpy(w.atype).to(dev))


def run_product(w: W.Workload, dtype, model=None, inputs=None):
    dpc = lib()
    model = model or product_model(w, dtype)
    x = inputs or to_dev(w, dtype)
    T = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    D = dpc.dp_descriptor_contract(T, w.M2)
    ds, dRt = dpc.dp_tabulate_fusion_grad(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel,
                                          x["dT"])
    torch.cuda.synchronize()
    return {k: v.double().cpu().numpy() for k, v in dict(T=T, D=D, ds=ds, dRt=dRt).items()}


def oracle_tables(w: W.Workload, dtype):
    o = oracle.default()
    info = o.table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    tabs = o.tables(w.params, w.widths, info)
    if dtype == torch.float32:
        tabs = tabs.astype(np.float32).astype(np.float64)
    return info, tabs


def run_oracle(w: W.Workload, dtype, atoms=None, tables=None):
    """Oracle outputs in f64 arithmetic; for f32 on the f32-rounded inputs and table."""
    o = oracle.default()
    info, tabs = tables or oracle_tables(w, dtype)
    r = (lambda a: a.astype(np.float32).astype(np.float64)) if dtype == torch.float32 else (lambda a: a)
    s, Rt, dT = r(w.s), r(w.Rt), r(w.dT)
    T = o.fwd(tabs, info, s, Rt, w.nvalid, w.atype, w.sel, atoms=atoms)
    D = o.descriptor(T, w.M2)
    ds, dRt = o.grad(tabs, info, s, Rt, w.nvalid, w.atype, w.sel, dT, atoms=atoms)
    return dict(T=T, D=D, ds=ds, dRt=dRt)


def assert_parity(got, ref, dtype, atoms=None, keys=("T", "D", "ds", "dRt"), tol=None):
    tol = tol or TOL[dtype]
    errs = {}
    for k in keys:
        g = got[k] if atoms is None else got[k][np.asarray(atoms)]
        errs[k] = rel(g, ref[k])
    bad = {k: e for k, e in errs.items() if not e <= tol}
    assert not bad, f"parity beyond {tol}: {errs}"
    return errs
