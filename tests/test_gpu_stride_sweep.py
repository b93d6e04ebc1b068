"""Accuracy of the compressed path against the uncompressed embedding net as the table step Dt
shrinks (Sec. III: the compression error against the step, the fp32 / fp64 comparison) (GPU).

For Dt = 0.1, 0.01, 0.001 the table is built on the GPU and the fused forward and the backward
run in f64, f32 and df64; the reference is the ORIGINAL model: G and G' from the embedding net
itself at every valid row (the oracle's long-double net), contracted by the plain definitions
    T = R~^T G / N_c,   dR~_j = dT G_j / N_c,   ds_j = sum_m (dT^T R~_j)_m G'_jm / N_c.
The quintic Hermite error falls as Dt^6 (Sec. II error bound) until rounding takes over: in f64
and df64 the error must fall by orders of magnitude from 0.1 to 0.01 and reach the double-rounding
floor by 0.001; in f32 it stops at the single-precision floor.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_common import lib, need_gpu, rel, workload

pytestmark = pytest.mark.gpu
STEPS = (0.1, 0.01, 0.001)


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _uncompressed(w):
    """T, ds, dR~ of the original (uncompressed) model in double, by the plain definitions."""
    o = oracle.default()
    off = np.concatenate([[0], np.cumsum(w.sel)])
    idx, pair = [], []
    for b in range(w.ntypes):
        for j in range(int(w.sel[b])):
            ok = np.flatnonzero(w.nvalid[:, b] > j)
            idx.append(np.stack([ok, np.full(ok.size, off[b] + j)], axis=1))
            pair.append(w.atype[ok] * w.ntypes + b)
    idx, pair = np.concatenate(idx), np.concatenate(pair)
    G, dG = o.net_rows(w.params, w.widths, w.s[idx[:, 0], idx[:, 1]], pair)
    Rt = w.Rt[idx[:, 0], idx[:, 1]]                        # [rows][4]
    dT = w.dT[idx[:, 0]]                                   # [rows][4][M1]
    inv = 1.0 / w.nnei
    T = np.zeros((w.nloc, 4, w.M1))
    np.add.at(T, idx[:, 0], Rt[:, :, None] * G[:, None, :] * inv)
    dRt = np.zeros((w.nloc, w.nnei, 4))
    dRt[idx[:, 0], idx[:, 1]] = np.einsum("rkm,rm->rk", dT, G) * inv
    ds = np.zeros((w.nloc, w.nnei))
    ds[idx[:, 0], idx[:, 1]] = np.einsum("rkm,rk,rm->r", dT, Rt, dG) * inv
    return dict(T=T, ds=ds, dRt=dRt)


def _compressed(w, step, arith):
    dpc = lib()
    info = dpc.dp_table_info_make(w.s_min, w.s_max, step, 0.1, w.ext)
    tdt = {"f64": torch.float64, "f32": torch.float32, "df64": dpc.DF64}[arith]
    model = dpc.Model.compress(torch.from_numpy(w.params).cuda(), w.widths, info, tdt)
    io = torch.float32 if arith == "f32" else torch.float64
    cast = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(io)  # noqa: E731
    s, Rt, dT = cast(w.s), cast(w.Rt), cast(w.dT)
    nv, at = torch.from_numpy(w.nvalid).cuda(), torch.from_numpy(w.atype).cuda()
    if arith == "df64":
        T = dpc.dp_tabulate_fusion_fwd_moments_df64(model.table, info, s, Rt, nv, at, w.sel)
        ds, dRt = dpc.dp_tabulate_fusion_grad_moments_df64(model.table, info, s, Rt, nv, at, w.sel, dT)
    else:
        T = dpc.dp_tabulate_fusion_fwd(model.table, info, s, Rt, nv, at, w.sel)
        ds, dRt = dpc.dp_tabulate_fusion_grad(model.table, info, s, Rt, nv, at, w.sel, dT)
    torch.cuda.synchronize()
    nbytes = model.table.numel() * model.table.element_size()
    return {k: v.double().cpu().numpy() for k, v in dict(T=T, ds=ds, dRt=dRt).items()}, nbytes


def test_error_against_the_uncompressed_net_by_step():
    w = workload("water", nmol=128)
    ref = _uncompressed(w)
    err = {}
    for arith in ("f64", "df64", "f32"):
        for step in STEPS:
            got, nbytes = _compressed(w, step, arith)
            err[arith, step] = max(rel(got[k], ref[k]) for k in ("T", "ds", "dRt"))
            print(f"stride-sweep water(nmol=128) {arith:4s} Dt={step:<6g} table {nbytes / 2**20:8.3f} MiB  "
                  f"max-norm relative error vs the uncompressed net "
                  + "  ".join(f"{k} {rel(got[k], ref[k]):.3e}" for k in ("T", "ds", "dRt")))
    for arith in ("f64", "df64"):
        e1, e2, e3 = (err[arith, s] for s in STEPS)
        assert e1 / e2 > 1e3, (arith, e1, e2)   # order-6 convergence: 10^6 per decade until rounding
        assert e2 < 1e-9 and e3 < 1e-11, (arith, e2, e3)
    f1, f2, f3 = (err["f32", s] for s in STEPS)
    assert f1 > f2 and f3 < 1e-4, (f1, f2, f3)       # single precision: a floor near 1e-6
    assert f3 > 10 * err["f64", 0.001]               # f32 cannot reach the double floor
