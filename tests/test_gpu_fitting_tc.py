"""The f64 fitting net with its GEMMs on the tensor cores (exact digit splitting) against the oracle
(Sec. II: E_i from D_i and dE_i/dD_i), against the FP64-pipe path, and on its own edge cases (GPU).
Tolerance 1e-11 (max-norm relative per output array), as for every f64 output; the splitting keeps
the error near that of an f64 GEMM, which the comparison with the FP64-pipe path bounds tighter."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import TOL, lib, need_gpu, rel

pytestmark = pytest.mark.gpu
F64 = TOL[torch.float64]


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64)).cuda()


def _tc(dpc, params, widths, ts, D, g=None, work=None):
    p = _cuda(params)
    E, act = dpc.dp_fitting_fwd_tc_f64(p, widths, ts, _cuda(D), work=work)
    dD = dpc.dp_fitting_grad_tc_f64(p, widths, ts, act, g=None if g is None else _cuda(g), work=work)
    torch.cuda.synchronize()
    return E.cpu().numpy(), act.cpu().numpy(), dD.cpu().numpy()


@pytest.mark.parametrize("hidden,nat,ntypes", [((240, 240, 240), (300, 0, 77), 3), ((37, 37, 50), (65,), 1),
                                               ((24,), (33, 31), 2), ((8, 8), (129, 1), 2),
                                               ((100, 100), (1000,), 1)],
                         ids=["paper", "ragged", "one-hidden", "tiny-tiles", "many-row-tiles"])
def test_tc_fitting_against_oracle(hidden, nat, ntypes):
    """E and dE/dD for several centre types (one empty), widths that are not multiples of the 32 x 80
    tiles or of the 32-deep K slices, K = 1600 (two fp32 partial sums per output), one hidden layer."""
    dpc = lib()
    K = 1600 if hidden == (240, 240, 240) else 70
    widths, params = W.fitting_net(7, K, hidden, ntypes)
    ts = np.concatenate([[0], np.cumsum(nat)]).astype(np.int64)
    n = int(ts[-1])
    D = W.normal(8, (n, K), 0.0, 0.3)
    g = W.normal(9, (n,))
    at = np.repeat(np.arange(ntypes), nat).astype(np.int32)
    E, _, dD = _tc(dpc, params, widths, ts, D, g)
    Eo, dDo = oracle.default().fitting(params, widths, D, at, g=g)
    assert rel(E, Eo) <= F64, rel(E, Eo)
    assert rel(dD, dDo) <= F64, rel(dD, dDo)


def test_tc_matches_the_fp64_pipe_path_closely():
    """Same net and inputs through both f64 paths: the tensor-core one stays within a few f64 roundings
    of the FP64-pipe one (1e-13 relative), on E, every hidden layer's output and dE/dD."""
    dpc = lib()
    widths, params = W.fitting_net(21, 1600, (240, 240, 240), 2)
    ts = np.array([0, 700, 1100], dtype=np.int64)
    D = W.normal(22, (1100, 1600), 0.0, 0.3)
    E, act, dD = _tc(dpc, params, widths, ts, D)
    p = _cuda(params)
    E2, act2 = dpc.dp_fitting_fwd(p, widths, ts, _cuda(D))
    dD2 = dpc.dp_fitting_grad(p, widths, ts, act2)
    torch.cuda.synchronize()
    assert rel(act, act2.cpu().numpy()) <= 1e-13
    assert rel(E, E2.cpu().numpy()) <= 1e-13
    assert rel(dD, dD2.cpu().numpy()) <= 1e-13


def test_tc_row_scaling_zero_rows_and_nan():
    """Rows of D spread over 16 decades keep their own relative accuracy (each row has its own power
    of two: with one exponent for all rows the small rows' D W would vanish and move E by ~1e-8); an
    all-zero row gives the bias-only energy; a NaN in one row makes that atom's E NaN and leaves the
    others untouched.  dE/dD is checked row by row where the first layer is not saturated: in a
    saturated row 1 - tanh^2 ~ 1e-10 carries the cancellation of any f64 evaluation."""
    dpc = lib()
    widths, params = W.fitting_net(31, 64, (48, 48), 1)
    n = 90
    D = W.normal(32, (n, 64), 0.0, 0.3)
    scale = 10.0 ** np.linspace(-8, 8, n)
    D *= scale[:, None]
    D[5] = 0.0
    D[7, ::2] = 0.0
    ts = np.array([0, n], dtype=np.int64)
    E, _, dD = _tc(dpc, params, widths, ts, D)
    Eo, dDo = oracle.default().fitting(params, widths, D)
    for i in range(n):  # per atom: E, and its row of dE/dD where |D| <= 1
        assert abs(E[i] - Eo[i]) <= F64 * max(1.0, abs(Eo[i])), (i, E[i], Eo[i])
        if scale[i] <= 1.0:
            assert rel(dD[i], dDo[i]) <= F64, (i, rel(dD[i], dDo[i]))
    assert rel(dD, dDo) <= F64
    Dn = D.copy()
    Dn[11, 3] = np.nan
    En, _, _ = _tc(dpc, params, widths, ts, Dn)
    assert np.isnan(En[11])
    ok = np.arange(n) != 11
    assert np.array_equal(En[ok], E[ok])


def test_tc_work_buffer_rules_and_reuse():
    """The work size query, a short or misaligned buffer refused on the host, and two calls in a row on
    one buffer giving bit-identical results (nothing carried over from the previous call)."""
    dpc = lib()
    widths, params = W.fitting_net(41, 70, (37, 37, 50), 2)
    ts = np.array([0, 40, 65], dtype=np.int64)
    D = W.normal(42, (65, 70), 0.0, 0.3)
    need = dpc.dp_fitting_tc_work_bytes(widths, 65)
    assert need > 2 * 65 * 50 * 8
    work = torch.empty((need + 256,), dtype=torch.uint8, device="cuda")
    a = _tc(dpc, params, widths, ts, D, work=work[:need])
    work.fill_(0xff)
    b = _tc(dpc, params, widths, ts, D, work=work[:need])
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    p = _cuda(params)
    with pytest.raises((ValueError, dpc.DPError)):
        dpc.dp_fitting_fwd_tc_f64(p, widths, ts, _cuda(D), work=work[:need - 1])
    with pytest.raises(dpc.DPError):
        dpc.dp_fitting_fwd_tc_f64(p, widths, ts, _cuda(D), work=work[16:need + 16])
    E0, act0 = dpc.dp_fitting_fwd_tc_f64(p, widths, [0, 0, 0], torch.empty((0, 70), dtype=torch.float64,
                                                                            device="cuda"))
    assert E0.numel() == 0


def test_tc_forward_tanh_against_numpy():
    """The forward's tanh (evaluated in double-float on the FP32 pipes, rounded to double once) read
    through a 1 -> 1 -> 1 net with W = 1, b = 0, so that act = tanh(D): within 3e-14 relative of
    numpy's tanh from 1e-300 to 19, exactly +-1 beyond 19.1, x itself below 1e-20, NaN kept."""
    dpc = lib()
    widths = [1, 1, 1]
    params = np.array([[1.0, 0.0, 1.0, 0.0]])
    z = np.concatenate([np.linspace(-25.0, 25.0, 4001), 10.0 ** np.linspace(-300, 1.28, 2000),
                        -(10.0 ** np.linspace(-300, 1.28, 2000)), [0.0, -0.0, 19.1, -19.1, 19.0999, np.nan]])
    ts = np.array([0, z.size], dtype=np.int64)
    E, act = dpc.dp_fitting_fwd_tc_f64(_cuda(params), widths, ts, _cuda(z[:, None]))
    t = act.cpu().numpy()[:, 0]
    ref = np.tanh(z)
    ok = ~np.isnan(z)
    relerr = np.abs(t[ok] - ref[ok]) / np.maximum(np.abs(ref[ok]), 1e-300)
    assert relerr.max() <= 3e-14, (relerr.max(), z[ok][np.argmax(relerr)])
    big = np.abs(z) >= 19.1
    assert np.array_equal(t[big], np.sign(z[big]))
    assert np.isnan(t[~ok]).all()
    tiny = np.abs(z) < 1e-20
    assert np.array_equal(t[tiny], z[tiny])


def test_tc_many_atoms_in_row_chunks():
    """More atoms of one type than one chunk of digit planes holds (16,384), a second type after
    them, a width that is no multiple of 48: against the FP64-pipe path (1e-13) and the oracle on a
    sample of atoms."""
    dpc = lib()
    widths, params = W.fitting_net(51, 40, (56, 56), 2)
    ts = np.array([0, 20000, 20300], dtype=np.int64)
    D = W.normal(52, (20300, 40), 0.0, 0.3)
    E, act, dD = _tc(dpc, params, widths, ts, D)
    p = _cuda(params)
    E2, act2 = dpc.dp_fitting_fwd(p, widths, ts, _cuda(D))
    dD2 = dpc.dp_fitting_grad(p, widths, ts, act2)
    torch.cuda.synchronize()
    assert rel(E, E2.cpu().numpy()) <= 1e-13
    assert rel(dD, dD2.cpu().numpy()) <= 1e-13
    pick = np.r_[0:5, 16380:16390, 19995:20005, 20295:20300]
    at = np.repeat(np.arange(2), [20000, 300]).astype(np.int32)
    Eo, dDo = oracle.default().fitting(params, widths, D[pick], at[pick])
    assert rel(E[pick], Eo) <= F64 and rel(dD[pick], dDo) <= F64
