"""The fitting-net backward without allocation (GPU).

dp_fitting_grad_noalloc_f64 serves callers that cannot give the library scratch memory -- a host
program that owns all device memory and hands a plugin only its inputs and outputs.  It takes its
scratch from a fixed array inside the library.  This test calls it through the C ABI twice in a
row, a larger problem and then a smaller one on other inputs, and compares each result with the
allocating dp_fitting_grad_f64 at the f64 tolerance of the other tests; the second call also shows
that what the first left in the shared array does not leak into the result, and that the call
leaves the device's free memory unchanged.  A problem larger than the array is refused with an error.
The file name makes pytest collect it last.
"""
import numpy as np
import pytest
import torch

import workloads as W
from gpu_common import TOL, lib, need_gpu, rel

pytestmark = pytest.mark.gpu


def _case(net_seed, hidden, ts, in_seed):
    widths, params = W.fitting_net(net_seed, 96, hidden, 2)
    n = ts[-1]
    D = torch.from_numpy(W.normal(in_seed, (n, 96), 0.0, 0.5)).cuda()
    g = torch.from_numpy(W.normal(in_seed + 100, (n,))).cuda()
    return widths, torch.from_numpy(params).cuda(), D, g


def test_noalloc_fitting_grad_matches_the_allocating_call():
    """A larger call (2,000 atoms, width 128: 512,000 doubles of scratch) and then a smaller one (700
    atoms, width 64) on other inputs: each equals dp_fitting_grad_f64, so the larger call's leftovers
    in the shared array do not reach the smaller one's result.  Around the second call the device's
    free memory (cudaMemGetInfo) does not change: the call allocates nothing."""
    need_gpu()
    dpc = lib()
    cases = [(31, (128, 128, 128), [0, 1200, 2000], 41), (33, (64, 64, 64), [0, 500, 700], 42)]
    for call, (net_seed, hidden, ts, in_seed) in enumerate(cases):
        widths, p, D, g = _case(net_seed, hidden, ts, in_seed)
        E, act = dpc.dp_fitting_fwd(p, widths, ts, D)
        ref = dpc.dp_fitting_grad(p, widths, ts, act, g=g)
        out = torch.full_like(ref, float("nan"))
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        got = dpc.dp_fitting_grad_noalloc_f64(p, widths, ts, act, g=g, out=out)
        torch.cuda.synchronize()
        free1 = torch.cuda.mem_get_info()[0]
        err = rel(got.cpu().numpy(), ref.cpu().numpy())
        assert err <= TOL[torch.float64], (call, err)
        if call > 0:
            assert free1 == free0, (free0, free1)


def test_noalloc_fitting_grad_refuses_more_than_its_array():
    need_gpu()
    dpc = lib()
    widths, params = W.fitting_net(32, 16, (240, 240), 1)
    ts = [0, 3000]  # 2 x 3000 x 240 = 1,440,000 doubles > 1,048,576
    p = torch.from_numpy(params).cuda()
    E, act = dpc.dp_fitting_fwd(p, widths, ts, torch.zeros((3000, 16), dtype=torch.float64, device="cuda"))
    with pytest.raises(dpc.DPError) as exc:
        dpc.dp_fitting_grad_noalloc_f64(p, widths, ts, act)
    assert "scratch" in str(exc.value)
