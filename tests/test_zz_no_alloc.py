"""The fitting-net backward without allocation (GPU).

dp_fitting_grad_noalloc_f64 serves callers that cannot give the library scratch memory -- a host
program that owns all device memory and hands a plugin only its inputs and outputs.  It takes its
scratch from a fixed array inside the library.  This test calls it through the C ABI twice in a
row, on different inputs, and compares each result with the allocating dp_fitting_grad_f64 at the
f64 tolerance of the other tests; the second call also shows that what the first left in the shared
array does not leak into the result.  A problem larger than the array is refused with an error.
The file name makes pytest collect it last.
"""
import numpy as np
import pytest
import torch

import workloads as W
from gpu_common import TOL, lib, need_gpu, rel

pytestmark = pytest.mark.gpu


def test_noalloc_fitting_grad_matches_the_allocating_call():
    need_gpu()
    dpc = lib()
    widths, params = W.fitting_net(31, 96, (64, 64, 64), 2)
    ts = [0, 700, 1000]  # 2 x 1000 atoms x 64 = 128,000 doubles of scratch, inside the 1,048,576
    p = torch.from_numpy(params).cuda()
    for call, seed in enumerate((41, 42)):
        D = torch.from_numpy(W.normal(seed, (1000, 96), 0.0, 0.5)).cuda()
        g = torch.from_numpy(W.normal(seed + 100, (1000,))).cuda()
        E, act = dpc.dp_fitting_fwd(p, widths, ts, D)
        ref = dpc.dp_fitting_grad(p, widths, ts, act, g=g)
        got = dpc.dp_fitting_grad_noalloc_f64(p, widths, ts, act, g=g,
                                              out=torch.full_like(ref, float("nan")))
        torch.cuda.synchronize()
        err = rel(got.cpu().numpy(), ref.cpu().numpy())
        assert err <= TOL[torch.float64], (call, err)


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
