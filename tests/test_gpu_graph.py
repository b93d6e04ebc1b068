"""The whole model from coordinates to energy, forces and virial (environment matrix, fused forward,
descriptor, fitting net on the tensor cores and its backward, descriptor backward, fused backward,
forces) captured once as a CUDA graph and replayed: the library's calls allocate nothing and never
wait, so they capture as they are, and the replays give the eager results (GPU)."""
import numpy as np
import pytest
import torch

import workloads as W
from gpu_common import lib, need_gpu, rel

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def test_whole_model_replays_as_a_cuda_graph():
    dpc = lib()
    from test_gpu_env_force import _system
    w, coord, nlist, owner, env = _system("water", dict(seed=61, nmol=96), 0, None)
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    model = dpc.Model.compress(torch.from_numpy(w.params).cuda(), w.widths, info, torch.float64)
    widths, fparams = W.fitting_net(17, w.M1 * w.M2, (64, 64, 64), w.ntypes)
    ts = [0] + [int(x) for x in np.cumsum(np.bincount(w.atype, minlength=w.ntypes))]
    cg, ng, at = torch.from_numpy(coord).cuda(), torch.from_numpy(nlist).cuda(), torch.from_numpy(w.atype).cuda()
    fp = torch.from_numpy(fparams).cuda()
    ei = dpc.env_info(*env)
    f64 = dict(dtype=torch.float64, device="cuda")
    H = sum(widths[1:-1])
    buf = dict(s=torch.empty((w.nloc, w.nnei), **f64), Rt=torch.empty((w.nloc, w.nnei, 4), **f64),
               nvalid=torch.empty((w.nloc, w.ntypes), dtype=torch.int32, device="cuda"),
               T=torch.empty((w.nloc, 4, w.M1), **f64), D=torch.empty((w.nloc, w.M1, w.M2), **f64),
               E=torch.empty((w.nloc,), **f64), act=torch.empty((w.nloc, H), **f64),
               dD=torch.empty((w.nloc, w.M1 * w.M2), **f64), dT=torch.empty((w.nloc, 4, w.M1), **f64),
               ds=torch.empty((w.nloc, w.nnei), **f64), dRt=torch.empty((w.nloc, w.nnei, 4), **f64),
               F=torch.empty((coord.shape[0], 3), **f64), virial=torch.empty((3, 3), **f64),
               work=torch.empty((dpc.dp_fitting_tc_work_bytes(widths, w.nloc),), dtype=torch.uint8, device="cuda"))

    def step():
        dpc.dp_env_mat(cg, ng, w.sel, ei, out=(buf["s"], buf["Rt"], buf["nvalid"]))
        dpc.dp_tabulate_fusion_fwd_moments(model.table, model.info, buf["s"], buf["Rt"], buf["nvalid"], at, w.sel,
                                           out=buf["T"])
        dpc.dp_descriptor_contract(buf["T"], w.M2, out=buf["D"])
        dpc.dp_fitting_fwd_tc_f64(fp, widths, ts, buf["D"], out=(buf["E"], buf["act"]), work=buf["work"])
        dpc.dp_fitting_grad_tc_f64(fp, widths, ts, buf["act"], out=buf["dD"], work=buf["work"])
        dpc.dp_descriptor_contract_grad(buf["T"], buf["dD"].view(w.nloc, w.M1, w.M2), out=buf["dT"])
        dpc.dp_tabulate_fusion_grad_moments(model.table, model.info, buf["s"], buf["Rt"], buf["nvalid"], at, w.sel,
                                            buf["dT"], out=(buf["ds"], buf["dRt"]))
        dpc.dp_force_virial(cg, ng, ei, buf["ds"], buf["dRt"], out=(buf["F"], buf["virial"]))

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # eager, on the capture stream: the one-time setup of the calls
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    eager = {k: buf[k].clone() for k in ("E", "dD", "F", "virial")}
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        step()
    for k in ("E", "dD", "F", "virial", "T", "ds"):
        buf[k].fill_(float("nan"))  # the replays must rewrite every output
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(buf["E"], eager["E"])        # no atomics on the way to E: bit for bit
    assert torch.equal(buf["dD"], eager["dD"])
    for k in ("F", "virial"):                        # forces and virial add with atomics
        assert rel(buf[k].cpu().numpy(), eager[k].cpu().numpy()) <= 1e-13, k


def test_tc_calls_replay_as_a_cuda_graph():
    """The tensor-core forward (writing D) and backward (reusing the forward's runs) captured as a graph
    at a size of several backward GEMM units per CTA: the replays give the eager bits."""
    dpc = lib()
    w = W.make("water", seed=67, nmol=1536)  # 4,608 atoms
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    model = dpc.Model.compress(torch.from_numpy(w.params).cuda(), w.widths, info, torch.float64)
    plan = dpc.dp_tabulate_tc_plan_f64(model.table, info, w.nnei)
    x = {k: torch.from_numpy(getattr(w, k)).cuda() for k in ("s", "Rt", "dT", "nvalid", "atype")}
    f64 = dict(dtype=torch.float64, device="cuda")
    buf = dict(T=torch.empty((w.nloc, 4, w.M1), **f64), D=torch.empty((w.nloc, w.M1, w.M2), **f64),
               ds=torch.empty((w.nloc, w.nnei), **f64), dRt=torch.empty((w.nloc, w.nnei, 4), **f64),
               work=torch.empty((dpc.dp_tabulate_tc_work_bytes(info, w.nloc, w.nnei, w.ntypes, w.M1),),
                                dtype=torch.uint8, device="cuda"))
    args = (plan, info, x["s"], x["Rt"], x["nvalid"], x["atype"], [int(v) for v in w.sel])

    def step():
        dpc.dp_tabulate_fusion_fwd_tc_f64(*args, out=buf["T"], work=buf["work"], M2=w.M2, D=buf["D"])
        dpc.dp_tabulate_fusion_grad_tc_f64(*args, x["dT"], out=(buf["ds"], buf["dRt"]), work=buf["work"],
                                           flags=dpc.DP_TC_REUSE_RUNS)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # eager, on the capture stream: the one-time setup of the calls
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    eager = {k: buf[k].clone() for k in ("T", "D", "ds", "dRt")}
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        step()
    for k in eager:
        buf[k].fill_(float("nan"))  # the replays must rewrite every output
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    for k in eager:
        assert torch.equal(buf[k], eager[k]), k
