"""Benchmark of the DP Compress tabulate-fusion hot path on GB300.

One step = one pass of the whole hot path over one synthetic batch:
fused forward T = R~^T G / N_c (dp_tabulate_fusion_fwd), descriptor
D = S S<^T (dp_descriptor_contract) and the backward from a given dE/dT
(dp_tabulate_fusion_grad).  The table build (compression) is setup and is
not timed.  Metric: valid neighbour x channel evaluations per second for
fwd + grad (each valid (atom, neighbour, channel) triple counts once).
--algo tc (the default in f64) runs the interval moments with their
per-interval contraction on the tensor cores (f64 by exact digit
splitting), --algo moments (the default in f32 and df64) the interval
moments on the FMA pipes, --algo direct the per-row kernels; all give the
same outputs, and the roofline fraction is taken on the dominant kernel
of the path that ran (inside the tc calls: the events they record).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload cu85] [--dtype f64]
  python bench.py --impl reference ...   # the oracle on the host cores (bounded sample)

N > 1 runs under torch.distributed.run, one rank per GPU; every rank works on
its own seeded instance of the workload (weak scaling, no collective on the
data path); the reported time is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "tabulate-fusion fwd+grad neighbour·channel evals/s (fp64) and % of roofline"
UNIT = "evals/s"
NSM = 152  # GB300; run_native reads the device's own count and passes it on
SM_MAX_MHZ = 2070.0
# FP64 / FP32 FMA lanes per SM per clock: GB300 is specified at 1.25 TFLOP/s FP64
# (2 lanes/clk/SM at 2.07 GHz over 152 SMs) and 128 FP32 lanes/clk/SM.
FMA_LANES = {"f64": 2, "f32": 128}
# df64 (double-float) arithmetic runs on the FP32 pipe; one df64 FMA is 12 FP32 instructions
# (FMUL, 3 FFMA for the exact product and the cross terms, 8 FADD for the exact sum and the lows).
DF64_OPS_PER_FMA = 12
# algorithmic FMAs per valid neighbour x channel
FMA_PER_EVAL = {"fwd": 9, "grad": 18}
DESC_FMA_PER_ATOM = lambda M1, M2: 4 * M1 * M2  # noqa: E731
# backward of D: dT[k][m] = sum_n dD[m][n] T[k][n] + [m < M2] sum_m' dD[m'][m] T[k][m']
DESC_GRAD_FMA_PER_ATOM = lambda M1, M2: 8 * M1 * M2  # noqa: E731


def footprint(w, esize: int, hbm_bytes: float = 280e9) -> dict:
    """Device memory of one fwd + descriptor + grad pass per atom (the memory side of Sec. III's
    comparison): s, R~, T, dE/dT, D, ds, dR~ and the two int32 count / type arrays.  An uncompressed
    model also materialises the embedding matrix G and keeps every embedding-net layer's output per
    neighbour row for its backward: sum(widths[1:]) values per row.  Atoms per GPU = hbm_bytes / that."""
    ours = esize * (5 * w.nnei + 8 * w.M1 + w.M1 * w.M2 + 5 * w.nnei) + 4 * (w.ntypes + 1)
    net = esize * w.nnei * sum(int(x) for x in w.widths[1:])
    return {"bytes_per_atom": ours, "uncompressed_extra_bytes_per_atom": net,
            "atoms_per_280GB": int(hbm_bytes // ours), "atoms_per_280GB_uncompressed": int(hbm_bytes // (ours + net))}


# f64 fitting GEMMs on the tensor cores: every operand element is split into 9 digits and the 45 digit
# products with s + t <= 10 run as fp16 MMAs, so a GEMM of 2 n K N FP64 flop issues 45 times as many
# fp16 MMA flop; their roofline is the dense 16-bit tensor rate (fp16 and bf16 run at the same rate).
TC_DIGIT_PRODUCTS = 45  # fp16 digit products per FP64-equivalent FMA: nine 6-bit digits (s + t <= 10)


def tc_products(kernel: str, M1: int) -> int:
    """Digit products per FP64-equivalent FMA of a tensor-core tabulation GEMM: the backward uses seven
    8-bit digits (28 products) while its K, M1 padded to 16, is at most 144; else nine 6-bit (45)."""
    return 28 if kernel == "tc_gemm_grad" and -(-M1 // 16) * 16 <= 144 else TC_DIGIT_PRODUCTS


def tensor_peak() -> tuple:
    """(TFLOP/s, basis): the measured dense bf16 GEMM burst rate, else the stated fallback."""
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["bf16_tflops"]), "measured dense bf16 GEMM burst (MEASURED_PEAKS.json)"
    except (OSError, KeyError, ValueError):
        return 1900.0, "fallback 1.9 PFLOP/s dense bf16"


# the C entry point behind each timed kernel
KERNEL_API = {"fwd": "dp_tabulate_fusion_fwd", "grad": "dp_tabulate_fusion_grad", "descriptor": "dp_descriptor_contract",
              "descriptor_grad": "dp_descriptor_contract_grad", "fitting_fwd": "dp_fitting_fwd",
              "fitting_grad": "dp_fitting_grad", "env_mat": "dp_env_mat", "force_virial": "dp_force_virial"}


def fitting_model(w, head=None):
    """The fitting net of the --fitting chain: the paper's (240, 240, 240) hidden layers per centre type
    on the flattened descriptor, random-init (seeded) weights; one output (the energy), or M1 (the
    weights of a vector or tensor head)."""
    import workloads as W
    widths, params = W.fitting_net(W._sub_seed(w.seed, 606), w.M1 * w.M2, (240, 240, 240), w.ntypes)
    if head:
        widths = widths[:-1] + [w.M1]
        params = W.net_params(W._sub_seed(w.seed, 607), widths, w.ntypes)
    return widths, params


def fitting_fmas(w, widths) -> dict:
    """FMAs per step of the fitting net: every layer's w_{l-1} w_l per atom forward, the hidden layers'
    again backward (the output layer's backward is a scaling of its weights)."""
    f = sum(widths[l - 1] * widths[l] for l in range(1, len(widths)))
    b = sum(widths[l - 1] * widths[l] for l in range(1, len(widths) - 1))
    return {"fitting_fwd": f * w.nloc, "fitting_grad": b * w.nloc}


def chain_bytes(w, esize: int, nall: int) -> dict:
    """Algorithmic DRAM bytes of the chain's front and back end (the unique data each one must move):
    env_mat reads the neighbour list and the coordinates once and writes s, R~ (every row) and the counts;
    force_virial reads the neighbour list, the coordinates, ds and dR~ once and writes forces and virial."""
    rows = w.nloc * w.nnei
    coord = 3 * esize * nall
    return {"env_mat": rows * (4 + 5 * esize) + coord + 4 * w.nloc * w.ntypes,
            "force_virial": rows * (4 + 5 * esize) + 2 * coord + 9 * esize}


# Interval-moment path: a run of L consecutive valid rows of one atom in one table
# interval costs, in FMAs, the cheaper of its per-row form and its moment form:
#   forward   min(9 M1 L,  24 M1 + 24 L)   (W[k][q] = sum_j R~_jk t_j^q, then T += C_l W)
#   backward  min(18 M1 L, 24 M1 + 40 L)   (H[k][q] = sum_m dT_km C_lmq, then each row from H)
MOMENT_FMA = {"fwd": (9, 24, 24), "grad": (18, 24, 40)}


def interval_runs(w, info, n0: int, n1: int):
    """Lengths of the runs of consecutive valid rows that share an atom, a type segment and a table
    interval (the interval search of the kernels, on the host in f64)."""
    off = np.concatenate([[0], np.cumsum(w.sel)])
    valid = np.zeros(w.s.shape, bool)
    seg = np.zeros(w.s.shape[1], np.int64)
    for b in range(w.ntypes):
        valid[:, off[b]:off[b + 1]] = np.arange(w.sel[b])[None, :] < w.nvalid[:, b:b + 1]
        seg[off[b]:off[b + 1]] = b
    s = w.s
    nint = n0 + n1
    with np.errstate(invalid="ignore"):
        fine = np.minimum(np.floor((s - info.lower) / info.stride0), n0 - 1)
        coarse = n0 + np.minimum(np.floor((s - info.upper) / info.stride1), n1 - 1)
        l = np.where(s < info.lower, 0, np.where(s < info.upper, fine, np.where(s < info.upper_ext, coarse, nint - 1)))
    key = (np.arange(w.nloc)[:, None] * w.ntypes + seg[None, :]) * nint + np.nan_to_num(l).astype(np.int64)
    k = key[valid]  # row-major: atom, then segment, then row
    if k.size == 0:
        return np.zeros(0, np.int64)
    starts = np.flatnonzero(np.concatenate([[True], k[1:] != k[:-1]]))
    return np.diff(np.concatenate([starts, [k.size]]))


# --algo tc: algorithmic FMAs of its kernels, per valid row (FP64 pipe) or per run x M1 (the
# per-interval contraction on the tensor cores, each FMA as 45 fp16 digit products):
#   tc_runs_moments  W[k][q] += R~_k u^q                 24 per row
#   tc_rows          dE/dR~ and dE/ds by Horner in u     40 per row (20 + 16 + 4)
#   tc_gemm_fwd      T += W C' per run                    24 M1 per run
#   tc_gemm_grad     dW = dT C'^T per run                 24 M1 per run
TC_FMA = {"tc_runs_moments": ("row", 24), "tc_rows": ("row", 40), "tc_gemm_fwd": ("run", 24),
          "tc_gemm_grad": ("run", 24), "tc_finish_fwd": ("atom", 0)}  # the finish: D's 4 M1 M2 per atom
TC_KERNEL = {"tc_runs_moments": "runs_kernel<moments> (dp_tabulate_fusion_fwd_tc_f64)",
             "tc_finish_fwd": "fwd_finish_kernel: T of cut items and D (dp_tabulate_fusion_fwd_tc_f64)",
             "tc_rows": "rows_kernel (dp_tabulate_fusion_grad_tc_f64)",
             "tc_gemm_fwd": "tgemm_kernel (dp_tabulate_fusion_fwd_tc_f64)",
             "tc_gemm_grad": "bgemm_kernel (dp_tabulate_fusion_grad_tc_f64)"}
TC_CHUNK_ATOMS = 16416  # atoms per chunk of the tc calls


def tc_profile_events(w) -> int:
    """Events one step of the tc calls records (an upper bound): a start per call, then per chunk forward
    runs, split, slice lists, and per centre type GEMM and epilogue; backward runs (unless the forward's
    are reused), dT split, per type GEMM, rows."""
    chunks = -(-w.nloc // TC_CHUNK_ATOMS)
    return min(4096, 4 + chunks * (2 + 2 * w.ntypes + 3 + w.ntypes) + 8)


def tc_fmas(w, runs) -> dict:
    rows = float(w.evals) / w.M1
    return {k: (n * rows if per == "row" else DESC_FMA_PER_ATOM(w.M1, w.M2) * w.nloc if per == "atom"
                else n * w.M1 * float(len(runs))) for k, (per, n) in TC_FMA.items()}


def moment_fmas(runs, M1: int) -> dict:
    out = {}
    for kern, (per_row, per_run, per_row_m) in MOMENT_FMA.items():
        out[kern] = float(np.minimum(per_row * M1 * runs, per_run * M1 + per_row_m * runs).sum())
    return out


# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of a kernel, from the one
# `ncu --set full` capture of its current version (the commit the capture was taken at beside each);
# absent means no capture of the current kernel exists and `traffic` is reported as null.
PROFILED_DRAM_BYTES = {("cu85", "f64", "grad", "moments"): 83838464 + 32080640,   # commit 7987c32
                       ("cu85", "f64", "tc_rows", "tc"): 104717312 + 32222720}    # commit a508952


def peak_tflops(dtype: str, mhz: float = SM_MAX_MHZ, nsm: int = NSM) -> float:
    """FMA-pipe peak in TFLOP/s (an FMA = 2 flop); for df64 the FP32 pipe's rate of df64 FMAs."""
    if dtype == "df64":
        return nsm * FMA_LANES["f32"] * 2 * mhz * 1e6 / 1e12 / DF64_OPS_PER_FMA
    return nsm * FMA_LANES[dtype] * 2 * mhz * 1e6 / 1e12


def peak_basis(dtype: str, nsm: int = NSM) -> str:
    if dtype == "df64":
        return (f"FP32 pipe: {nsm} SMs x {FMA_LANES['f32']} lanes/clk x {SM_MAX_MHZ:.0f} MHz / "
                f"{DF64_OPS_PER_FMA} FP32 instructions per df64 FMA, x 2 flop")
    return (f"FP{64 if dtype == 'f64' else 32} FMA pipe: {nsm} SMs (the device's count) x {FMA_LANES[dtype]} "
            f"lanes/clk x 2 flop x {SM_MAX_MHZ:.0f} MHz")


def hbm_peak() -> tuple:
    """(GB/s, basis): the measured copy bandwidth, else the stated fallback."""
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured copy bandwidth (MEASURED_PEAKS.json)"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback 6.8 TB/s"


def step_bytes(w, esize: int) -> dict:
    """Algorithmic DRAM bytes of one fwd + descriptor + grad step: the forward reads s and R~ of the valid
    rows and writes T; the descriptor reads T and writes D; the backward reads s and R~ of the valid rows
    and dE/dT and writes ds and dR~ of every row (padding included); tables are L2-resident."""
    rows = float(w.evals) / w.M1
    t = 4 * w.M1 * esize * w.nloc
    return {"fwd": 5 * esize * rows + t, "descriptor": t + w.M1 * w.M2 * esize * w.nloc,
            "grad": 5 * esize * rows + t + 5 * esize * w.nloc * w.nnei}


def tc_step_bound(w, nruns: float, nsm: int, ms_step: float) -> dict:
    """The roofline of the step the tensor-core path runs: the slowest of its FP64-pipe work (the per-row
    moments, 24 FMA, and derivatives, 40 FMA, per valid row, and the descriptor's 4 M1 M2 per atom) at the
    FP64 peak, its digit-product MMAs (24 M1 FMA per run and direction, 45 fp16 products each forward and
    28 backward) at the measured dense 16-bit tensor peak, and its algorithmic bytes at the measured HBM
    bandwidth."""
    rows = float(w.evals) / w.M1
    fp64_fma = (24 + 40) * rows + DESC_FMA_PER_ATOM(w.M1, w.M2) * w.nloc
    tensor_flop = 2.0 * (tc_products("tc_gemm_fwd", w.M1) + tc_products("tc_gemm_grad", w.M1)) * 24 * w.M1 * float(nruns)
    hbm, hbasis = hbm_peak()
    tpk, tbasis = tensor_peak()
    t = {"fp64": 2.0 * fp64_fma / (peak_tflops("f64", nsm=nsm) * 1e12) * 1e3,
         "tensor": tensor_flop / (tpk * 1e12) * 1e3,
         "hbm": sum(step_bytes(w, 8).values()) / (hbm * 1e9) * 1e3}
    bound = max(t, key=t.get)
    return {"t_roof_ms": round(t[bound], 4), "bound": bound, "fp64_ms": round(t["fp64"], 4),
            "tensor_ms": round(t["tensor"], 4), "hbm_ms": round(t["hbm"], 4), "ms_per_step": round(ms_step, 4),
            "frac": round(t[bound] / ms_step, 4),
            "basis": (f"fwd + descriptor + grad as the tc path computes them: FP64 {fp64_fma:.4g} FMA "
                      f"({peak_basis('f64', nsm)}); tensor {tensor_flop:.4g} flop ({tbasis}); "
                      f"{sum(step_bytes(w, 8).values()):.4g} B ({hbasis})")}


def rank_seed(seed: int, rank: int) -> int:
    """Seed of rank's own instance of the workload (weak scaling: every rank does the full per-GPU work)."""
    return seed + 7919 * rank


def rank_workload(args, rank: int, world: int, **kw):
    """This rank's share of the work.  weak: its own seeded instance of the whole workload (per-GPU work
    fixed as N grows).  strong: one instance, its atoms split into contiguous ranges over the ranks."""
    import workloads as W
    if getattr(args, "scaling", "weak") == "weak":
        return W.make(args.workload, seed=rank_seed(args.seed, rank), **kw)
    w = W.make(args.workload, seed=args.seed, **kw)
    lo, hi = W.shard(w.nloc, rank, world)
    part = {k: getattr(w, k)[lo:hi] for k in ("s", "Rt", "nvalid", "atype", "dT")}
    w.__dict__.update(part, pos=None, box=None, name=f"{w.name}[{lo}:{hi}]")
    return w


def reduce_over_ranks(total_s: float, evals: float, world: int, device) -> tuple[float, float]:
    """Max of the timed seconds and sum of the work over ranks (timing only; the data path has no collective)."""
    if world == 1:
        return total_s, evals
    import torch
    t = torch.tensor([total_s], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    e = torch.tensor([evals], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(e)
    return float(t.item()), float(e.item())


def workload_label(w) -> str:
    d = w.describe()
    return (f"{w.name}: nloc={w.nloc}, sel={d['sel']}, M1={w.M1}, M2={w.M2}, "
            f"mean valid neighbours={d['mean_valid_neighbours']}")


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: str):
        self.idx = gpu
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=5)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "sm_mhz_min": min(sm)}


# --------------------------------------------------------------- native arm
def build_step(args, w, dpc, model, info, sel, dtype, npdt, dev):
    """Host inputs, resident device inputs and outputs, the kernel names and one step of the path.

    Default step: fwd -> descriptor -> grad, from resident s, R~, nvalid, atype and a given dE/dT.
    --chain: the whole descriptor chain from coordinates to forces, env_mat -> fwd -> descriptor ->
    descriptor_grad (a given dE/dD) -> grad -> force_virial, from resident coordinates (periodic images
    as extra rows), the neighbour list, atype and dE/dD."""
    import torch

    import workloads as W
    fwd = dpc.dp_tabulate_fusion_fwd_moments if args.algo == "moments" else dpc.dp_tabulate_fusion_fwd
    grad = dpc.dp_tabulate_fusion_grad_moments if args.algo == "moments" else dpc.dp_tabulate_fusion_grad
    if args.algo == "tc":  # the per-interval contraction on the tensor cores; plan and scratch stay resident
        tcw = torch.empty((dpc.dp_tabulate_tc_work_bytes(info, w.nloc, w.nnei, w.ntypes, w.M1),), dtype=torch.uint8,
                          device=dev)
        plan = dpc.dp_tabulate_tc_plan_f64(model.table, info, w.nnei)  # setup, once per table (like the build)

        def fwd(table, *a, out=None, D=None):  # with D: the descriptor written by the same call
            return dpc.dp_tabulate_fusion_fwd_tc_f64(plan, *a, out=out, work=tcw, M2=None if D is None else w.M2, D=D)

        def grad(table, *a, out=None):  # on the forward's inputs: it takes the forward's interval runs
            return dpc.dp_tabulate_fusion_grad_tc_f64(plan, *a, out=out, work=tcw, flags=dpc.DP_TC_REUSE_RUNS)
    arith = dpc.DF64 if args.dtype == "df64" else None  # the table picks the fusion kernels' arithmetic
    fused_d = args.algo == "tc"  # D from the tensor-core forward itself (no descriptor_kernel launch)
    T = torch.empty((w.nloc, 4, w.M1), dtype=dtype, device=dev)
    D = torch.empty((w.nloc, w.M1, w.M2), dtype=dtype, device=dev)
    ds = torch.empty((w.nloc, w.nnei), dtype=dtype, device=dev)
    dRt = torch.empty((w.nloc, w.nnei, 4), dtype=dtype, device=dev)
    if not args.chain:
        host = {"s": np.ascontiguousarray(w.s.astype(npdt)), "Rt": np.ascontiguousarray(w.Rt.astype(npdt)),
                "nvalid": w.nvalid, "atype": w.atype, "dT": np.ascontiguousarray(w.dT.astype(npdt))}
        d = {k: torch.from_numpy(v).to(dev) for k, v in host.items()}
        outs = dict(T=T, D=D, ds=ds, dRt=dRt)
        names = ["fwd", "grad"] if fused_d else ["fwd", "descriptor", "grad"]

        def step(rec, x, o):
            rec(k := 0)
            if fused_d:  # the tensor-core forward writes D as well
                fwd(model.table, info, x["s"], x["Rt"], x["nvalid"], x["atype"], sel, out=o["T"], D=o["D"])
            else:
                fwd(model.table, info, x["s"], x["Rt"], x["nvalid"], x["atype"], sel, out=o["T"])
                rec(k := k + 1)
                dpc.dp_descriptor_contract(o["T"], w.M2, out=o["D"], arith=arith)
            rec(k := k + 1)
            grad(model.table, info, x["s"], x["Rt"], x["nvalid"], x["atype"], sel, x["dT"], out=(o["ds"], o["dRt"]))
            rec(k := k + 1)
        return host, d, outs, names, step

    coord, nlist, _ = W.ghost_system(w)
    nv = w.env["norm"]
    env = dpc.env_info(w.env["rcs"], w.env["rc"], w.env["kind"], nv)
    host = {"coord": np.ascontiguousarray(coord.astype(npdt)), "nlist": nlist, "atype": w.atype}
    if args.fitting:  # the energy of the whole model: dE/dD comes from the fitting net
        fwidths, fparams = fitting_model(w, args.head)
        fpar = torch.from_numpy(np.ascontiguousarray(fparams.astype(npdt))).to(dev)  # parameters stay resident
        ts = [0] + [int(x) for x in np.cumsum(w.ncentre())]
    else:
        dD = W.normal(W._sub_seed(w.seed, 404), (w.nloc, w.M1, w.M2))
        host["dD"] = np.ascontiguousarray(dD.astype(npdt))
    d = {k: torch.from_numpy(v).to(dev) for k, v in host.items()}
    work = dict(s=torch.empty((w.nloc, w.nnei), dtype=dtype, device=dev),
                Rt=torch.empty((w.nloc, w.nnei, 4), dtype=dtype, device=dev),
                nvalid=torch.empty((w.nloc, w.ntypes), dtype=torch.int32, device=dev),
                dT=torch.empty((w.nloc, 4, w.M1), dtype=dtype, device=dev), T=T, ds=ds, dRt=dRt)
    outs = dict(D=D, F=torch.empty((coord.shape[0], 3), dtype=dtype, device=dev),
                virial=torch.empty((3, 3), dtype=dtype, device=dev))
    names = ["env_mat", "fwd", "descriptor", "descriptor_grad", "grad", "force_virial"]
    fused_env = fused_d and not args.unfused  # rows formed and forces added inside the tensor-core calls
    if fused_d:
        names.remove("descriptor")
    if fused_env:
        names = [n for n in names if n not in ("env_mat", "force_virial")]
    if args.head:  # dE/dv or dE/dA of the vector or tensor model: a resident synthetic input
        hshape = (w.nloc, 3) if args.head == "vector" else (w.nloc, 3, 3)
        host["dhead"] = np.ascontiguousarray(W.normal(W._sub_seed(w.seed, 405), hshape).astype(npdt))
        d["dhead"] = torch.from_numpy(host["dhead"]).to(dev)
        outs["head"] = torch.empty(hshape, dtype=dtype, device=dev)
        work["da"] = torch.empty((w.nloc, w.M1), dtype=dtype, device=dev)
        head_fwd = dpc.dp_vector_head if args.head == "vector" else dpc.dp_tensor_head
        head_grad = dpc.dp_vector_head_grad if args.head == "vector" else dpc.dp_tensor_head_grad
    if args.fitting:
        H = sum(fwidths[1:-1])
        outs["E"] = torch.empty((w.nloc, fwidths[-1]) if args.head else (w.nloc,), dtype=dtype, device=dev)
        work["act"] = torch.empty((w.nloc, H), dtype=dtype, device=dev)
        work["dD"] = torch.empty((w.nloc, w.M1 * w.M2), dtype=dtype, device=dev)
        work["fit_scratch"] = torch.empty((2, w.nloc, max(fwidths[1:-1])), dtype=dtype, device=dev)
        if args.fitting_tc:
            work["fit_tc"] = torch.empty((dpc.dp_fitting_tc_work_bytes(fwidths, w.nloc),), dtype=torch.uint8,
                                         device=dev)
        names = ["env_mat", "fwd", "descriptor", "fitting_fwd", "fitting_grad", "descriptor_grad", "grad",
                 "force_virial"]
        if args.head:
            names = ["env_mat", "fwd", "descriptor", "fitting_fwd", "head", "head_grad_da", "fitting_grad",
                     "descriptor_grad", "head_grad_dT", "grad", "force_virial"]
        if fused_d:
            names.remove("descriptor")
        if fused_env:
            names = [n for n in names if n not in ("env_mat", "force_virial")]

    def step(rec, x, o):
        k = 0
        rec(k)
        if fused_env:  # coordinates -> T, D (and the valid-row counts) in one call
            dpc.dp_tabulate_fusion_env_fwd_tc_f64(plan, info, x["coord"], x["nlist"], sel, env, x["atype"],
                                                  out=work["T"], work=tcw, M2=w.M2, D=o["D"], nvalid=work["nvalid"])
        else:
            dpc.dp_env_mat(x["coord"], x["nlist"], sel, env, out=(work["s"], work["Rt"], work["nvalid"]), arith=arith)
            rec(k := k + 1)
        if fused_env:
            pass
        elif fused_d:
            fwd(model.table, info, work["s"], work["Rt"], work["nvalid"], x["atype"], sel, out=work["T"], D=o["D"])
        else:
            fwd(model.table, info, work["s"], work["Rt"], work["nvalid"], x["atype"], sel, out=work["T"])
            rec(k := k + 1)
            dpc.dp_descriptor_contract(work["T"], w.M2, out=o["D"], arith=arith)
        rec(k := k + 1)
        if args.fitting:
            if args.fitting_tc:
                dpc.dp_fitting_fwd_tc_f64(fpar, fwidths, ts, o["D"], out=(o["E"], work["act"]), work=work["fit_tc"])
            else:
                dpc.dp_fitting_fwd(fpar, fwidths, ts, o["D"], out=(o["E"], work["act"]), arith=arith)
            rec(k := k + 1)
            if args.head:  # v or A from T and the net's M1 outputs; dE/da for the net's backward
                head_fwd(work["T"], o["E"], out=o["head"])
                rec(k := k + 1)
                head_grad(work["T"], o["E"], x["dhead"], da=work["da"], want=("da",))
                rec(k := k + 1)
            g_fit = work["da"] if args.head else None
            if args.fitting_tc:
                dpc.dp_fitting_grad_tc_f64(fpar, fwidths, ts, work["act"], g=g_fit, out=work["dD"],
                                           work=work["fit_tc"])
            else:
                dpc.dp_fitting_grad(fpar, fwidths, ts, work["act"], g=g_fit, out=work["dD"],
                                    work=work["fit_scratch"], arith=arith)
            rec(k := k + 1)
            dD_in = work["dD"].view(w.nloc, w.M1, w.M2)
        else:
            dD_in = x["dD"]
        dpc.dp_descriptor_contract_grad(work["T"], dD_in, out=work["dT"], arith=arith)
        rec(k := k + 1)
        if args.head:  # the head's own dE/dT added to the descriptor's
            head_grad(work["T"], o["E"], x["dhead"], dT=work["dT"], accumulate=True, want=("dT",))
            rec(k := k + 1)
        if fused_env:  # dE/dT -> forces and virial in one call, on the forward's interval runs
            dpc.dp_tabulate_fusion_env_grad_tc_f64(plan, info, x["coord"], x["nlist"], sel, env, x["atype"], work["dT"],
                                                   out=(o["F"], o["virial"]), work=tcw, flags=dpc.DP_TC_REUSE_RUNS)
            rec(k := k + 1)
            return
        grad(model.table, info, work["s"], work["Rt"], work["nvalid"], x["atype"], sel, work["dT"],
             out=(work["ds"], work["dRt"]))
        rec(k := k + 1)
        dpc.dp_force_virial(x["coord"], x["nlist"], env, work["ds"], work["dRt"], out=(o["F"], o["virial"]),
                            arith=arith)
        rec(k := k + 1)
    return host, d, outs, names, step


def run_native(args, rank, world, local_rank):
    import torch

    import paper_2107_02103_gb300 as dpc

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    args.nsm = int(torch.cuda.get_device_properties(dev).multi_processor_count)  # the peaks use the device's count
    dtype = torch.float32 if args.dtype == "f32" else torch.float64
    npdt = np.float32 if args.dtype == "f32" else np.float64
    kw = {}
    if args.workload == "alcumg":
        kw["pad"] = args.pad
    w = rank_workload(args, rank, world, **kw)
    if args.chain and w.env is None:
        raise SystemExit(f"--chain needs positions and a neighbour list; workload {w.name} has none")
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    model = dpc.Model.compress(torch.from_numpy(w.params).to(dev), w.widths, info,
                               dpc.DF64 if args.dtype == "df64" else dtype)
    sel = [int(x) for x in w.sel]
    host, d, outs, names, step = build_step(args, w, dpc, model, info, sel, dtype, npdt, dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)  # 256 MiB > 126 MiB L2
    stream = torch.cuda.current_stream(dev)
    nk = len(names)

    def run_step(ev=None, x=None, o=None):
        step((lambda k: ev[k].record(stream)) if ev else (lambda k: None), x or d, o or outs)

    for _ in range(args.warmup):
        run_step()
    torch.cuda.synchronize(dev)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nk + 1)] for _ in range(args.steps)]
    pev, pnames = None, []
    if args.algo == "tc":  # per-kernel times inside the tc calls, from events they record themselves
        pev = [[torch.cuda.Event(enable_timing=True) for _ in range(tc_profile_events(w))] for _ in range(args.steps)]
        for e in (e for row in pev for e in row):
            e.record(stream)  # creates the CUDA events before the timed region
    vis = [x for x in os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",") if x.strip()]
    clocks = ClockSampler(vis[local_rank] if local_rank < len(vis) else str(local_rank))
    barrier()
    torch.cuda.synchronize(dev)
    if rank == 0:
        clocks.start()
    t_wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.zero_()  # evict the previous step's data from L2 (outside the timed events)
        if pev:
            dpc.dp_profile_begin(pev[k])
        run_step(evs[k])
        if pev:
            pnames.append(dpc.dp_profile_end())
    torch.cuda.synchronize(dev)
    t_wall = time.perf_counter() - t_wall0
    barrier()
    clk = clocks.stop() if rank == 0 else None

    step_ms = [e[0].elapsed_time(e[nk]) for e in evs]
    k_ms = {n: [e[j].elapsed_time(e[j + 1]) for e in evs] for j, n in enumerate(names)}
    tc_ms = None
    if pev:
        tc_ms = {}
        for k, nm in enumerate(pnames):
            for i in range(1, len(nm)):
                if nm[i] not in ("tc_fwd", "tc_grad"):  # a call's start closes nothing
                    tc_ms.setdefault(nm[i], [0.0] * args.steps)[k] += pev[k][i - 1].elapsed_time(pev[k][i])
    total_s, evals_all = reduce_over_ranks(sum(step_ms) / 1e3, float(w.evals), world, dev)

    # ---- the same step captured once as a CUDA graph (the chain's many launches in one)
    graph = measure_graph(run_step, flush, dev, args.steps) if (args.chain and not args.no_graph) else None

    # ---- end to end through the public API: pinned host inputs -> device -> path -> host results
    e2e = None if args.no_e2e else measure_e2e(args, host, d, outs, run_step, stream, dev, world, barrier,
                                                evals_all)
    if rank != 0:
        return None
    fmas = None
    if args.algo in ("moments", "tc"):
        fmas = moment_fmas(interval_runs(w, info, *dpc.dp_table_info_sizes(info)), w.M1)
    nall = int(host["coord"].shape[0]) if "coord" in host else w.nloc
    tcf = tc_fmas(w, interval_runs(w, info, *dpc.dp_table_info_sizes(info))) if tc_ms else None
    per_mark = {"tc_split_dT": 1 if -(-w.M1 // 16) * 16 <= 144 else 2, "tc_slice_lists": 2, "tc_fwd": 0,
                "tc_grad": 0}  # kernels per mark
    out = report(args, w, world, step_ms, k_ms, total_s, evals_all, e2e, clk, t_wall, fmas, nall, tc_ms, tcf,
                 [sum(per_mark.get(x, 1) for x in nm) for nm in pnames])
    if graph is not None:
        graph["evals_per_s"] = w.evals / (graph["ms_per_step"] * 1e-3)
        out["graph"] = graph
    if world == 1 and not args.no_variants and not args.chain and args.dtype == "f64" and args.algo in ("moments",
                                                                                                         "tc"):
        out["variants"] = measure_variants(args, w, dpc, info, sel, d, outs, flush, stream, dev, fmas)
    return out


def measure_graph(run_step, flush, dev, nsteps):
    """The step captured once as a CUDA graph and replayed: its launches (a few dozen in the chain with
    the fitting net) leave the host as one.  The library's calls allocate nothing and never wait, so
    they capture as they are; one eager step on the capture stream first does their one-time setup.
    Inputs resident, L2 flushed between replays (outside the events), CUDA events around each replay."""
    import torch
    side = torch.cuda.Stream(device=dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    with torch.cuda.stream(side):
        run_step()
    torch.cuda.current_stream(dev).wait_stream(side)
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        run_step()
    g.replay()
    torch.cuda.synchronize(dev)
    st = torch.cuda.current_stream(dev)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nsteps)]
    for e0, e1 in evs:
        flush.zero_()
        e0.record(st)
        g.replay()
        e1.record(st)
    torch.cuda.synchronize(dev)
    ms = sum(a.elapsed_time(b) for a, b in evs) / nsteps
    return {"ms_per_step": round(ms, 4), "replays": nsteps,
            "note": "the same step captured once as a CUDA graph and replayed (per-kernel times above: eager)"}


def measure_variants(args, w, dpc, info, sel, d, ref_outs, flush, stream, dev, fmas):
    """The same step by the other f64-accurate kernels, on the same resident inputs, timed the same way
    (L2 flushed between steps, CUDA events per kernel): the per-row kernels (the paper's per-neighbour
    evaluation) and the df64 moment kernels (double arrays, double-float arithmetic on the FP32 pipes),
    with the max-norm relative difference of each output from the default path's."""
    import torch
    model_df = dpc.Model.compress(torch.from_numpy(w.params).to(dev), w.widths, info, dpc.DF64)
    model_64 = dpc.Model.compress(torch.from_numpy(w.params).to(dev), w.widths, info, torch.float64)
    nsteps = max(3, min(args.steps, 100))
    res = {}
    todo = [("f64_per_row", model_64, dpc.dp_tabulate_fusion_fwd, dpc.dp_tabulate_fusion_grad, None),
            ("df64_moments", model_df, dpc.dp_tabulate_fusion_fwd_moments, dpc.dp_tabulate_fusion_grad_moments,
             dpc.DF64)]
    if args.algo == "tc":
        todo.insert(0, ("f64_moments", model_64, dpc.dp_tabulate_fusion_fwd_moments,
                        dpc.dp_tabulate_fusion_grad_moments, None))
    for name, model, fwd, grad, arith in todo:
        o = {k: torch.empty_like(v) for k, v in ref_outs.items()}

        def step(rec):
            rec(0)
            fwd(model.table, info, d["s"], d["Rt"], d["nvalid"], d["atype"], sel, out=o["T"])
            rec(1)
            dpc.dp_descriptor_contract(o["T"], w.M2, out=o["D"], arith=arith)
            rec(2)
            grad(model.table, info, d["s"], d["Rt"], d["nvalid"], d["atype"], sel, d["dT"], out=(o["ds"], o["dRt"]))
            rec(3)
        for _ in range(args.warmup):
            step(lambda k: None)
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(nsteps)]
        torch.cuda.synchronize(dev)
        for k in range(nsteps):
            flush.zero_()
            step(lambda j, k=k: evs[k][j].record(stream))
        torch.cuda.synchronize(dev)
        ms = {n: sum(e[j].elapsed_time(e[j + 1]) for e in evs) / nsteps for j, n in enumerate(("fwd", "descriptor", "grad"))}
        tot = sum(ms.values())
        pk = peak_tflops("df64" if arith else "f64", nsm=getattr(args, "nsm", NSM))
        fm = fmas if name.endswith("moments") else {"fwd": FMA_PER_EVAL["fwd"] * w.evals,
                                                     "grad": FMA_PER_EVAL["grad"] * w.evals}
        diff = {k: float(((o[k] - ref_outs[k]).abs().max() / ref_outs[k].abs().max()).item()) for k in ref_outs}
        res[name] = {"value": w.evals / (tot * 1e-3), "unit": UNIT, "ms_per_step": round(tot, 4), "steps": nsteps,
                     "dtype": "df64" if arith else "f64",
                     "kernels": {k: {"ms": round(v, 4)} for k, v in ms.items()},
                     "frac": {k: round(2.0 * fm[k] / (ms[k] * 1e-3) / 1e12 / pk, 4) for k in ("fwd", "grad")},
                     "peak_tflops": round(pk, 4), "max_rel_diff_vs_default": diff}
    return res


def measure_e2e(args, host, d, outs, step, stream, dev, world, barrier, evals_all):
    """The metric end to end through the public API with host buffers: every step uploads its inputs
    (s, R~, nvalid, atype, dT; with --chain coordinates, neighbour list, atype and dE/dD or, with
    --fitting, nothing more) from pinned host memory and downloads its results (T, D, ds, dR~; with
    --chain D, forces and virial, and with --fitting the atomic energies).  Steps
    are pipelined the way a streaming caller would run them: double-buffered device inputs and outputs,
    the upload of step k+1 and the download of step k-1 on their own streams while step k computes."""
    import torch
    import paper_2107_02103_gb300 as dpc  # noqa: F401  (the path runs through `step`)
    pin = {k: torch.from_numpy(v).pin_memory() for k, v in host.items()}
    outs_h = {k: torch.empty(t.shape, dtype=t.dtype).pin_memory() for k, t in outs.items()}
    h2d = sum(v.numel() * v.element_size() for v in pin.values())
    d2h = sum(v.numel() * v.element_size() for v in outs_h.values())
    bufs_in = [d, {k: torch.empty_like(v) for k, v in d.items()}]
    bufs_out = [outs, {k: torch.empty_like(v) for k, v in outs.items()}]
    up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    uploaded = [torch.cuda.Event() for _ in range(2)]
    computed = [torch.cuda.Event() for _ in range(2)]
    downloaded = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]

    def upload(k):
        b = k % 2
        with torch.cuda.stream(up):
            up.wait_event(consumed[b])
            for name, v in pin.items():
                bufs_in[b][name].copy_(v, non_blocking=True)
            uploaded[b].record(up)

    def run(n):
        for e in consumed + downloaded:
            e.record(stream)
        upload(0)
        for k in range(n):
            b = k % 2
            if k + 1 < n:
                upload(k + 1)
            stream.wait_event(uploaded[b])
            stream.wait_event(downloaded[b])
            step(None, bufs_in[b], bufs_out[b])
            consumed[b].record(stream)
            computed[b].record(stream)
            with torch.cuda.stream(down):
                down.wait_event(computed[b])
                for name, t in bufs_out[b].items():
                    outs_h[name].copy_(t, non_blocking=True)
                downloaded[b].record(down)
        stream.wait_stream(down)

    run(max(1, args.warmup))
    torch.cuda.synchronize(dev)
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    run(args.steps)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    e2e_s, _ = reduce_over_ranks(e0.elapsed_time(e1) / 1e3, 0.0, world, dev)
    barrier()
    return {"value": evals_all * args.steps / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "pipelined": "double-buffered, uploads and downloads on their own streams"}


def report(args, w, world, step_ms, k_ms, total_s, evals_all, e2e, clk, t_wall, fmas=None, nall=0, tc_ms=None,
           tcf=None, tc_launches=None):
    head = getattr(args, "head", None)  # a vector or tensor model
    value = evals_all * args.steps / total_s
    # ---- roofline of the dominant kernel (FMA pipe of the path's dtype), on the FMAs of the
    # algorithm the kernels run: per-row evaluation, or interval moments (fmas, from the run lengths)
    mean = {k: sum(v) / len(v) for k, v in k_ms.items()}
    fmas = fmas or {"fwd": FMA_PER_EVAL["fwd"] * w.evals, "grad": FMA_PER_EVAL["grad"] * w.evals}
    flops = {"fwd": 2.0 * fmas["fwd"], "grad": 2.0 * fmas["grad"],
             "descriptor": 2.0 * DESC_FMA_PER_ATOM(w.M1, w.M2) * w.nloc,
             "descriptor_grad": 2.0 * DESC_GRAD_FMA_PER_ATOM(w.M1, w.M2) * w.nloc}
    if "descriptor" not in k_ms:  # the forward wrote D as well (tensor-core path)
        flops["fwd"] += flops["descriptor"]
    if getattr(args, "fitting", False):
        flops.update({k: 2.0 * v for k, v in fitting_fmas(w, fitting_model(w, getattr(args, "head", None))[0]).items()})
    nbytes = chain_bytes(w, 4 if args.dtype == "f32" else 8, nall) if args.chain else {}
    nsm = getattr(args, "nsm", NSM)
    pk = peak_tflops(args.dtype, nsm=nsm)
    tc = bool(getattr(args, "fitting_tc", False))
    tpk, tbasis = tensor_peak()
    kernels = {}
    for k in mean:
        e = {"ms": round(mean[k], 4), "share": round(mean[k] / sum(mean.values()), 4)}
        if k in flops:
            e["tflops"] = round(flops[k] / (mean[k] * 1e-3) / 1e12, 4)
            e["frac"] = round(flops[k] / (mean[k] * 1e-3) / 1e12 / pk, 4)
        if k in nbytes:
            e["gbs"] = round(nbytes[k] / (mean[k] * 1e-3) / 1e9, 1)
        if tc and k in ("fitting_fwd", "fitting_grad"):  # FP64-equivalent above; the MMAs it takes here
            e["tensor_tflops"] = round(TC_DIGIT_PRODUCTS * flops[k] / (mean[k] * 1e-3) / 1e12, 2)
            e["tensor_frac"] = round(e["tensor_tflops"] / tpk, 4)
        kernels[k] = e
    dom = max((k for k in mean if k in flops), key=mean.get)  # the roofline covers the FMA-counted kernels
    achieved = flops[dom] / (mean[dom] * 1e-3) / 1e12
    path_tflops = (flops["fwd"] + flops["grad"]) / ((mean["fwd"] + mean["grad"]) * 1e-3) / 1e12
    api = KERNEL_API[dom] + ("_tc_f64" if tc and dom.startswith("fitting") else "")
    roofline = {"bound": "alu", "achieved": round(achieved, 4), "peak": round(pk, 4), "unit": "TFLOP/s",
                "frac": round(achieved / pk, 4), "traffic": PROFILED_DRAM_BYTES.get((w.name, args.dtype, dom, args.algo)),
                "kernel": api,
                "peak_basis": peak_basis(args.dtype, nsm),
                "fwd_grad_frac": round(path_tflops / pk, 4)}
    if tc and dom.startswith("fitting"):
        roofline.update({"bound": "tensor", "achieved": kernels[dom]["tensor_tflops"], "peak": round(tpk, 1),
                         "frac": kernels[dom]["tensor_frac"], "traffic": None,
                         "peak_basis": f"{tbasis}; achieved counts all {TC_DIGIT_PRODUCTS} fp16 digit products"})
    if tc_ms:  # the tensor-core tabulation: its own kernels, timed by the events its calls record
        step_mean = sum(step_ms) / len(step_ms)
        tmean = {k: sum(v) / len(v) for k, v in tc_ms.items()}
        for k, ms in tmean.items():
            e = {"ms": round(ms, 4), "share": round(ms / step_mean, 4)}
            if k in tcf:
                e["tflops"] = round(2.0 * tcf[k] / (ms * 1e-3) / 1e12, 4)  # FP64 (equivalent) flop
                if k.startswith("tc_gemm"):
                    e["tensor_tflops"] = round(tc_products(k, w.M1) * e["tflops"], 2)
                    e["tensor_frac"] = round(e["tensor_tflops"] / tpk, 4)
                else:
                    e["frac"] = round(e["tflops"] / pk, 4)
            kernels[k] = e
        dom = max(tmean, key=tmean.get)
        if dom in tcf:
            e = kernels[dom]
            gemm = dom.startswith("tc_gemm")
            roofline = {"bound": "tensor" if gemm else "alu",
                        "achieved": e["tensor_tflops"] if gemm else e["tflops"],
                        "peak": round(tpk, 1) if gemm else round(pk, 4), "unit": "TFLOP/s",
                        "frac": e["tensor_frac"] if gemm else e["frac"],
                        "traffic": PROFILED_DRAM_BYTES.get((w.name, args.dtype, dom, args.algo)),
                        "kernel": TC_KERNEL[dom],
                        "peak_basis": (f"{tbasis}; achieved counts all {tc_products(dom, w.M1)} fp16 digit products"
                                       if gemm else peak_basis(args.dtype, nsm)),
                        "fwd_grad_frac_fp64_equivalent": round(path_tflops / pk, 4)}
        if not args.chain:  # the whole step against the bound of the algorithm it runs
            roofline["step"] = tc_step_bound(w, tcf["tc_gemm_fwd"] / (24.0 * w.M1), nsm, step_mean)
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": sum(step_ms) / len(step_ms), "higher_is_better": True,
        "scaling": args.scaling, "vs_baseline": None, "dtype": args.dtype, "data": "synthetic",
        "config": {"workload": workload_label(w),
                   "parallelism": (f"replicas x{world} (independent seeded instances)" if args.scaling == "weak"
                                   else f"atoms split over {world} ranks"),
                   "step": ((f"env_mat + fwd + descriptor + fitting_fwd (M1 outputs) + {head}_head + its "
                             "backward + fitting_grad + descriptor_grad + grad + force_virial (the "
                             f"{head} model and the forces of <dE/d{head}, {head}>)")
                            if head else
                            ("env_mat + fwd + descriptor + fitting_fwd + fitting_grad + descriptor_grad + grad + "
                             "force_virial (energy and forces of the whole model)") if args.fitting else
                            "env_mat + fwd + descriptor + descriptor_grad + grad + force_virial" if args.chain
                            else "fwd + descriptor + grad" if "descriptor" in k_ms
                            else "fwd (writing D) + grad"), "algo": args.algo,
                   "fma_basis": ("interval moments: per run min(9 M1 L, 24 M1 + 24 L) fwd, "
                                 "min(18 M1 L, 24 M1 + 40 L) grad" if args.algo in ("moments", "tc")
                                 else "per row: 9 M1 fwd, 18 M1 grad"),
                   **({"tc": ("per-interval contraction on the tensor cores (f64 by exact 9-digit splitting, "
                              "fp16 MMAs); per-row work on the FP64 pipe: moments 24 FMA, derivatives 40 FMA "
                              "per valid row")} if args.algo == "tc" else {}),
                   "l2": "flushed between steps (256 MiB write)",
                   **({"fitting_gemm": ("tensor cores (tcgen05): f64 by exact 9-digit splitting, fp16 MMAs"
                                        if tc else "FP64 pipe")} if getattr(args, "fitting", False) else {}),
                   "evals_per_step_per_gpu": w.evals, "atoms_per_step_per_gpu": w.nloc, "fill": round(w.fill, 4),
                   "device_sms": nsm,
                   "footprint": footprint(w, 4 if args.dtype == "f32" else 8)},
        "atoms_per_s": w.nloc * world * args.steps / total_s,
        "roofline": roofline,
        "kernels": kernels,
        "e2e": e2e,
        # the tc fwd and grad calls count as the kernels they launched (their recorded marks)
        "gpu_launches": (len(k_ms) * args.steps + (sum(tc_launches) - 2 * args.steps if tc_launches else 0)) * world,
        "clocks": clk,
        "wall_s_timed_region": round(t_wall, 4),
    }
    if world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(w, args.dtype, args.cpu_seconds)
    return out


# ------------------------------------------------------------- oracle timing
def _oracle_pass(o, tabs, info, w, atoms, r, nthreads=0):
    s, Rt, dT = r(w.s), r(w.Rt), r(w.dT)
    T = o.fwd(tabs, info, s, Rt, w.nvalid, w.atype, w.sel, atoms=atoms, nthreads=nthreads)
    o.descriptor(T, w.M2)
    o.grad(tabs, info, s, Rt, w.nvalid, w.atype, w.sel, dT, atoms=atoms, nthreads=nthreads)


def _oracle_setup(w, dtype):
    import oracle
    o = oracle.default()
    info = o.table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    tabs = o.tables(w.params, w.widths, info)
    r = (lambda a: a)
    if dtype == "f32":
        tabs = tabs.astype(np.float32).astype(np.float64)
        r = lambda a: a.astype(np.float32).astype(np.float64)  # noqa: E731
    return o, info, tabs, r


def _cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _calibrate(o, info, tabs, w, r, target_s):
    """Atoms per oracle pass so one pass takes about target_s seconds."""
    n = min(w.nloc, 64)
    t0 = time.perf_counter()
    _oracle_pass(o, tabs, info, w, np.arange(n), r)
    dt = max(time.perf_counter() - t0, 1e-4)
    return int(max(1, min(w.nloc, n * target_s / dt)))


def cpu_baseline(w, dtype, target_s):
    """The oracle, as it stands, on all host cores: repeated passes over (a prefix of) the same workload
    until about target_s seconds of CPU work have run."""
    o, info, tabs, r = _oracle_setup(w, dtype)
    n = _calibrate(o, info, tabs, w, r, target_s)
    atoms = np.arange(n)
    ev = int(w.nvalid[:n].astype(np.int64).sum()) * w.M1
    reps, t0 = 0, time.perf_counter()
    while True:
        _oracle_pass(o, tabs, info, w, atoms, r)
        reps += 1
        dt = time.perf_counter() - t0
        if dt >= target_s:
            break
    # the same on one thread, over a shorter prefix, for about a tenth of the time
    n1 = max(1, n // max(1, _cores()))
    ev1 = int(w.nvalid[:n1].astype(np.int64).sum()) * w.M1
    reps1, t1 = 0, time.perf_counter()
    while True:
        _oracle_pass(o, tabs, info, w, np.arange(n1), r, nthreads=1)
        reps1 += 1
        dt1 = time.perf_counter() - t1
        if dt1 >= target_s / 10:
            break
    ev1 *= reps1
    return {"value": reps * ev / dt, "unit": UNIT, "cores": _cores(), "kind": "oracle",
            "sample": (f"{reps} pass(es) of fwd + descriptor + grad over the first {n} of {w.nloc} atoms of "
                       f"{w.name} ({reps * ev} evals in {dt:.1f} s)"),
            "single_thread": {"value": ev1 / dt1, "unit": UNIT, "cores": 1,
                              "sample": f"{reps1} pass(es) over the first {n1} atoms ({ev1} evals in {dt1:.1f} s)"}}


def run_reference(args, rank, world):
    """Reference arm: the oracle on the host cores, one bounded sample of the workload per step."""
    if rank != 0:
        return None
    import workloads as W
    kw = {"pad": args.pad} if args.workload == "alcumg" else {}
    w = W.make(args.workload, seed=args.seed, **kw)
    o, info, tabs, r = _oracle_setup(w, args.dtype)
    per_step = max(0.5, min(10.0, 150.0 / max(1, args.steps + args.warmup)))
    n = _calibrate(o, info, tabs, w, r, per_step)
    atoms = np.arange(n)
    for _ in range(args.warmup):
        _oracle_pass(o, tabs, info, w, atoms, r)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _oracle_pass(o, tabs, info, w, atoms, r)
    dt = time.perf_counter() - t0
    ev = int(w.nvalid[:n].astype(np.int64).sum()) * w.M1
    value = ev * args.steps / dt
    sample = f"first {n} of {w.nloc} atoms of {w.name} per step (fwd + descriptor + grad, {ev} evals)"
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": args.dtype, "data": "synthetic", "impl": "reference",
            "config": {"workload": workload_label(w), "parallelism": "host cores (oracle)",
                       "step": "fwd + descriptor + grad on a bounded atom sample"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": _cores(), "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--workload", default="cu85", choices=["tiny", "cu85", "cugeo", "water", "alcumg", "water_large"])
    ap.add_argument("--pad", type=float, default=0.3, help="alcumg padding fraction")
    ap.add_argument("--dtype", choices=["f64", "f32", "df64"], default="f64",
                    help="df64: f64 arrays, double-float arithmetic on the FP32 pipes (moment path)")
    ap.add_argument("--seed", type=int, default=2)
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="oracle CPU-baseline sample length")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end (host buffers) measurement")
    ap.add_argument("--algo", choices=["direct", "moments", "tc"], default=None,
                    help="direct: per-neighbour evaluation (the paper's fused kernel); moments: interval moments; "
                         "tc: interval moments with the per-interval contraction on the tensor cores (f64; the "
                         "default for f64)")
    ap.add_argument("--scaling", choices=["weak", "strong"], default="weak",
                    help="weak: one instance per rank; strong: one instance split over the ranks")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="with --chain: skip the CUDA-graph replay timing")
    ap.add_argument("--no-variants", action="store_true",
                    help="skip the per-row and df64 timings added to the default f64 line")
    ap.add_argument("--unfused", action="store_true",
                    help="with --chain --algo tc: the front and back end as separate kernels (dp_env_mat, "
                         "dp_force_virial) instead of fused into the tensor-core calls")
    ap.add_argument("--chain", action="store_true",
                    help="time the whole chain from coordinates to forces (env_mat ... force_virial)")
    ap.add_argument("--fitting", action="store_true",
                    help="with --chain: add the fitting net, so the step yields the model's energy and forces")
    ap.add_argument("--head", choices=["vector", "tensor"], default=None,
                    help="with --fitting: a vector or tensor model, the net's M1 outputs weighting T's "
                         "rotation-covariant rows; the backward is that of <dE/dv, v> (dE/dv synthetic)")
    ap.add_argument("--fitting-tc", action="store_true",
                    help="with --fitting and double arrays (f64, df64): the fitting net's f64 GEMMs on the tensor "
                         "cores (exact splitting)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.algo is None:  # f64: the tensor-core path; f32 and df64: the interval moments
        args.algo = "tc" if args.dtype == "f64" else "moments"
    if args.dtype == "df64" and args.algo != "moments":
        ap.error("--dtype df64 runs the moment path only")
    if args.algo == "tc" and args.dtype != "f64":
        ap.error("--algo tc is the f64 path (exact digit splitting on the tensor cores)")
    if args.fitting and not args.chain:
        ap.error("--fitting extends the --chain step")
    if args.fitting_tc and (not args.fitting or args.dtype not in ("f64", "df64")):
        ap.error("--fitting-tc needs --fitting and double arrays (--dtype f64 or df64)")
    if args.head and (not args.fitting or args.dtype == "df64"):
        ap.error("--head needs --fitting in f64 or f32")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        print(f"warning: --gpus {args.gpus} but WORLD_SIZE={world}", file=sys.stderr)
    if args.impl == "reference":
        out = run_reference(args, rank, world)
    else:
        if world > 1:
            import torch
            torch.cuda.set_device(local_rank)
            torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
        out = run_native(args, rank, world, local_rank)
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
