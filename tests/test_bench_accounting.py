"""The bench's FMA accounting for the interval-moment path (CPU only): run lengths against a
row-by-row walk, and the per-run cost rule on hand-made runs."""
import math

import numpy as np

import bench
import oracle
import workloads as W


def _walk_runs(w, info):
    """Row by row: a new run starts at every atom, type segment or interval change."""
    off = np.concatenate([[0], np.cumsum(w.sel)])
    runs = []
    for i in range(w.nloc):
        prev, n = None, 0
        for b in range(w.ntypes):
            for j in range(int(w.nvalid[i, b])):
                x = float(w.s[i, off[b] + j])
                if x < info.lower:
                    l = 0
                elif x < info.upper:
                    l = min(int(math.floor((x - info.lower) / info.stride0)), info.n0 - 1)
                elif x < info.upper_ext:
                    l = info.n0 + min(int(math.floor((x - info.upper) / info.stride1)), info.n1 - 1)
                else:
                    l = info.n0 + info.n1 - 1
                if (b, l) == prev:
                    n += 1
                else:
                    if n:
                        runs.append(n)
                    prev, n = (b, l), 1
        if n:
            runs.append(n)
    return np.array(runs)


def test_interval_runs_match_a_row_walk():
    o = oracle.default()
    for w in (W.water(seed=3, nmol=128), W.tiny(seed=4, nloc=17, nreal=29, sel=31, rmin=2.6, rmax=3.0)):
        info = o.table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
        s = w.s.copy()
        s[0, 0], s[1, 1] = info.upper_ext + 1.0, info.lower - 1.0  # clamped rows join the end intervals
        w = W.Workload(**{**w.__dict__, "s": s})
        got = bench.interval_runs(w, info, info.n0, info.n1)
        ref = _walk_runs(w, info)
        assert np.array_equal(got, ref)
        assert got.sum() == int(w.nvalid.sum())


def test_moment_fmas_take_the_cheaper_form():
    M1 = 100
    runs = np.array([1, 2, 3, 10, 400])
    f = bench.moment_fmas(runs, M1)
    fwd = sum(min(9 * M1 * L, 24 * M1 + 24 * L) for L in runs)
    grad = sum(min(18 * M1 * L, 24 * M1 + 40 * L) for L in runs)
    assert f == {"fwd": float(fwd), "grad": float(grad)}
    # singletons stay per row, long runs go through moments
    assert bench.moment_fmas(np.array([1]), M1)["fwd"] == 9 * M1
    assert bench.moment_fmas(np.array([400]), M1)["grad"] == 24 * M1 + 40 * 400


def test_footprint_counts_every_array():
    """Bytes per atom of the pass: s and R~ in, ds and dR~ out (5 values per row each way), T and dT
    (4 M1 each), D (M1 M2), two int32 arrays; the uncompressed model adds every layer output per row."""
    w = W.tiny()
    f = bench.footprint(w, 8)
    assert f["bytes_per_atom"] == 8 * (10 * 32 + 8 * 32 + 32 * 4) + 4 * 2
    assert f["uncompressed_extra_bytes_per_atom"] == 8 * 32 * (8 + 16 + 32)
    assert f["atoms_per_280GB"] > f["atoms_per_280GB_uncompressed"] > 0


def test_tensor_core_path_accounting():
    """--algo tc: the FP64 kernels' FMAs per valid row (moments 24, rows 40), the GEMMs' 24 M1 per
    run, and enough timing events per step for every kernel mark of every chunk and centre type."""
    w = W.tiny(seed=5, nloc=9, nreal=13, sel=16, widths=(1, 4, 8), M2=4)
    rows = int(w.nvalid.sum())
    runs = np.array([3, 5, 5])
    f = bench.tc_fmas(w, runs)
    assert f["tc_runs_moments"] == 24 * rows and f["tc_rows"] == 40 * rows
    assert f["tc_gemm_fwd"] == f["tc_gemm_grad"] == 24 * w.M1 * len(runs)
    assert w.evals == rows * w.M1
    for nloc, ntypes in ((100, 1), (4104, 1), (4105, 2), (12288, 2), (32768, 3), (1048576, 2)):
        chunks = -(-nloc // bench.TC_CHUNK_ATOMS)
        marks = 2 + 2 + chunks * ((2 + 2 * ntypes) + (2 + ntypes + 1))  # starts, coefficients, per chunk
        ww = W.Workload(**{**w.__dict__, "s": np.zeros((nloc, 1)), "ntypes": ntypes})
        assert bench.tc_profile_events(ww) >= min(marks, 4096)


def test_report_takes_the_roofline_on_the_dominant_tc_kernel():
    """report() with per-kernel times from the tc calls: the roofline names the dominant kernel with
    its own algorithmic FLOPs and peak (FP64 for the rows and moments kernels, the tensor peak and 45
    digit products for a GEMM), and the launch count includes the kernels inside the calls."""
    import argparse
    w = W.tiny(seed=5, nloc=9, nreal=13, sel=16, widths=(1, 4, 8), M2=4)
    args = argparse.Namespace(dtype="f64", algo="tc", steps=2, warmup=3, scaling="weak", chain=False,
                              fitting=False, fitting_tc=False, no_cpu_baseline=True)
    runs = np.array([3, 5, 5])
    tcf = bench.tc_fmas(w, runs)
    step_ms = [1.0, 1.0]
    k_ms = {"fwd": [0.4, 0.4], "descriptor": [0.1, 0.1], "grad": [0.5, 0.5]}
    for dom, ms in (("tc_rows", 0.3), ("tc_gemm_grad", 0.45)):
        tc_ms = {"tc_runs_moments": [0.2, 0.2], "tc_gemm_fwd": [0.1, 0.1], "tc_rows": [0.3, 0.3],
                 "tc_gemm_grad": [0.05, 0.05]}
        tc_ms[dom] = [ms, ms]
        out = bench.report(args, w, 1, step_ms, k_ms, 2e-3, float(w.evals), None, None, 0.01,
                           bench.moment_fmas(runs, w.M1), 0, tc_ms, tcf, [16, 16])
        r = out["roofline"]
        assert r["kernel"] == bench.TC_KERNEL[dom]
        if dom == "tc_rows":
            assert r["bound"] == "alu"
            assert abs(r["achieved"] - 2 * 40 * w.evals / w.M1 / (ms * 1e-3) / 1e12) < 1e-3
            assert r["peak"] == round(bench.peak_tflops("f64"), 4)
        else:
            assert r["bound"] == "tensor"
            assert abs(r["achieved"] - 45 * 2 * 24 * w.M1 * len(runs) / (ms * 1e-3) / 1e12) < 0.02
            assert r["peak"] == round(bench.tensor_peak()[0], 1)
        assert "tensor_frac" in out["kernels"]["tc_gemm_fwd"] and "frac" in out["kernels"]["tc_rows"]
        assert out["gpu_launches"] == 3 * 2 + 16 * 2 - 2 * 2
        # the step against the bound of the algorithm it runs: FP64 per-row work and D, digit products, bytes
        st = r["step"]
        rows = w.evals / w.M1
        fp64_ms = 2 * (64 * rows + 4 * w.M1 * w.M2 * w.nloc) / (bench.peak_tflops("f64") * 1e12) * 1e3
        tensor_ms = 45 * 2 * 2 * 24 * w.M1 * len(runs) / (bench.tensor_peak()[0] * 1e12) * 1e3
        nbytes = 8 * (2 * 5 * rows + 3 * 4 * w.M1 * w.nloc + w.M1 * w.M2 * w.nloc + 5 * w.nloc * w.nnei)
        hbm_ms = nbytes / (bench.hbm_peak()[0] * 1e9) * 1e3
        assert abs(st["fp64_ms"] - fp64_ms) < 1e-4 and abs(st["tensor_ms"] - tensor_ms) < 1e-4
        assert abs(st["hbm_ms"] - hbm_ms) < 1e-4
        assert st["t_roof_ms"] == max(st["fp64_ms"], st["tensor_ms"], st["hbm_ms"])
        assert abs(st["frac"] - st["t_roof_ms"] / 1.0) < 1e-4


def test_head_options_and_their_fitting_net(monkeypatch):
    """--head needs the fitting net of the chain, in f64 or f32 (refused before any device work
    otherwise), and its net ends in M1 outputs, the head's weights, where the energy model's in one."""
    import pytest
    for argv in (["--head", "vector"], ["--chain", "--head", "tensor"],
                 ["--chain", "--fitting", "--dtype", "df64", "--head", "vector"]):
        monkeypatch.setattr("sys.argv", ["bench.py", *argv])
        with pytest.raises(SystemExit) as e:
            bench.main()
        assert e.value.code == 2, argv
    w = W.tiny()
    we, pe = bench.fitting_model(w)
    wv, pv = bench.fitting_model(w, "vector")
    assert we[-1] == 1 and wv[-1] == w.M1 and we[:-1] == wv[:-1]
    P = sum((wv[l - 1] + 1) * wv[l] for l in range(1, len(wv)))
    assert pv.shape == (w.ntypes, P)
