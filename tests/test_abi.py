"""The C ABI library loads, exports every symbol include/dp_compress.h declares, and validates
arguments on the host before any CUDA call (CPU only: nothing here launches a kernel)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dp_compress.h")


@pytest.fixture(scope="module")
def dpc():
    import __graft_entry__
    __graft_entry__._load_builder().build()
    import paper_2107_02103_gb300 as m
    return m


def declared():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:int|size_t|const char \*)\s*(dp_\w+)\s*\(", src, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared()
    for required in ("dp_table_build_f64", "dp_tabulate_fusion_fwd_f64", "dp_tabulate_fusion_grad_f64",
                     "dp_descriptor_contract_f64", "dp_tabulate_fusion_fwd_f32", "dp_tabulate_fusion_grad_f32"):
        assert required in names


def test_every_declared_symbol_is_exported(dpc):
    lib = ctypes.CDLL(dpc.LIB_PATH)
    missing = [n for n in declared() if not hasattr(lib, n)]
    assert not missing, missing
    assert sorted(dpc.EXPORTS) == declared()


def test_header_compiles_as_c(tmp_path):
    c = tmp_path / "t.c"
    c.write_text('#include "dp_compress.h"\nint main(void){ dp_table_info i; (void)i; return DP_OK; }\n')
    import subprocess
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), "-c", str(c), "-o",
                    str(tmp_path / "t.o")], check=True)


def test_table_info_host_rules(dpc):
    import oracle
    o = oracle.default()
    for smin, smax in ((0.0, 1.05), (-0.237, 0.42), (0.2, 0.2)):
        a = dpc.dp_table_info_make(smin, smax)
        b = o.table_info(smin, smax)
        assert (a.lower, a.upper, a.upper_ext, a.stride0, a.stride1) == b.as_tuple()
        assert dpc.dp_table_info_sizes(a) == (b.n0, b.n1)
    with pytest.raises(dpc.DPError) as e:
        dpc.dp_table_info_make(0.0, -1.0)
    assert e.value.code == dpc.DP_ERR_TABLE_INFO
    with pytest.raises(dpc.DPError) as e:
        dpc.dp_table_info_make(0.0, 1.0, 0.03, 0.1)  # stride1/stride0 not integral
    assert e.value.code == dpc.DP_ERR_TABLE_INFO
    bad = dpc.dp_table_info(lower=0.0, upper=1.0, upper_ext=5.0, stride0=0.03, stride1=0.1)
    with pytest.raises(dpc.DPError) as e:
        dpc.dp_table_info_sizes(bad)
    assert e.value.code == dpc.DP_ERR_TABLE_INFO and "stride0" in str(e.value)


def _call(lib, name, *args):
    return getattr(lib, name)(*args)


def test_validation_codes_without_gpu(dpc):
    """Every check below fails before the library touches CUDA; the fake pointers are never dereferenced."""
    lib = dpc._lib
    info = dpc.dp_table_info_make(0.0, 1.05)
    fake = ctypes.c_void_p(0x1000)
    sel = (ctypes.c_int32 * 2)(3, 4)
    args = lambda **kw: dict(dict(table=fake, s=fake, Rt=fake, nloc=5, nnei=7, ntypes=2, sel=sel, M1=16, T=fake),  # noqa: E731
                              **kw)

    def fwd(**kw):
        a = args(**kw)
        return lib.dp_tabulate_fusion_fwd_f64(a["table"], ctypes.byref(info), a["s"], a["Rt"], None, None, a["nloc"],
                                              a["nnei"], a["ntypes"], a["sel"], a["M1"], a["T"], None)

    assert fwd(table=None) == dpc.DP_ERR_NULL
    assert fwd(T=None) == dpc.DP_ERR_NULL
    assert fwd(nloc=-1) == dpc.DP_ERR_SHAPE
    assert fwd(nnei=8) == dpc.DP_ERR_SHAPE and "sum(sel)" in dpc.dp_last_error()
    assert fwd(M1=0) == dpc.DP_ERR_SHAPE
    assert fwd(M1=257) == dpc.DP_ERR_UNSUPPORTED
    assert fwd(ntypes=9, sel=(ctypes.c_int32 * 9)(*([1] * 9)), nnei=9) == dpc.DP_ERR_UNSUPPORTED
    assert fwd(ntypes=0) == dpc.DP_ERR_SHAPE
    assert fwd(sel=None) == dpc.DP_ERR_NULL
    assert fwd(nloc=0) == dpc.DP_OK  # empty input: nothing enqueued
    badinfo = dpc.dp_table_info(lower=0.0, upper=-1.0, upper_ext=5.0, stride0=0.01, stride1=0.1)
    assert lib.dp_tabulate_fusion_fwd_f64(fake, ctypes.byref(badinfo), fake, fake, None, None, 5, 7, 2, sel, 16, fake,
                                          None) == dpc.DP_ERR_TABLE_INFO
    assert lib.dp_tabulate_fusion_grad_f64(fake, ctypes.byref(info), fake, fake, None, None, 5, 7, 2, sel, 16, None,
                                           fake, fake, None) == dpc.DP_ERR_NULL
    assert lib.dp_descriptor_contract_f64(fake, 5, 16, 17, fake, None) == dpc.DP_ERR_SHAPE
    assert lib.dp_descriptor_contract_f32(fake, 5, 16, 0, fake, None) == dpc.DP_ERR_SHAPE
    assert lib.dp_descriptor_contract_f64(None, 5, 16, 4, fake, None) == dpc.DP_ERR_NULL
    assert lib.dp_table_build_f64(fake, fake, None, 1, 16, ctypes.byref(info), fake, None) == dpc.DP_ERR_NULL
    assert lib.dp_table_build_f32(fake, fake, fake, 0, 16, ctypes.byref(info), fake, None) == dpc.DP_ERR_SHAPE
    w = (ctypes.c_int32 * 3)(2, 4, 8)
    assert lib.dp_embedding_net_nodes_f64(fake, w, 2, 1, ctypes.byref(info), fake, fake, fake, None) == dpc.DP_ERR_SHAPE
    w = (ctypes.c_int32 * 3)(1, 4, 2000)
    assert lib.dp_embedding_net_nodes_f64(fake, w, 2, 1, ctypes.byref(info), fake, fake, fake,
                                          None) == dpc.DP_ERR_UNSUPPORTED
    assert dpc.dp_last_error() != ""
    env = dpc.env_info(0.5, 6.0)
    assert lib.dp_env_mat_f64(fake, fake, -1, 7, 2, sel, ctypes.byref(env), fake, fake, fake, None) == dpc.DP_ERR_SHAPE
    assert lib.dp_env_mat_f64(fake, fake, 5, 8, 2, sel, ctypes.byref(env), fake, fake, fake, None) == dpc.DP_ERR_SHAPE
    assert lib.dp_env_mat_f32(fake, fake, 5, 7, 2, sel, None, fake, fake, fake, None) == dpc.DP_ERR_NULL
    for bad in (dpc.env_info(6.0, 0.5), dpc.env_info(0.0, 6.0), dpc.env_info(0.5, 6.0, kind=2),
                dpc.env_info(0.5, 6.0, norm=(0.0, 0.0, 1.0)), dpc.env_info(0.5, 6.0, norm=(0.0, 1.0, -1.0))):
        assert lib.dp_env_mat_f64(fake, fake, 5, 7, 2, sel, ctypes.byref(bad), fake, fake, fake,
                                  None) == dpc.DP_ERR_TABLE_INFO
    assert lib.dp_env_mat_f64(None, None, 0, 7, 2, sel, ctypes.byref(env), None, None, None, None) == dpc.DP_OK
    assert lib.dp_env_mat_f64(None, fake, 5, 7, 2, sel, ctypes.byref(env), fake, fake, fake, None) == dpc.DP_ERR_NULL
    fv = lib.dp_force_virial_f64
    assert fv(fake, fake, 5, 4, 7, ctypes.byref(env), fake, fake, fake, fake, None) == dpc.DP_ERR_SHAPE  # nall < nloc
    assert fv(fake, fake, 5, 9, 0, ctypes.byref(env), fake, fake, fake, fake, None) == dpc.DP_ERR_SHAPE
    assert fv(fake, fake, 5, 9, 7, ctypes.byref(env), fake, fake, fake, None, None) == dpc.DP_ERR_NULL
    assert fv(fake, None, 5, 9, 7, ctypes.byref(env), fake, fake, fake, fake, None) == dpc.DP_ERR_NULL
    bad = dpc.env_info(0.5, 6.0, kind=3)
    assert fv(fake, fake, 5, 9, 7, ctypes.byref(bad), fake, fake, fake, fake, None) == dpc.DP_ERR_TABLE_INFO


def test_binding_rejects_cpu_tensors(dpc):
    import torch
    info = dpc.dp_table_info_make(0.0, 1.05)
    with pytest.raises(TypeError):
        dpc.dp_tabulate_fusion_fwd(torch.zeros(1, 10, 4, 6, dtype=torch.float64), info,
                                   torch.zeros(2, 3, dtype=torch.float64), torch.zeros(2, 3, 4, dtype=torch.float64),
                                   None, None, [3])


def test_tc_plan_and_work_validation_without_gpu(dpc):
    """The tensor-core calls refuse, on the host and before any CUDA call, a missing plan, a plan made for
    another geometry or too short, a missing, short or misaligned work buffer, and unknown flags; the
    plan builder refuses a missing, short or misaligned buffer.  The fake pointers are never dereferenced."""
    lib = dpc._lib
    info = dpc.dp_table_info_make(0.0, 1.05)
    fake = ctypes.c_void_p(0x1000)
    sel = (ctypes.c_int32 * 1)(8)
    need = dpc.dp_tabulate_tc_plan_bytes(info, 8, 1, 16)
    wb = dpc.dp_tabulate_tc_work_bytes(info, 5, 8, 1, 16)

    def plan(**kw):
        d = dict(data=0x1000, bytes=need, info=info, nnei=8, ntypes=1, M1=16)
        d.update(kw)
        return dpc.dp_tc_plan(**d)

    def fwd(rec, work=fake, nbytes=wb, M2=0, D=None):
        return lib.dp_tabulate_fusion_fwd_tc_f64(None if rec is None else ctypes.byref(rec), ctypes.byref(info), fake,
                                                 fake, None, None, 5, 8, 1, sel, 16, fake, M2, D, work, nbytes, None)

    def grad(rec, flags=0, work=fake, nbytes=wb):
        return lib.dp_tabulate_fusion_grad_tc_f64(None if rec is None else ctypes.byref(rec), ctypes.byref(info),
                                                  fake, fake, None, None, 5, 8, 1, sel, 16, fake, fake, fake, work,
                                                  nbytes, flags, None)

    assert fwd(None) == dpc.DP_ERR_NULL and grad(None) == dpc.DP_ERR_NULL
    assert fwd(plan(data=None)) == dpc.DP_ERR_NULL
    other = dpc.dp_table_info_make(0.0, 1.25)
    for bad in (plan(nnei=9), plan(M1=32), plan(bytes=need - 1), plan(info=other)):
        assert fwd(bad) == dpc.DP_ERR_SHAPE and grad(bad) == dpc.DP_ERR_SHAPE
    assert fwd(plan(), work=None) == dpc.DP_ERR_NULL
    assert fwd(plan(), nbytes=wb - 1) == dpc.DP_ERR_SHAPE
    assert fwd(plan(), work=ctypes.c_void_p(0x1010)) == dpc.DP_ERR_SHAPE
    assert grad(plan(), flags=2) == dpc.DP_ERR_SHAPE and "flags" in dpc.dp_last_error()
    for bad_m2 in (0, 17):  # the descriptor's M2 outside 1 .. M1 (16), refused on the host
        assert fwd(plan(), M2=bad_m2, D=fake) == dpc.DP_ERR_SHAPE and "M2" in dpc.dp_last_error()
    rec = dpc.dp_tc_plan()
    build = lambda buf, n: lib.dp_tabulate_tc_plan_f64(fake, ctypes.byref(info), 8, 1, 16, buf, n,  # noqa: E731
                                                       ctypes.byref(rec), None)
    assert build(None, need) == dpc.DP_ERR_NULL
    assert build(fake, need - 1) == dpc.DP_ERR_SHAPE
    assert build(ctypes.c_void_p(0x1010), need) == dpc.DP_ERR_SHAPE
