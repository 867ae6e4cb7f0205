"""The C-ABI library builds, loads without a GPU, and exports every function that
include/nnjit.h declares; host-only entry points behave as documented."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2309_08978_gb300.build_lib import build
    path = build()
    return ctypes.CDLL(path)


def _declared():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            src = open(os.path.join(ROOT, "include", h)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(nnjit_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert "nnjit_matmul_plan" in names and "nnjit_matmul_run" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, f"declared but not exported: {missing}"


def test_status_strings_and_version(lib):
    import paper_2309_08978_gb300 as nj
    assert nj.nnjit_status_string(0) == "NNJIT_OK"
    assert nj.nnjit_status_string(5) == "NNJIT_ERR_TIMEOUT"
    assert nj.nnjit_status_string(99) == "NNJIT_ERR_UNKNOWN"
    assert nj.nnjit_version() >= 100


def test_null_plan_arguments_are_rejected(lib):
    import paper_2309_08978_gb300 as nj
    st = nj.load_library().nnjit_matmul_run(None, None, None, None, None, None)
    assert st == nj.NNJIT_ERR_INVALID_ARG
    assert "plan" in nj.nnjit_last_error()
    assert nj.load_library().nnjit_plan_destroy(None) == nj.NNJIT_OK


def test_invalid_descriptors(lib):
    import paper_2309_08978_gb300 as nj
    from conftest_limits import gb300_limits
    L = gb300_limits()
    bad = [nj.make_desc(-1, 4, 4, "bf16"), nj.make_desc(4, 4, 4, "bf16", batch=0),
           nj.make_desc(4, 4, 4, 7), nj.make_desc(4, 4, 4, "bf16", b_layout=5),
           nj.make_desc(4, 4, 8, "bf16", lda=4), nj.make_desc(4, 8, 4, "bf16", "KN", ldb=4),
           nj.make_desc(4, 8, 4, "bf16", ldc=7), nj.make_desc(4, 4, 4, "bf16", epilogue=9),
           nj.make_desc(4, 4, 4, "bf16", epilogue=-1), nj.make_desc(4, 4, 4, "bf16", epilogue=0x14),
           nj.make_desc(4, 4, 4, "bf16", epilogue=0x30)]
    for d in bad:
        with pytest.raises(nj.NnjitError) as ei:
            nj.nnjit_space_enumerate(d, L)
        assert ei.value.status == nj.NNJIT_ERR_INVALID_ARG


def test_unaligned_tensor_core_strides_unsupported(lib):
    import paper_2309_08978_gb300 as nj
    from conftest_limits import gb300_limits
    L = gb300_limits()
    with pytest.raises(nj.NnjitError) as ei:
        nj.nnjit_space_enumerate(nj.make_desc(64, 64, 30, "bf16", "NK"), L)   # 60-byte rows
    assert ei.value.status == nj.NNJIT_ERR_UNSUPPORTED
    with pytest.raises(nj.NnjitError) as ei:
        nj.nnjit_space_enumerate(nj.make_desc(64, 30, 64, "tf32", "KN"), L)   # 120-byte rows of B
    assert ei.value.status == nj.NNJIT_ERR_UNSUPPORTED
    # the exact FFMA path takes any stride
    cands, _ = nj.nnjit_space_enumerate(nj.make_desc(64, 30, 31, "f32_ffma", "KN"), L)
    assert cands and all(c["family"] == nj.NNJIT_FAMILY_FFMA for c in cands)


def test_cache_file_format(lib, tmp_path):
    import paper_2309_08978_gb300 as nj
    nj.nnjit_cache_clear()
    empty = tmp_path / "empty.cache"
    nj.nnjit_cache_save(str(empty))
    assert empty.read_text().splitlines() == ["nnjit-plan-cache v3"]
    assert nj.nnjit_cache_load(str(empty)) == 0
    bad = tmp_path / "bad.cache"
    bad.write_text("something else\n")
    with pytest.raises(nj.NnjitError) as ei:
        nj.nnjit_cache_load(str(bad))
    assert ei.value.status == nj.NNJIT_ERR_INVALID_ARG
    # a well-formed entry round-trips through load and save
    entry = ("t=matmul|s=1,2,3,1|dt=2|bl=1|ld=3,3,2|st=3,6,2|bias=0|dev=X,cc103,sm152\t"
             "1 128 256 64 0 0 4 1 0 192 230656 512 72 1 1 1000000 2 9 0 1\t0 6 336 12.5 1\t2 0 3.5 1 4.25\n")
    good = tmp_path / "good.cache"
    good.write_text("nnjit-plan-cache v3\n" + entry)
    assert nj.nnjit_cache_load(str(good)) == 1
    assert nj.nnjit_cache_size() == 1
    out = tmp_path / "out.cache"
    nj.nnjit_cache_save(str(out))
    lines = out.read_text().splitlines()
    assert lines[0] == "nnjit-plan-cache v3" and lines[1].split("\t")[0] == entry.split("\t")[0]
    assert lines[1].split("\t")[1] == entry.split("\t")[1]
    nj.nnjit_cache_clear()
    assert nj.nnjit_cache_size() == 0


def test_w4_layout_matches_the_documented_blob(lib):
    import paper_2309_08978_gb300 as nj
    # code block N * ldb / 2 bytes rounded up to 256, then ceil(K / 128) * N bf16 scales
    assert nj.nnjit_w4_layout(4096, 11008) == (4096 * 5504, 4096 * 5504 + 86 * 4096 * 2)
    assert nj.nnjit_w4_layout(8, 200, 224) == (1024, 1024 + 2 * 8 * 2)
    assert nj.nnjit_w4_layout(24, 32) == (512, 512 + 24 * 2)
    for bad in ((4096, 4096, 4100), (4096, 100, 0), (1004, 4096, 0), (8, 64, 32)):
        with pytest.raises(nj.NnjitError) as ei:
            nj.nnjit_w4_layout(*bad)
        assert ei.value.status == nj.NNJIT_ERR_INVALID_ARG


def test_settings_roundtrip_and_validation(lib):
    """nnjit_settings_set/get: values round-trip, out-of-range values are refused without
    changing the current settings, NULL clears (host only)."""
    import paper_2309_08978_gb300 as nj
    assert nj.nnjit_settings_get() == {"raster": -1, "kgroup": -1, "reduce": -1}
    try:
        nj.nnjit_settings_set({"raster": 1, "reduce": 0})
        assert nj.nnjit_settings_get() == {"raster": 1, "kgroup": -1, "reduce": 0}
        # every reduction a candidate can carry is a legal fixed value (a settings study may
        # vote for the CTA-pair stream-K one, 2)
        nj.nnjit_settings_set({"raster": 1, "reduce": 2})
        assert nj.nnjit_settings_get() == {"raster": 1, "kgroup": -1, "reduce": 2}
        nj.nnjit_settings_set({"raster": 1, "reduce": 0})
        for bad in ({"kgroup": 0}, {"kgroup": 3}, {"raster": 2}, {"reduce": -2}, {"reduce": 3}, {"reduce": 5}):
            with pytest.raises(nj.NnjitError) as ei:
                nj.nnjit_settings_set(bad)
            assert ei.value.status == nj.NNJIT_ERR_INVALID_ARG
        assert nj.nnjit_settings_get() == {"raster": 1, "kgroup": -1, "reduce": 0}
    finally:
        nj.nnjit_settings_set(None)
    assert nj.nnjit_settings_get()["raster"] == -1


def test_attention_refusals_without_a_gpu(lib):
    """nnjit_attention checks its descriptor and pointers before any CUDA call: invalid
    sizes, flags, kernels and NULL pointers give INVALID_ARG, an unsupported head dimension
    or a pointer off a 16-byte boundary UNSUPPORTED, and Lq = 0 returns OK with nothing to
    do.  The pointers are never dereferenced on these paths."""
    import paper_2309_08978_gb300 as nj
    f = nj.load_library().nnjit_attention
    p = 1 << 20  # a 16-byte-aligned address, never touched
    cases = (((1, 4, 4, 96, 0, 1.0), nj.NNJIT_ERR_UNSUPPORTED), ((0, 4, 4, 64, 0, 1.0), nj.NNJIT_ERR_INVALID_ARG),
             ((1, 4, 4, 64, 2, 1.0), nj.NNJIT_ERR_INVALID_ARG), ((1, -1, 4, 64, 0, 1.0), nj.NNJIT_ERR_INVALID_ARG),
             ((1, 4, -2, 64, 0, 1.0), nj.NNJIT_ERR_INVALID_ARG),
             ((1, 4, 4, 64, 0, float("nan")), nj.NNJIT_ERR_INVALID_ARG),
             ((1, 4, 4, 64, 0, 1.0, 4), nj.NNJIT_ERR_INVALID_ARG), ((1, 4, 4, 64, 0, 1.0, -1), nj.NNJIT_ERR_INVALID_ARG))
    for d, st in cases:
        assert f(nj.nnjit_attention_desc(*d), p, p, p, p, None) == st, d
    desc = nj.nnjit_attention_desc(1, 4, 4, 64, 0, 1.0)
    assert f(desc, p + 4, p, p, p, None) == nj.NNJIT_ERR_UNSUPPORTED
    assert f(desc, p, p, p, p + 8, None) == nj.NNJIT_ERR_UNSUPPORTED
    assert f(desc, None, p, p, p, None) == nj.NNJIT_ERR_INVALID_ARG
    assert f(desc, p, None, p, p, None) == nj.NNJIT_ERR_INVALID_ARG
    assert f(None, p, p, p, p, None) == nj.NNJIT_ERR_INVALID_ARG
    assert f(nj.nnjit_attention_desc(2, 0, 5, 128, 1, 1.0), None, None, None, None, None) == nj.NNJIT_OK


def test_run_host_seq_refusals_without_a_gpu(lib):
    """nnjit_matmul_run_host_seq checks its arrays before any CUDA call: a negative count or
    NULL arrays are INVALID_ARG, and count 0 is a no-op."""
    import ctypes
    import paper_2309_08978_gb300 as nj
    f = nj.load_library().nnjit_matmul_run_host_seq
    assert f(0, None, None, None, None, None, None) == nj.NNJIT_OK
    assert f(-1, None, None, None, None, None, None) == nj.NNJIT_ERR_INVALID_ARG
    assert f(2, None, None, None, None, None, None) == nj.NNJIT_ERR_INVALID_ARG
    assert "NULL" in nj.nnjit_last_error()
