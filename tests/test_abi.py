"""The C-ABI library loads on a machine without a GPU, exports every entry
point include/goldy.h declares, and its host-only calls validate arguments
(no compute call is made here)."""
import ctypes
import os
import re

import pytest

from paper_2409_02227_gb300 import goldy as G

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "goldy.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(goldy_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("goldy_plan", "goldy_run", "goldy_schedule_query", "goldy_lut_load",
                 "goldy_graph_create", "goldy_last_error"):
        assert must in names


def test_every_declared_symbol_is_exported():
    lib = ctypes.CDLL(G.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_version_and_registry():
    assert G.goldy_abi_version() == 2
    n = G.goldy_variant_count()
    assert n == 132
    seen = set()
    for v in range(n):
        info = G.goldy_variant_info_get(v)
        assert info["id"] == v and info["mma_m"] == 128 * info["cta_pair"]
        assert info["split_k"] in (1, 2, 4, 8) and info["rc_div"] in (1, 2, 4)
        assert info["tmem_cols"] in (32, 64, 128, 256, 512)
        assert info["tmem_cols"] >= info["mma_n"] * info["acc_stages"]
        # footprint: "half" kinds leave room for a second CTA on the SM
        if info["ctas_per_sm"] == 2:
            assert info["smem_bytes"] <= 113 * 1024 and info["tmem_cols"] <= 256
        assert info["smem_bytes"] <= 227 * 1024
        seen.add((info["kind"], info["split_k"], info["rc_div"]))
    assert len(seen) == n                   # every id a distinct (kind, split, grid cap)
    with pytest.raises(G.GoldyError) as e:
        G.goldy_variant_info_get(n)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG


def _lut_bytes():
    from oracle import planner_ref as pr
    return pr.write_lut([pr.Entry((8, 8, 9, 1), 2, (0, 1, 2, 3, 4))], 120)


def test_plan_error_paths():
    lut = G.goldy_lut_from_memory(_lut_bytes())
    d = G.desc(256, 256, 512)
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([], lut)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([d] * 65, lut)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([d], lut, G.GOLDY_PLAN_FORCE_CD)        # forced CD missing
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([d], lut, 0x10000)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([d], None)
    assert e.value.status == G.GOLDY_ERR_LUT
    bad = G.desc(256, 256, 512)
    bad.trans_a = 1
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([bad], lut)
    assert e.value.status == G.GOLDY_ERR_UNSUPPORTED
    bad = G.desc(256, 256, 512)
    bad.a_dtype = G.GOLDY_F32
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([bad], lut)
    assert e.value.status == G.GOLDY_ERR_UNSUPPORTED
    bad = G.desc(256, 256, 512, lda=516)                      # 516 * 2 bytes is not a 16-byte row
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([bad], lut)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    bad = G.desc(256, 256, 512, ldc=100)                      # ldc < N
    with pytest.raises(G.GoldyError) as e:
        G.goldy_plan([bad], lut)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    assert "leading dimension" in G.goldy_last_error()
    bad = G.desc(-1, 256, 512)
    with pytest.raises(G.GoldyError):
        G.goldy_plan([bad], lut)


def test_lut_error_paths(tmp_path):
    with pytest.raises(G.GoldyError) as e:
        G.goldy_lut_from_memory(b"GOLDYLUX" + bytes(24))
    assert e.value.status == G.GOLDY_ERR_LUT
    with pytest.raises(G.GoldyError) as e:
        G.goldy_lut_load(str(tmp_path / "missing.bin"))
    assert e.value.status == G.GOLDY_ERR_LUT
    data = bytearray(_lut_bytes())
    data[16] = 133                                            # variant bound beyond this library
    with pytest.raises(G.GoldyError):
        G.goldy_lut_from_memory(bytes(data))
    p = tmp_path / "ok.bin"
    p.write_bytes(_lut_bytes())
    G.goldy_lut_load(str(p))


def test_schedule_build_and_query():
    descs = [G.desc(256, 256, 512), G.desc(128, 1024, 4096, G.GOLDY_BF16), G.desc(32, 4096, 1024)]
    s = G.goldy_schedule_build(descs, [0, 0, 1], [0, 9, 80], [0, 3, 0])
    n, ng, ms, ws = G.goldy_schedule_query(s)
    assert (n, ng, ms) == (3, 2, 4)
    assert G.goldy_schedule_entry(s, 1) == (0, 9, 3, 2)
    assert G.goldy_schedule_entry(s, 2) == (1, 80, 0, 1)
    # variant 9 = kind 0 (128 x 64 tiles), split 8: 128 x 1024 -> 16 tiles x 8 splits;
    # variant 80 = kind 6 (transposed 32 x 128 tiles), split 4: 32 x 4096 -> 32 tiles x 4
    part1 = 16 * 8 * 128 * 64 * 4
    part2 = 32 * 4 * 128 * 32 * 4
    assert ws == (part1 + 256) + (part2 + 256)
    with pytest.raises(G.GoldyError):
        G.goldy_schedule_build(descs, [0, 2, 2], [0, 0, 0], [0, 0, 0])   # group 1 empty
    with pytest.raises(G.GoldyError):
        G.goldy_schedule_build(descs, [0, 0, 0], [0, 0, 132], [0, 0, 0])
    with pytest.raises(G.GoldyError):
        G.goldy_schedule_build(descs, [0, 0, 0], [0, 0, 0], [0, 0, 16])
    with pytest.raises(G.GoldyError):
        G.goldy_schedule_entry(s, 3)
    with pytest.raises(G.GoldyError):
        G.goldy_schedule_build(descs, [0, 0, 1], [0, 9, 80], [0, 3, 0], flags=1)
    f = G.goldy_schedule_build(descs, [0, 0, 1], [0, 9, 80], [0, 3, 0], flags=G.GOLDY_PLAN_FUSED)
    assert G.goldy_schedule_serialize(f)[20:24] == bytes([0x10, 0, 0, 0])


def test_bucket_key_matches_reference():
    from oracle import planner_ref as pr
    for (M, N, K, c) in [(256, 256, 512, 1), (1, 1, 1, 0), (0, 0, 0, 1), (4095, 8193, 64, 0),
                         (2 ** 30, 3, 5, 1)]:
        d = G.desc(M, N, K, c, lda=max(8, (K + 7) // 8 * 8), ldb=max(8, (N + 7) // 8 * 8), ldc=max(N, 1))
        lm, ln, lk, out = pr.bucket_key(M, N, K, c)
        assert G.goldy_bucket_key(d) == (lm << 24) | (ln << 16) | (lk << 8) | out


def test_partition_and_exec_error_paths():
    # no GPU here: creating a partition fails with a status, never a crash
    with pytest.raises(G.GoldyError) as ei:
        G.goldy_partition_create(38, 4)
    assert ei.value.status in (G.GOLDY_ERR_UNSUPPORTED, G.GOLDY_ERR_CUDA)
    lib = G._lib
    import ctypes
    out = ctypes.c_void_p()
    assert lib.goldy_partition_create(38, 0, ctypes.byref(out)) == G.GOLDY_ERR_INVALID_ARG
    assert lib.goldy_partition_create(38, 17, ctypes.byref(out)) == G.GOLDY_ERR_INVALID_ARG
    assert lib.goldy_partition_create(38, 4, None) == G.GOLDY_ERR_INVALID_ARG
    sm = ctypes.c_int()
    assert lib.goldy_partition_query(None, ctypes.byref(sm), None, 0) == G.GOLDY_ERR_INVALID_ARG
    lib.goldy_partition_free(None)
    ms = ctypes.c_float()
    assert lib.goldy_exec_time(None, 1, 0, 1, ctypes.byref(ms)) == G.GOLDY_ERR_INVALID_ARG
    assert lib.goldy_exec_launch(None) == G.GOLDY_ERR_INVALID_ARG
    lib.goldy_exec_free(None)


def test_packaged_tables_and_predictor_load():
    import glob
    import os
    from oracle import planner_ref as pr
    from oracle import predictor_ref as P
    paths = [G.DEFAULT_LUT] + sorted(glob.glob(os.path.join(os.path.dirname(G.DEFAULT_LUT), "scaling", "*.bin")))
    assert len(paths) >= 4
    for p in paths:
        data = open(p, "rb").read()
        G.goldy_lut_from_memory(data)
        pr.parse_lut(data)
    m = open(G.DEFAULT_PREDICTOR, "rb").read()
    G.goldy_predictor_from_memory(m)
    assert P.parse_model(m).sm_count == 152


def test_fused_schedules_reserve_unit_counters():
    # a fused schedule of several GEMMs reserves 8 bytes of unit counters per
    # GEMM (256-byte aligned) after the split-K regions; other schedules none
    descs = [G.desc(256, 256, 512), G.desc(128, 512, 256), G.desc(64, 256, 1024)]
    v = G.variant_id(0, 1, 1)                      # no split-K: no partial regions
    plain = G.goldy_schedule_build(descs, [0, 0, 0], [v] * 3, [0, 1, 2])
    fused = G.goldy_schedule_build(descs, [0, 0, 0], [v] * 3, [0, 1, 2], G.GOLDY_PLAN_FUSED)
    one = G.goldy_schedule_build(descs[:1], [0], [v], [0], G.GOLDY_PLAN_FUSED)
    assert G.goldy_schedule_query(plain)[3] == 0
    assert G.goldy_schedule_query(one)[3] == 0
    assert G.goldy_schedule_query(fused)[3] == 256
    vs = G.variant_id(0, 2, 1)                     # split 2 on the first GEMM
    split = G.goldy_schedule_build(descs, [0, 0, 0], [vs, v, v], [0, 1, 2])
    split_fused = G.goldy_schedule_build(descs, [0, 0, 0], [vs, v, v], [0, 1, 2], G.GOLDY_PLAN_FUSED)
    assert G.goldy_schedule_query(split_fused)[3] == G.goldy_schedule_query(split)[3] + 256
