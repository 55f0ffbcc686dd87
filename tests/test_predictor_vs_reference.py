"""The C++ predictor path (goldy_lr_features, goldy_predict_cd, goldy_plan_ex)
against the independent restatement in oracle/predictor_ref.py: identical
features, identical predictions (both sides decide in IEEE double, in the
same order, without fused multiply-add), Eq. 1 probabilities to rounding,
byte-identical schedules, and rejection of malformed model files."""
import ctypes
import random

import pytest

from oracle import planner_ref as pr
from oracle import predictor_ref as P
from paper_2409_02227_gb300 import goldy as G

NV = 132


def random_lut(rng, n_entries):
    keys = set()
    while len(keys) < n_entries:
        keys.add((rng.randint(3, 13), rng.randint(7, 14), rng.randint(7, 14), rng.randint(0, 1)))
    return pr.write_lut([pr.Entry(k, rng.choice(pr.CD_CLASSES), tuple(rng.randrange(NV) for _ in range(5)))
                         for k in keys], NV)


def random_model(rng, sm):
    lo, hi = [], []
    for j in range(18):
        a = rng.choice([0.0, rng.uniform(0, 100), 16.0])
        lo.append(a)
        hi.append(a if rng.random() < 0.1 else a + rng.choice([rng.uniform(1, 9000), 1.0, 8192.0 - 16]))
    W = [[rng.gauss(0, 3) for _ in range(18)] for _ in range(5)]
    b = [rng.gauss(0, 1) for _ in range(5)]
    return P.write_model(P.Model(tuple(lo), tuple(hi), tuple(tuple(r) for r in W), tuple(b), sm))


def random_desc(rng):
    return (rng.choice([rng.randint(1, 5000), rng.choice([16, 32, 128, 512, 2048, 4096])]),
            64 * rng.randint(1, 130), 64 * rng.randint(1, 130), rng.randint(0, 1))


@pytest.mark.parametrize("chunk", range(4))
def test_features_and_predictions_identical(chunk):
    rng = random.Random(500 + chunk)
    for _ in range(100):
        lut_bytes = random_lut(rng, rng.randint(1, 30))
        entries, _ = pr.parse_lut(lut_bytes)
        lut = G.goldy_lut_from_memory(lut_bytes)
        sm = rng.choice([152, 148, 76, 38, 1])
        mb = random_model(rng, sm)
        m = P.parse_model(mb)
        pred = G.goldy_predictor_from_memory(mb)
        for _ in range(20):
            t = random_desc(rng)
            d = G.desc(*t)
            pd = pr.Desc(*t)
            e = pr.lookup(entries, pr.bucket_key(*t))
            assert G.goldy_lut_lookup(lut, d) == (e.pref_cd, list(e.variants))
            assert G.goldy_lr_features(d, lut, sm) == P.features(pd, e, sm)
            cd, probs = G.goldy_predict_cd(pred, lut, d)
            assert cd == P.predict_cd(pd, entries, m)
            ref = P.probabilities(P.scores(P.normalise(P.features(pd, e, sm), m), m))
            assert probs == pytest.approx(ref, rel=1e-12, abs=1e-300)


@pytest.mark.parametrize("chunk", range(4))
def test_plan_ex_byte_identical(chunk):
    rng = random.Random(900 + chunk)
    for trial in range(500):
        lut_bytes = random_lut(rng, rng.randint(1, 30))
        lut = G.goldy_lut_from_memory(lut_bytes)
        mb = random_model(rng, 152)
        pred = G.goldy_predictor_from_memory(mb)
        n = rng.choice([1, 2, 3, 4, 5, 8, 16, rng.randint(1, 64)])
        shapes = []
        descs = []
        for _ in range(n):
            t = rng.choice(shapes) if shapes and rng.random() < 0.6 else random_desc(rng)
            shapes.append(t)
            descs.append(t)
        flags = rng.choice([0, 0, 0, 0x10, 1, 2, 3, 4 | (rng.randint(1, 20) << 8)])
        ref = pr.serialize(P.plan([pr.Desc(*t) for t in descs], lut_bytes, mb, flags))
        got = G.goldy_schedule_serialize(G.goldy_plan_ex([G.desc(*t) for t in descs], lut, pred, flags))
        assert got == ref, (trial, descs, flags)


def test_plan_ex_without_predictor_is_plan():
    rng = random.Random(3)
    lut_bytes = random_lut(rng, 20)
    lut = G.goldy_lut_from_memory(lut_bytes)
    descs = [G.desc(*random_desc(rng)) for _ in range(9)]
    assert (G.goldy_schedule_serialize(G.goldy_plan_ex(descs, lut, None)) ==
            G.goldy_schedule_serialize(G.goldy_plan(descs, lut)))


@pytest.mark.parametrize("mutate", ["magic", "version", "nf", "sm", "size", "nan", "hi_lo"])
def test_malformed_model_rejected(mutate):
    import struct
    data = bytearray(P.write_model(P.Model((0.0,) * 18, (1.0,) * 18, ((0.0,) * 18,) * 5, (0.0,) * 5, 152)))
    if mutate == "magic":
        data[0] ^= 1
    elif mutate == "version":
        data[8] = 2
    elif mutate == "nf":
        data[12] = 17
    elif mutate == "sm":
        data[20:24] = b"\0\0\0\0"
    elif mutate == "size":
        data = data[:-8]
    elif mutate == "nan":
        data[32 + 8 * 40: 32 + 8 * 41] = struct.pack("<d", float("inf"))
    elif mutate == "hi_lo":
        data[32 + 8 * 18: 32 + 8 * 19] = struct.pack("<d", -1.0)
    with pytest.raises(G.GoldyError) as ei:
        G.goldy_predictor_from_memory(bytes(data))
    assert ei.value.status == G.GOLDY_ERR_LUT


def test_feature_argument_errors():
    lut = G.goldy_lut_from_memory(random_lut(random.Random(1), 3))
    with pytest.raises(G.GoldyError):
        G.goldy_lr_features(G.desc(10, 64, 64), lut, 0)
    with pytest.raises(G.GoldyError):
        G.goldy_lr_features(G.desc(10, 64, 64, lda=3), lut, 152)


@pytest.mark.parametrize("chunk", range(2))
def test_corun_plan_identical(chunk):
    rng = random.Random(77 + chunk)
    for _ in range(300):
        keys = set()
        while len(keys) < rng.randint(1, 25):
            keys.add((rng.randint(3, 13), rng.randint(7, 14), rng.randint(7, 14), rng.randint(0, 1)))
        lut_bytes = pr.write_lut([pr.Entry(k, rng.choice(pr.CD_CLASSES), tuple(rng.randrange(NV) for _ in range(5)),
                                           rng.randint(0, 3) | (rng.randint(0, 2) << 2)) for k in keys], NV)
        lut = G.goldy_lut_from_memory(lut_bytes)
        t = random_desc(rng)
        pol = rng.choice([0, 1, 2, 3])
        c = G.goldy_corun_plan(G.desc(*t), t[0] * t[1], t[3], lut, pol)
        conc, v, rc, _ = G.goldy_corun_query(c)
        assert (conc, v, rc) == pr.corun_plan(pr.Desc(*t), lut_bytes, pol)


def test_corun_argument_errors():
    lut = G.goldy_lut_from_memory(random_lut(random.Random(2), 3))
    with pytest.raises(G.GoldyError):
        G.goldy_corun_plan(G.desc(64, 64, 64), 10, 0, lut, 4)        # force-CD is not a co-run policy
    with pytest.raises(G.GoldyError):
        G.goldy_corun_plan(G.desc(64, 64, 64), -1, 0, lut, 0)
    with pytest.raises(G.GoldyError):
        G.goldy_corun_plan(G.desc(64, 64, 64), 10, 7, lut, 0)
    with pytest.raises(G.GoldyError):
        G.goldy_ewise_add(0, 0, 0, 10, 0, 3, 0)                       # rc_div must be 1, 2 or 4


def test_lut_flag_byte_validated_by_library():
    data = bytearray(pr.write_lut([pr.Entry((7, 10, 12, 0), 4, (1, 2, 3, 4, 5), 1)], NV))
    G.goldy_lut_from_memory(bytes(data))
    for bad_flags in (0x10, 0b1100):
        data[32 + 5] = bad_flags
        with pytest.raises(G.GoldyError):
            G.goldy_lut_from_memory(bytes(data))


@pytest.mark.parametrize("chunk", range(2))
def test_batched_descs_plan_identically(chunk):
    """Strided-batched GEMMs: bucket by M * batch, FLOPs times batch, the
    predictor's features over all entries — C++ and reference agree."""
    rng = random.Random(300 + chunk)
    for trial in range(300):
        lut_bytes = random_lut(rng, rng.randint(1, 30))
        entries, _ = pr.parse_lut(lut_bytes)
        lut = G.goldy_lut_from_memory(lut_bytes)
        mb = random_model(rng, 152)
        pred = G.goldy_predictor_from_memory(mb)
        n = rng.choice([1, 2, 3, 4, 8, 16])
        ts = []
        for _ in range(n):
            M, N, K, o = random_desc(rng)
            M = min(M, 2048)
            ts.append((M, N, K, o, rng.choice([1, 1, 2, 7, 16, 64])))
        gd = [G.desc(M, N, K, o, batch=b) for (M, N, K, o, b) in ts]
        pd = [pr.Desc(M, N, K, o, b) for (M, N, K, o, b) in ts]
        for d, p in zip(gd, pd):
            e = pr.lookup(entries, pr.bucket_key(p.M * p.batch, p.N, p.K, p.out_dtype))
            assert G.goldy_lr_features(d, lut, 152) == P.features(p, e, 152)
        flags = rng.choice([0, 0x10, 1, 2])
        assert (G.goldy_schedule_serialize(G.goldy_plan(gd, lut, flags)) ==
                pr.serialize(pr.plan(pd, lut_bytes, flags))), (trial, ts, flags)
        assert (G.goldy_schedule_serialize(G.goldy_plan_ex(gd, lut, pred, flags)) ==
                pr.serialize(P.plan(pd, lut_bytes, mb, flags))), (trial, ts, flags)


def test_batched_desc_validation():
    lut = G.goldy_lut_from_memory(random_lut(random.Random(4), 3))
    ok = G.desc(64, 128, 64, batch=4)
    G.goldy_plan([ok], lut)
    bad = [G.desc(64, 128, 64, batch=0),
           G.desc(64, 128, 64, batch=4, stride_a=64 * 64 - 8),        # entries of A overlap
           G.desc(64, 128, 64, batch=4, stride_b=64 * 128 + 4),       # not 16-byte aligned
           G.desc(64, 128, 64, batch=4, stride_c=10)]
    for d in bad:
        with pytest.raises(G.GoldyError) as ei:
            G.goldy_plan([d], lut)
        assert ei.value.status == G.GOLDY_ERR_INVALID_ARG
    # strides are ignored for a single GEMM
    G.goldy_plan([G.desc(64, 128, 64, batch=1, stride_a=0, stride_b=0, stride_c=0)], lut)
    # the no-allocation entry point takes plain GEMMs only
    assert G._lib.goldy_gemm_noalloc(ctypes.byref(ok), 0, None, None, None, None) == G.GOLDY_ERR_UNSUPPORTED
