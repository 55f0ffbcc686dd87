"""The C++ predictor path (goldy_lr_features, goldy_predict_cd, goldy_plan_ex)
against the independent restatement in oracle/predictor_ref.py: identical
features, identical predictions (both sides decide in IEEE double, in the
same order, without fused multiply-add), Eq. 1 probabilities to rounding,
byte-identical schedules, and rejection of malformed model files."""
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
