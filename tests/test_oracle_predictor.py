"""Pins for the predictor's reference (oracle/predictor_ref.py) against what
the paper and the mathematics fix: Eq. 1 is a softmax (probabilities sum to
one; two classes reduce to the logistic sigmoid of the score difference; the
most probable class is the largest score), hand-worked features of known
kernels, the min-max normalisation's end points, the model file layout, and
the special case where the predictor reproduces the table's planner."""
import math
import random
import struct

import pytest

from oracle import planner_ref as pr
from oracle import predictor_ref as P


def vid(kind, split_idx, rc_idx):
    return (kind * 4 + split_idx) * 3 + rc_idx


def model(W=None, b=None, lo=None, hi=None, sm=152):
    return P.Model(tuple(lo or [0.0] * 18), tuple(hi or [1.0] * 18),
                   tuple(tuple(r) for r in (W or [[0.0] * 18 for _ in range(5)])), tuple(b or [0.0] * 5), sm)


def test_softmax_sums_to_one_and_is_shift_invariant():
    rng = random.Random(0)
    for _ in range(200):
        s = [rng.uniform(-30, 30) for _ in range(5)]
        p = P.probabilities(s)
        assert sum(p) == pytest.approx(1.0, abs=1e-12)
        q = P.probabilities([v + 7.5 for v in s])
        assert p == pytest.approx(q, rel=1e-12, abs=1e-15)
        assert max(range(5), key=lambda c: (p[c], -c)) == P.predict_class(s)


def test_two_classes_reduce_to_the_logistic_sigmoid():
    # with every other class at -inf in effect, softmax of two scores is the
    # sigmoid of their difference: P1 = 1 / (1 + exp(-(s1 - s0)))
    for s0, s1 in [(0.0, 0.0), (1.0, -2.0), (-3.5, 4.25), (10.0, 9.0)]:
        p = P.probabilities([s0, s1, -1e9, -1e9, -1e9])
        assert p[1] == pytest.approx(1.0 / (1.0 + math.exp(-(s1 - s0))), rel=1e-12)
        assert p[2] == 0.0


def test_ties_go_to_the_smaller_cd():
    assert P.predict_class([1.0, 1.0, 0.0, 0.0, 0.0]) == 0
    assert P.predict_class([0.0, 2.0, 2.0, 2.0, 1.0]) == 1
    assert P.predict_class([0.0] * 5) == 0


def test_kernel_features_hand_worked():
    # n128_full, split 1, whole GPU, on 128 x 1024: 1 x 8 tiles; 1 CTA/SM; cap 152
    assert P.kernel_features(128, 1024, vid(2, 0, 0), 152) == (8, 1, 1)
    # n128_full split 4, a quarter of the GPU: 32 CTAs of work, cap 38 -> 1 wave
    assert P.kernel_features(128, 1024, vid(2, 2, 2), 152) == (32, 1, 1)
    # t32_half split 2, half GPU on 40 x 296: 2 x 3 tiles x 2 = 12; 2 CTAs/SM; cap 152
    assert P.kernel_features(40, 296, vid(7, 1, 1), 152) == (12, 2, 1)
    # CTA pair on 2048 x 8192: 8 x 32 tiles, 2 CTAs each = 512; cap 152 -> 4 waves
    assert P.kernel_features(2048, 8192, vid(10, 0, 0), 152) == (512, 1, 4)
    # n64_full split 8, quarter GPU on 4096 x 8192: 32 x 128 tiles x 8 = 32768;
    # cap 38: 38 x 862 = 32756 < 32768 -> 863 waves
    assert P.kernel_features(4096, 8192, vid(0, 3, 2), 152) == (32768, 1, 863)
    # the pair kind with split 8 on 300 x 300: 2 x 2 tiles x 8 splits x 2 CTAs = 64
    assert P.kernel_features(300, 300, vid(10, 3, 0), 152) == (64, 1, 1)


def test_feature_vector_order():
    e = pr.Entry((7, 10, 12, 0), 4, (vid(2, 0, 0), vid(2, 2, 2), vid(2, 2, 2), vid(0, 0, 0), vid(0, 0, 1)))
    x = P.features(pr.Desc(128, 1024, 4096, 0), e, 152)
    # n64_full split 1 on 128 x 1024: 16 tiles; half-GPU cap 76 -> 1 wave
    assert x == [128.0, 1024.0, 4096.0, 8, 1, 1, 32, 1, 1, 32, 1, 1, 16, 1, 1, 16, 1, 1]


def test_min_max_normalisation_end_points():
    m = model(lo=[2.0] * 17 + [5.0], hi=[6.0] * 17 + [5.0])
    x = [2.0] * 9 + [6.0] * 8 + [123.0]
    assert P.normalise(x, m) == [0.0] * 9 + [1.0] * 8 + [0.0]
    assert P.normalise([4.0] * 18, m)[:17] == [0.5] * 17


def test_model_file_layout_by_hand():
    W = [[c * 100.0 + j for j in range(18)] for c in range(5)]
    m = model(W=W, b=[0.5, 1.5, 2.5, 3.5, 4.5], lo=[float(-j) for j in range(18)], hi=[float(j) for j in range(18)])
    data = P.write_model(m)
    assert len(data) == 32 + 8 * (18 + 18 + 90 + 5)
    assert data[:8] == b"GOLDYLRM"
    assert struct.unpack_from("<IIIIII", data, 8) == (1, 18, 5, 152, 0, 0)
    assert struct.unpack_from("<d", data, 32 + 8 * 17)[0] == -17.0          # lo[17]
    assert struct.unpack_from("<d", data, 32 + 8 * (36 + 18 + 3))[0] == 103.0   # W[1][3]
    assert struct.unpack_from("<d", data, len(data) - 8)[0] == 4.5         # b[4]
    assert P.parse_model(data) == m


@pytest.mark.parametrize("mutate", ["magic", "version", "nf", "sm", "size", "nan", "hi_lo"])
def test_malformed_model_rejected(mutate):
    data = bytearray(P.write_model(model()))
    if mutate == "magic":
        data[0] ^= 1
    elif mutate == "version":
        data[8] = 2
    elif mutate == "nf":
        data[12] = 17
    elif mutate == "sm":
        data[20:24] = b"\0\0\0\0"
    elif mutate == "size":
        data += b"\0" * 8
    elif mutate == "nan":
        data[32 + 8 * 40: 32 + 8 * 41] = struct.pack("<d", float("nan"))
    elif mutate == "hi_lo":
        data[32 + 8 * 18: 32 + 8 * 19] = struct.pack("<d", -1.0)
    with pytest.raises(P.ModelError):
        P.parse_model(bytes(data))


def _random_lut(rng, n_entries, pref=None):
    keys = set()
    while len(keys) < n_entries:
        keys.add((rng.randint(3, 13), rng.randint(7, 14), rng.randint(7, 14), rng.randint(0, 1)))
    return [pr.Entry(k, pref if pref else rng.choice(pr.CD_CLASSES), tuple(rng.randrange(132) for _ in range(5)))
            for k in keys]


@pytest.mark.parametrize("cls", range(5))
def test_constant_model_reproduces_table_planner(cls):
    """A model that always predicts CD class c plans exactly like the table
    planner over a table whose every preferred CD is c."""
    rng = random.Random(40 + cls)
    b = [0.0] * 5
    b[cls] = 1.0
    m = P.write_model(model(b=b))
    for _ in range(200):
        ents = _random_lut(rng, rng.randint(1, 20))
        lut_m = pr.write_lut(ents, 132)
        lut_c = pr.write_lut([pr.Entry(e.key, pr.CD_CLASSES[cls], e.variants) for e in ents], 132)
        n = rng.choice([1, 2, 3, 4, 7, 16, 33])
        descs = [pr.Desc(rng.randint(1, 5000), 64 * rng.randint(1, 130), 64 * rng.randint(1, 130),
                         rng.randint(0, 1)) for _ in range(n)]
        flags = rng.choice([0, 0x10])
        assert P.plan(descs, lut_m, m, flags) == pr.plan(descs, lut_c, flags)


def test_single_feature_model_thresholds():
    """Score of CD 16 grows with normalised K, CD 1 has a fixed bias: the
    prediction switches where 10 * (K - lo) / (hi - lo) crosses 5."""
    W = [[0.0] * 18 for _ in range(5)]
    W[4][2] = 10.0
    m = model(W=W, b=[5.0, 0, 0, 0, 0], lo=[0.0] * 2 + [1024.0] + [0.0] * 15, hi=[1.0] * 2 + [5120.0] + [1.0] * 15)
    ents = [pr.Entry((7, 10, 12, 0), 1, (0, 0, 0, 0, 0))]
    # K = 3072: x = 0.5 -> scores tie at 5 -> smaller CD (1); K = 3136 -> 16
    assert P.predict_cd(pr.Desc(128, 1024, 3072, 0), ents, m) == 1
    assert P.predict_cd(pr.Desc(128, 1024, 3136, 0), ents, m) == 16
    lut = pr.write_lut(ents, 132)
    mb = P.write_model(m)
    # two GEMMs of one bucket: the bucket takes the smaller prediction
    g, per, ms, _ = P.plan([pr.Desc(128, 1024, 3072, 0), pr.Desc(128, 1024, 3136, 0)], lut, mb)
    assert g == [(1, [0, 1])]
    g, per, ms, _ = P.plan([pr.Desc(128, 1024, 3136, 0)] * 3, lut, mb)
    assert g == [(3, [0, 1, 2])]      # min(16, 3 available)
    # forced policies ignore the model
    assert P.plan([pr.Desc(128, 1024, 3136, 0)] * 3, lut, mb, 1) == pr.plan([pr.Desc(128, 1024, 3136, 0)] * 3, lut, 1)
