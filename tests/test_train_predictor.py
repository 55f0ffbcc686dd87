"""The offline predictor trainer: exact gradient (finite differences), the
same optimum as an independent library (scikit-learn's multinomial logistic
regression, whose penalised objective has the same minimiser), separable data
fitted perfectly, and a written model that the library loads and evaluates
to the trainer's own argmax."""
import numpy as np
import pytest

from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import train_predictor as T


def synthetic(n=400, f=6, k=5, seed=0, noise=0.35):
    """Overlapping classes: each class has its own centre in [0, 1]^f."""
    rng = np.random.default_rng(seed)
    centres = rng.uniform(0, 1, (k, f))
    y = rng.integers(0, k, n)
    X = centres[y] + rng.normal(0, noise, (n, f))
    return X, y


def test_gradient_matches_finite_differences():
    X, y = synthetic(n=60, f=4)
    Y = np.eye(5)[y]
    rng = np.random.default_rng(1)
    th = rng.normal(0, 0.3, 5 * 4 + 5)
    f0, g = T.objective(th, X, Y, 0.7)
    h = 1e-6
    num = np.array([(T.objective(th + h * e, X, Y, 0.7)[0] - T.objective(th - h * e, X, Y, 0.7)[0]) / (2 * h)
                    for e in np.eye(len(th))])
    assert np.allclose(g, num, rtol=1e-6, atol=1e-6)


def test_loss_at_zero_is_n_log_k():
    X, y = synthetic(n=50)
    loss, _ = T.objective(np.zeros(5 * 6 + 5), X, np.eye(5)[y], 1.0)
    assert loss == pytest.approx(50 * np.log(5))


@pytest.mark.parametrize("C", [0.1, 1.0, 10.0])
def test_same_optimum_as_scikit_learn(C):
    sk = pytest.importorskip("sklearn.linear_model")
    X, y = synthetic(seed=2)
    W, b = T.fit(X, y, C)
    m = sk.LogisticRegression(C=C, tol=1e-12, max_iter=100000)
    m.fit(X, y)
    P_ours = T.probabilities(W, b, X)
    P_sk = m.predict_proba(X)
    assert np.abs(P_ours - P_sk).max() < 1e-4
    assert (P_ours.argmax(axis=1) == m.predict(X)).mean() > 0.995


def test_separable_data_fitted_perfectly():
    rng = np.random.default_rng(3)
    y = rng.integers(0, 5, 300)
    X = np.eye(5)[y] + rng.uniform(-0.1, 0.1, (300, 5))
    W, b = T.fit(X, y, 1e4)
    assert (T.scores(W, b, X).argmax(axis=1) == y).all()


def test_label_rule():
    # speedups 1, 1.9, 3.0, 3.02, 2.0 -> 4 and 8 within 1% -> the larger, 8
    t = {1: 10.0, 2: 2 * 10 / 1.9, 4: 4 * 10 / 3.0, 8: 8 * 10 / 3.02, 16: 16 * 10 / 2.0}
    assert T.label_of(t) == 8
    # 3.0 vs 3.1: 4 is more than 1% off the best -> 8
    assert T.label_of({1: 10.0, 2: 2 * 10 / 1.9, 4: 4 * 10 / 3.0, 8: 8 * 10 / 3.1, 16: 16 * 10 / 2.0}) == 8
    # 3.1 vs 3.0: 8 is more than 1% off the best -> 4
    assert T.label_of({1: 10.0, 2: 2 * 10 / 1.9, 4: 4 * 10 / 3.1, 8: 8 * 10 / 3.0, 16: 16 * 10 / 2.0}) == 4
    assert T.label_of(t, available=2) == 2
    # best gain below 5% -> sequential
    assert T.label_of({1: 10.0, 2: 2 * 10 / 1.04, 4: 40.0, 8: 80.0, 16: 160.0}) == 1


def test_written_model_loads_and_predicts_like_the_trainer():
    from oracle import planner_ref as pr
    import random
    rng = random.Random(5)
    keys = set()
    while len(keys) < 25:
        keys.add((rng.randint(4, 12), rng.randint(8, 13), rng.randint(8, 13), rng.randint(0, 1)))
    lut_bytes = pr.write_lut([pr.Entry(k, rng.choice(pr.CD_CLASSES), tuple(rng.randrange(132) for _ in range(5)))
                              for k in keys], 132, 152)
    lut = G.goldy_lut_from_memory(lut_bytes)
    shapes = [(rng.randint(16, 4096), 64 * rng.randint(4, 128), 64 * rng.randint(4, 128), rng.randint(0, 1))
              for _ in range(300)]
    X = np.array([G.goldy_lr_features(G.desc(*s), lut, 152) for s in shapes])
    y = np.array([(s[0] * s[1] // 4096 + s[2] // 1000) % 5 for s in shapes])
    lo, hi = X.min(axis=0), X.max(axis=0)
    W, b = T.fit(T.normalise(X, lo, hi), y, 1.0)
    pred = G.goldy_predictor_from_memory(T.model_bytes(lo, hi, W, b, 152))
    ours = T.scores(W, b, T.normalise(X, lo, hi))
    for s, row in zip(shapes, ours):
        cd, probs = G.goldy_predict_cd(pred, lut, G.desc(*s))
        srt = np.sort(row)
        if srt[-1] - srt[-2] > 1e-9:      # numpy's summation order may differ on near-ties
            assert cd == T.CD_CLASSES[int(row.argmax())]
        assert np.allclose(probs, np.exp(row - row.max()) / np.exp(row - row.max()).sum(), atol=1e-9)


def test_evaluate_counts_and_regret():
    recs = [{"t_us": {"1": 10.0, "2": 10.0, "4": 12.0, "8": 30.0, "16": 60.0}}]
    # per-GEMM time: 10, 5, 3, 3.75, 3.75 -> best <= 16 is 4
    ev = T.evaluate([4], recs)
    assert ev["16"]["accuracy"] == 1.0 and ev["16"]["geomean_regret"] == pytest.approx(0.0)
    ev = T.evaluate([16], recs)
    assert ev["16"]["accuracy"] == 0.0 and ev["16"]["geomean_regret"] == pytest.approx(0.25)
    assert ev["2"]["accuracy"] == 1.0      # min(16, 2) = 2 is the best of {1, 2}
