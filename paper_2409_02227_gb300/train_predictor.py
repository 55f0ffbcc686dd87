"""Offline training of the logistic-regression CD predictor (Sec. 4.3, Eq. 1).

Input: the training set recorded by ``profile_lut --dataset`` — per GEMM, the
co-run time of CD copies at every CD class with the table's GO-Kernel for
that CD.  Each GEMM is labelled with its preferred CD (largest speedup
CD * T(1) / T(CD) over running the copies one after another, exact ties to
the smaller CD; sequential unless some CD gains at least 5%), and described by the 18 features the library computes
(goldy_lr_features: M, N, K and, per CD class, the table kernel's CTAs of
work, CTAs per SM and waves).  As in the paper: min-max normalisation, a
seeded 90% / 10% train / test split, and a multi-class logistic regression
whose class probabilities are Eq. 1's softmax.

Fit: minimise sum_i CE_i + ||W||^2 / (2 C) over W (5 x 18) and the biases b
(not penalised), CE the softmax cross-entropy, with L-BFGS on the exact
gradient.  C is picked by 5-fold cross-validation on the training part.

Evaluation on the held-out part, for 2, 4, 8 and 16 GEMMs available (the
paper reports accuracy that way, Sec. 6.6): a prediction p counts as right
when min(p, n) is the best CD among the classes <= n; the regret is the time
per GEMM at the chosen CD over the best, against the table's preferred CD
for the same GEMMs as the baseline.

Usage:  python -m paper_2409_02227_gb300.train_predictor DATASET.jsonl
            [--lut LUT] [--out MODEL] [--report JSON]
"""
from __future__ import annotations

import argparse
import json
import math
import struct
import sys
from typing import Dict, List, Sequence, Tuple

import numpy as np

from . import goldy as G
from .profile_lut import preferred_cd

CD_CLASSES = (1, 2, 4, 8, 16)
N_FEATURES = G.LR_FEATURES
C_GRID = (0.01, 0.1, 1.0, 10.0, 100.0, 1000.0, 1e4, 1e5)


# ----------------------------------------------------------------------------- model
def objective(theta: np.ndarray, X: np.ndarray, Y: np.ndarray, C: float) -> Tuple[float, np.ndarray]:
    """Penalised softmax cross-entropy and its gradient.  theta packs W
    (classes x features, row-major) then b; Y is one-hot."""
    k, f = Y.shape[1], X.shape[1]
    W = theta[:k * f].reshape(k, f)
    b = theta[k * f:]
    S = X @ W.T + b
    S = S - S.max(axis=1, keepdims=True)
    E = np.exp(S)
    Z = E.sum(axis=1, keepdims=True)
    logP = S - np.log(Z)
    loss = -float((Y * logP).sum()) + float((W * W).sum()) / (2.0 * C)
    R = E / Z - Y
    gW = R.T @ X + W / C
    gb = R.sum(axis=0)
    return loss, np.concatenate([gW.ravel(), gb])


def fit(X: np.ndarray, y: np.ndarray, C: float, n_classes: int = 5) -> Tuple[np.ndarray, np.ndarray]:
    from scipy.optimize import minimize
    Y = np.zeros((len(y), n_classes))
    Y[np.arange(len(y)), y] = 1.0
    theta0 = np.zeros(n_classes * X.shape[1] + n_classes)
    res = minimize(objective, theta0, args=(X, Y, C), jac=True, method="L-BFGS-B",
                   options={"maxiter": 20000, "maxfun": 40000, "gtol": 1e-9, "ftol": 1e-14})
    th = res.x
    k, f = n_classes, X.shape[1]
    return th[:k * f].reshape(k, f), th[k * f:]


def scores(W: np.ndarray, b: np.ndarray, Xn: np.ndarray) -> np.ndarray:
    return Xn @ W.T + b


def probabilities(W: np.ndarray, b: np.ndarray, Xn: np.ndarray) -> np.ndarray:
    """Eq. 1."""
    S = scores(W, b, Xn)
    E = np.exp(S - S.max(axis=1, keepdims=True))
    return E / E.sum(axis=1, keepdims=True)


def normalise(X: np.ndarray, lo: np.ndarray, hi: np.ndarray) -> np.ndarray:
    span = hi - lo
    out = np.zeros_like(X)
    ok = span > 0
    out[:, ok] = (X[:, ok] - lo[ok]) / span[ok]
    return out


def model_bytes(lo: Sequence[float], hi: Sequence[float], W: np.ndarray, b: np.ndarray, sm_count: int) -> bytes:
    """The GOLDYLRM file goldy_predictor_load reads (include/goldy.h)."""
    out = bytearray(b"GOLDYLRM")
    out += struct.pack("<IIIIII", 1, N_FEATURES, len(CD_CLASSES), sm_count, 0, 0)
    vals = [float(v) for v in lo] + [float(v) for v in hi] + [float(v) for v in W.ravel()] + [float(v) for v in b]
    out += struct.pack("<%dd" % len(vals), *vals)
    return bytes(out)


def cross_validate(X: np.ndarray, y: np.ndarray, folds: int = 5, seed: int = 0) -> Dict[float, float]:
    rng = np.random.default_rng(seed)
    idx = rng.permutation(len(y))
    parts = np.array_split(idx, folds)
    acc = {}
    for C in C_GRID:
        right = 0
        for f in range(folds):
            te = parts[f]
            tr = np.concatenate([parts[g] for g in range(folds) if g != f])
            lo, hi = X[tr].min(axis=0), X[tr].max(axis=0)
            W, b = fit(normalise(X[tr], lo, hi), y[tr], C)
            right += int((scores(W, b, normalise(X[te], lo, hi)).argmax(axis=1) == y[te]).sum())
        acc[C] = right / len(y)
    return acc


# ----------------------------------------------------------------------------- data
def load_dataset(path: str) -> List[dict]:
    recs = []
    with open(path) as f:
        for line in f:
            line = line.strip()
            if line:
                recs.append(json.loads(line))
    return recs


def label_of(t_us: Dict[int, float], available: int = 16) -> int:
    """Preferred CD among the classes <= available."""
    t1 = t_us[1]
    return preferred_cd({c: c * t1 / t_us[c] for c in CD_CLASSES if c <= available})


def lut_sm_count(path: str) -> int:
    with open(path, "rb") as f:
        head = f.read(32)
    return struct.unpack_from("<I", head, 20)[0]


def evaluate(pred_cd: Sequence[int], recs: Sequence[dict]) -> Dict[str, dict]:
    """Accuracy and geomean regret (time per GEMM at min(p, n) over the best
    class <= n) for n = 2, 4, 8, 16 GEMMs available."""
    out = {}
    for n in (2, 4, 8, 16):
        right, logs = 0, []
        for p, r in zip(pred_cd, recs):
            t = {int(c): v for c, v in r["t_us"].items()}
            chosen = min(p, n)
            best = label_of(t, n)
            right += int(chosen == best)
            per = {c: t[c] / c for c in CD_CLASSES if c <= n}
            logs.append(math.log(per[chosen] / min(per.values())))
        out[str(n)] = {"accuracy": right / len(recs), "geomean_regret": math.exp(sum(logs) / len(logs)) - 1.0,
                       "max_regret": math.exp(max(logs)) - 1.0}
    return out


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("dataset")
    ap.add_argument("--lut", default=G.DEFAULT_LUT)
    ap.add_argument("--out", default=G.DEFAULT_PREDICTOR)
    ap.add_argument("--report", default=None)
    ap.add_argument("--seed", type=int, default=0, help="train/test split seed")
    args = ap.parse_args(argv)

    recs = load_dataset(args.dataset)
    lut = G.goldy_lut_load(args.lut)
    sm = lut_sm_count(args.lut)
    X = np.array([G.goldy_lr_features(G.desc(*r["shape"]), lut, sm) for r in recs], dtype=np.float64)
    labels = [label_of({int(c): v for c, v in r["t_us"].items()}) for r in recs]
    y = np.array([CD_CLASSES.index(c) for c in labels])
    rng = np.random.default_rng(args.seed)
    perm = rng.permutation(len(recs))
    n_test = max(1, len(recs) // 10)
    te, tr = perm[:n_test], perm[n_test:]

    cv = cross_validate(X[tr], y[tr])
    C = max(C_GRID, key=lambda c: (cv[c], -c))
    lo, hi = X[tr].min(axis=0), X[tr].max(axis=0)
    W, b = fit(normalise(X[tr], lo, hi), y[tr], C)
    data = model_bytes(lo, hi, W, b, sm)
    pred = G.goldy_predictor_from_memory(data)          # validate with the library's parser

    # predictions through the library (the path the planner takes)
    lr_cd = [G.goldy_predict_cd(pred, lut, G.desc(*r["shape"]))[0] for r in recs]
    lut_cd = [G.goldy_lut_lookup(lut, G.desc(*r["shape"]))[0] for r in recs]
    np_cd = [CD_CLASSES[i] for i in scores(W, b, normalise(X, lo, hi)).argmax(axis=1)]
    agree = sum(a == b_ for a, b_ in zip(lr_cd, np_cd)) / len(recs)

    test = [recs[i] for i in te]
    train = [recs[i] for i in tr]
    report = {
        "dataset": args.dataset, "gemms": len(recs), "train": len(tr), "test": len(te), "C": C,
        "cv_accuracy": {str(k): v for k, v in cv.items()},
        "label_counts": {str(c): labels.count(c) for c in CD_CLASSES},
        "library_vs_numpy_prediction_agreement": agree,
        "test": {"predictor": evaluate([lr_cd[i] for i in te], test),
                 "table": evaluate([lut_cd[i] for i in te], test),
                 "always_sequential": evaluate([1] * len(te), test)},
        "train": {"predictor": evaluate([lr_cd[i] for i in tr], train),
                  "table": evaluate([lut_cd[i] for i in tr], train)},
    }
    with open(args.out, "wb") as f:
        f.write(data)
    txt = json.dumps(report, indent=1)
    if args.report:
        with open(args.report, "w") as f:
            f.write(txt + "\n")
    print(txt)
    return 0


if __name__ == "__main__":
    sys.exit(main())
