"""Pins for the fp64 oracle GEMM (CPU only).

Each test checks the oracle against something other than itself: the bf16
format's definition, identity and permutation matrices, exact integer
arithmetic, a pure-Python triple loop, or numpy's float64 matmul.  A dropped
term, a sign slip, a wrong index or a transposed operand in the oracle fails
at least one of them.
"""
import os

import numpy as np
import pytest
import torch

from oracle import gemm as og
from paper_2409_02227_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "bf16_values.txt")


def _bits(t):
    return wl.bits_of(t)


def _bf16(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)


def test_bf16_decode_golden_table():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            b, v = line.split()
            rows.append((int(b, 16), float(v)))
    bits = np.array([b for b, _ in rows], dtype=np.uint16)
    got = og.bf16_decode(bits)
    for (b, want), g in zip(rows, got):
        assert g == want and np.signbit(g) == np.signbit(want), hex(b)
        assert og.bf16_value_python(b) == want


def test_bf16_decode_all_patterns_agree():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    c = og.bf16_decode(bits)
    py = np.array([og.bf16_value_python(int(b)) for b in bits])
    nan = np.isnan(py)
    assert np.array_equal(np.isnan(c), nan)
    assert np.array_equal(c[~nan], py[~nan])
    # every pattern is also what torch's bf16 -> fp32 conversion gives
    t = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(c[~nan], t[~nan])


@pytest.mark.parametrize("M,K", [(1, 1), (7, 13), (64, 64), (130, 96)])
def test_identity(M, K):
    a = wl.random_matrix(M, K, seed=11)
    eye = _bf16(np.eye(K))
    ref = og.gemm(_bits(a), _bits(eye))
    assert np.array_equal(ref, a.to(torch.float64).numpy())
    # identity on the left
    eye_m = _bf16(np.eye(M))
    ref2 = og.gemm(_bits(eye_m), _bits(a))
    assert np.array_equal(ref2, a.to(torch.float64).numpy())


def test_permutations_reorder_exactly():
    M, K, N = 9, 17, 11
    a = wl.random_matrix(M, K, seed=3)
    b = wl.random_matrix(K, N, seed=4)
    full = og.gemm(_bits(a), _bits(b))
    rng = np.random.default_rng(5)
    p_rows = rng.permutation(M)
    p_cols = rng.permutation(N)
    P = np.zeros((M, M), dtype=np.float32)
    P[np.arange(M), p_rows] = 1.0            # (P a)[i] = a[p_rows[i]]
    Q = np.zeros((N, N), dtype=np.float32)
    Q[p_cols, np.arange(N)] = 1.0            # (b Q)[:, j] = b[:, p_cols[j]]
    pa = og.gemm(_bits(_bf16(P)), _bits(a))
    assert np.array_equal(pa, a.to(torch.float64).numpy()[p_rows])
    pab = og.gemm(_bits(a[torch.from_numpy(p_rows)]), _bits(b))
    assert np.array_equal(pab, full[p_rows])
    bq = og.gemm(_bits(b), _bits(_bf16(Q)))
    assert np.array_equal(bq, b.to(torch.float64).numpy()[:, p_cols])
    abq = og.gemm(_bits(a), _bits(b[:, torch.from_numpy(p_cols)]))
    assert np.array_equal(abq, full[:, p_cols])


@pytest.mark.parametrize("M,N,K", [(5, 3, 7), (33, 65, 129), (128, 96, 512)])
def test_small_integers_exact(M, N, K):
    # |a|,|b| <= 8 and K <= 512: every partial sum is an integer below 2^24,
    # exact in fp32 and fp64; numpy's int64 matmul is exact by construction.
    a = wl.integer_matrix(M, K, seed=M + 1)
    b = wl.integer_matrix(K, N, seed=N + 2)
    ref = og.gemm(_bits(a), _bits(b))
    exact = a.to(torch.int64).numpy() @ b.to(torch.int64).numpy()
    assert np.array_equal(ref, exact.astype(np.float64))
    assert np.abs(exact).max() < 2 ** 24


def test_closed_forms():
    M, N, K = 6, 10, 300
    ones_a = _bf16(np.ones((M, K)))
    ones_b = _bf16(np.ones((K, N)))
    assert np.array_equal(og.gemm(_bits(ones_a), _bits(ones_b)), np.full((M, N), float(K)))
    # B columns constant c_j: C[i, j] = c_j * sum_k A[i, k]
    a = wl.integer_matrix(M, K, seed=9, lo=-3, hi=3)
    c = np.arange(-5, N - 5, dtype=np.float32)
    b = _bf16(np.tile(c, (K, 1)))
    rows = a.to(torch.int64).numpy().sum(axis=1)
    assert np.array_equal(og.gemm(_bits(a), _bits(b)), np.outer(rows, c).astype(np.float64))
    # K = 1 is an exact outer product
    u = wl.random_matrix(M, 1, seed=1)
    v = wl.random_matrix(1, N, seed=2)
    outer = np.outer(u.to(torch.float64).numpy()[:, 0], v.to(torch.float64).numpy()[0])
    assert np.array_equal(og.gemm(_bits(u), _bits(v)), outer)
    # K = 0 gives zeros
    z = og.gemm(np.zeros((M, 0), np.uint16), np.zeros((0, N), np.uint16))
    assert np.array_equal(z, np.zeros((M, N)))


def test_sign_and_negation():
    a = wl.random_matrix(8, 40, seed=21)
    b = wl.random_matrix(40, 12, seed=22)
    ref = og.gemm(_bits(a), _bits(b))
    assert np.array_equal(og.gemm(_bits(-a), _bits(b)), -ref)
    assert np.array_equal(og.gemm(_bits(a), _bits(-b)), -ref)


@pytest.mark.parametrize("M,N,K", [(1, 1, 1), (3, 5, 4), (7, 6, 9), (4, 9, 16)])
def test_matches_python_triple_loop(M, N, K):
    a = wl.random_matrix(M, K, seed=100 + M)
    b = wl.random_matrix(K, N, seed=200 + N)
    c = og.gemm(_bits(a), _bits(b))
    py = og.gemm_python(_bits(a), _bits(b))
    assert np.array_equal(c, py)       # same definition, same summation order


def test_matches_numpy_float64():
    M, N, K = 70, 90, 1000
    a = wl.random_matrix(M, K, seed=31)
    b = wl.random_matrix(K, N, seed=32)
    ref = og.gemm(_bits(a), _bits(b))
    npy = a.to(torch.float64).numpy() @ b.to(torch.float64).numpy()
    scale = np.abs(a.to(torch.float64).numpy()) @ np.abs(b.to(torch.float64).numpy())
    # two fp64 summation orders differ by at most ~K * 2^-53 * sum|a||b|
    assert np.all(np.abs(ref - npy) <= K * 2.0 ** -52 * scale)


def test_rows_and_entries_match_full():
    M, N, K = 40, 24, 200
    a = wl.random_matrix(M, K, seed=41)
    b = wl.random_matrix(K, N, seed=42)
    full = og.gemm(_bits(a), _bits(b))
    rows = [0, 5, 39, 17]
    assert np.array_equal(og.gemm_rows(_bits(a), _bits(b), rows), full[rows])
    ii = [0, 39, 12, 7]
    jj = [0, 23, 5, 11]
    assert np.array_equal(og.gemm_entries(_bits(a), _bits(b), ii, jj), full[ii, jj])
    with pytest.raises(IndexError):
        og.gemm_rows(_bits(a), _bits(b), [M])


def test_rejects_non_bits_and_bad_shapes():
    with pytest.raises(TypeError):
        og.gemm(np.zeros((2, 2), np.float32), np.zeros((2, 2), np.uint16))
    with pytest.raises(ValueError):
        og.gemm(np.zeros((2, 3), np.uint16), np.zeros((2, 2), np.uint16))


def test_tolerance_formula():
    ref = np.array([[3.0, -5.0], [0.5, 2.0]])
    assert og.tolerance(ref) == pytest.approx(1e-2 * 5.0 + 1e-3)
    assert og.tolerance(np.zeros((0, 3))) == pytest.approx(1e-3)


def test_workload_shapes_match_configs():
    for name, want in [("pair_256", [(256, 256, 512)] * 2),
                       ("ffn_slices", [(128, 1024, 4096)] * 4),
                       ("lstm_gates", [(32, 4096, 1024)] * 8),
                       ("hetero_pair", [(512, 1024, 1024)] * 3 + [(2048, 8192, 2048)])]:
        _, specs = wl.config_specs(name)
        assert [(s.M, s.N, s.K) for s in specs] == want
    for j in (0, 17, 63):
        _, specs, _ = wl.sweep_specs(j)
        assert 2 <= len(specs) <= 16
        for s in specs:
            assert 16 <= s.M <= 4096 and 256 <= s.N <= 8192 and 256 <= s.K <= 8192
            assert s.N % 64 == 0 and s.K % 64 == 0


def test_workload_is_seeded():
    s1 = wl.make_config("pair_256")
    s2 = wl.make_config("pair_256")
    assert np.array_equal(s1.a_bits(0), s2.a_bits(0))
    assert np.array_equal(s1.b_bits(1), s2.b_bits(1))
    assert not np.array_equal(s1.a_bits(0), s1.a_bits(1))
    v = s1.a[0].to(torch.float32)
    assert float(v.min()) >= -1.0 and float(v.max()) <= 1.0


def test_batched_gemm_is_block_diagonal_gemm():
    """A batch of two GEMMs equals one GEMM of the concatenated A panels with
    a block-diagonal B: [A0 A1] [[B0, 0], [0, B1]] = [A0 B0, A1 B1]."""
    rng = np.random.default_rng(31)
    M, K, N = 9, 70, 13
    a = rng.integers(0, 65536, size=(2, M, K), dtype=np.uint32).astype(np.uint16)
    a &= np.uint16(0xBFFF)        # finite values only (exponent below all-ones)
    b = rng.integers(0, 65536, size=(2, K, N), dtype=np.uint32).astype(np.uint16)
    b &= np.uint16(0xBFFF)
    big_a = np.concatenate([a[0], a[1]], axis=1)
    big_b = np.zeros((2 * K, 2 * N), dtype=np.uint16)          # bf16 +0
    big_b[:K, :N] = b[0]
    big_b[K:, N:] = b[1]
    whole = og.gemm(big_a, big_b)
    got = og.gemm_batched(a, b)
    assert np.array_equal(got[0], whole[:, :N])
    assert np.array_equal(got[1], whole[:, N:])
    assert np.array_equal(og.gemm_batched(a[:1], b[:1])[0], og.gemm(a[0], b[0]))
