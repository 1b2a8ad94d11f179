"""Pins for the fp64 oracle: each check reaches the oracle's result by another route (a
closed form, a library routine, brute force, an invariant, or a value the paper prints), so
a dropped term, a wrong sign, index or transposed operand in the oracle fails one of them.
CPU only."""
import itertools
import math
import os

import numpy as np
import pytest
from scipy.cluster.vq import vq

from oracle import crvq_oracle as O
import synthetic as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def _spd(rng, d, cond=20.0):
    Q, _ = np.linalg.qr(rng.standard_normal((d, d)))
    ev = np.exp(rng.uniform(0, math.log(cond), d))
    return ((Q * ev) @ Q.T).astype(np.float32)


def _sym32(A):
    A = np.asarray(A, np.float32)
    return ((A + A.T) * np.float32(0.5)).astype(np.float32)


# ---------------------------------------------------------------- generator pins
def test_splitmix64_published_sequence():
    for seed, ctr, hexv in _golden("splitmix64.txt"):
        assert O.splitmix64(int(seed), int(ctr)) == int(hexv, 16)
        assert int(S.splitmix64(int(seed), np.array([int(ctr)]))[0]) == int(hexv, 16)


def test_bf16_rounding_ties_to_even():
    a = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -9, -2.5], np.float32)
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7 -> even (1.0); 1 + 3*2^-8 -> 1 + 2^-6.
    exp = np.array([1.0, 1.0, 1.0 + 2 ** -6, 1.0, -2.5], np.float32)
    np.testing.assert_array_equal(S.round_to_bf16(a), exp)


# ---------------------------------------------------------------- O1 Hessian
def test_hessian_closed_form_scaled_identity():
    N = 16
    X = np.sqrt(N) * np.eye(N, dtype=np.float32)    # n = N tokens: X^T X / n = I
    H, xsq, Hb, delta = O.hessian(X, 0.25, 8)
    np.testing.assert_allclose(H, 1.25 * np.eye(N), rtol=0, atol=1e-6)
    np.testing.assert_allclose(xsq, np.ones(N), rtol=1e-6)
    assert abs(float(delta) - 0.25) < 1e-7
    np.testing.assert_allclose(Hb, np.broadcast_to(1.25 * np.eye(8), (2, 8, 8)), atol=1e-6)


def test_hessian_matches_matrix_free_product():
    rng = np.random.default_rng(1)
    X = rng.standard_normal((37, 24)).astype(np.float32) * rng.uniform(0.1, 3, 24)
    H, xsq, Hb, delta = O.hessian(X, 0.01, 8)
    v = rng.standard_normal(24)
    X64 = X.astype(np.float64)
    ref = X64.T @ (X64 @ v) / 37 + float(delta) * v
    np.testing.assert_allclose(H.astype(np.float64) @ v, ref, rtol=1e-5, atol=1e-5)
    assert np.allclose(H, H.T)
    np.testing.assert_allclose(xsq, (X64 ** 2).mean(axis=0), rtol=1e-6)
    np.testing.assert_allclose(float(delta), 0.01 * (X64 ** 2).mean(), rtol=1e-6)
    for g in range(3):
        np.testing.assert_array_equal(Hb[g], H[8 * g:8 * g + 8, 8 * g:8 * g + 8])


# ---------------------------------------------------------------- O2/O3 encode
def test_encode_isotropic_is_euclidean_nearest_codeword():
    rng = np.random.default_rng(2)
    M, G, d, K = 40, 3, 8, 16
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    C = rng.standard_normal((K, d)).astype(np.float32)
    Hb = np.stack([np.float32(c) * np.eye(d, dtype=np.float32) for c in (1.0, 2.0, 0.5)])
    codes, verr = O.encode_beam(T, d, Hb, [O.Codebook(C, None, G)], 0, 1)
    for g in range(G):
        ref, dist = vq(T[:, g * d:(g + 1) * d].astype(np.float64), C.astype(np.float64))
        np.testing.assert_array_equal(codes[0][:, g], ref)
        np.testing.assert_allclose(verr[:, g], Hb[g][0, 0] * dist ** 2, rtol=1e-5)


def test_encode_general_H_equals_whitened_nearest_codeword():
    """err(t,c) = ||L^T (t - c)||^2 with H = L L^T: nearest codeword after whitening."""
    rng = np.random.default_rng(3)
    M, G, d, K = 50, 2, 8, 32
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    C = rng.standard_normal((K, d)).astype(np.float32)
    Hb = np.stack([_spd(rng, d) for _ in range(G)])
    codes, verr = O.encode_beam(T, d, Hb, [O.Codebook(C, None, G)], 0, 1)
    for g in range(G):
        L = np.linalg.cholesky(Hb[g].astype(np.float64))
        ref, dist = vq(T[:, g * d:(g + 1) * d].astype(np.float64) @ L, C.astype(np.float64) @ L)
        np.testing.assert_array_equal(codes[0][:, g], ref)
        np.testing.assert_allclose(verr[:, g], dist ** 2, rtol=1e-5)


def test_encode_with_fixed_codebook_equals_encode_of_residual():
    rng = np.random.default_rng(4)
    M, G, d = 30, 2, 4
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    C0 = rng.standard_normal((8, d)).astype(np.float32)
    C1 = (0.3 * rng.standard_normal((8, d))).astype(np.float32)
    codes0 = rng.integers(0, 8, (M, G))
    Hb = np.stack([_spd(rng, d) for _ in range(G)])
    R = T.astype(np.float64).copy()
    for g in range(G):
        R[:, g * d:(g + 1) * d] -= C0[codes0[:, g]]
    a, ea = O.encode_beam(T, d, Hb, [O.Codebook(C0, codes0, G), O.Codebook(C1, None, G)], 1, 1)
    b, eb = O.encode_beam(R, d, Hb, [O.Codebook(C1, None, G)], 0, 1)
    np.testing.assert_array_equal(a[1], b[0])
    np.testing.assert_allclose(ea, eb, rtol=1e-4, atol=1e-6)


# ---------------------------------------------------------------- O4 beam vs exhaustive
@pytest.mark.parametrize("K,m,d", [(2, 1, 2), (4, 2, 4), (2, 3, 8), (4, 3, 2), (3, 2, 8)])
def test_beam_with_full_width_equals_exhaustive_search(K, m, d):
    rng = np.random.default_rng(10 * K + m + d)
    M, G = 12, 2
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    Cs = [(rng.standard_normal((K, d)) / (1 + s)).astype(np.float32) for s in range(m)]
    Hb = np.stack([_spd(rng, d) for _ in range(G)])
    B = K ** (m - 1)                                      # >= product of all but the last K
    cbs = [O.Codebook(C, None, G) for C in Cs]
    codes, verr = O.encode_beam(T, d, Hb, cbs, 0, B)
    for g in range(G):
        L = np.linalg.cholesky(Hb[g].astype(np.float64))
        for i in range(M):
            t = T[i, g * d:(g + 1) * d].astype(np.float64)
            best, arg = np.inf, None
            for tup in itertools.product(range(K), repeat=m):
                r = t - sum(Cs[s][tup[s]].astype(np.float64) for s in range(m))
                e = float(np.linalg.norm(L.T @ r) ** 2)
                if e < best:
                    best, arg = e, tup
            assert tuple(codes[s][i, g] for s in range(m)) == arg
            assert abs(verr[i, g] - best) <= 1e-5 * max(1.0, best)


def test_narrow_beam_never_beats_exhaustive_and_keep_if_better_keeps_optimum():
    rng = np.random.default_rng(11)
    K, m, d, M, G = 4, 3, 4, 20, 1
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    Cs = [(rng.standard_normal((K, d)) / (1 + s)).astype(np.float32) for s in range(m)]
    Hb = np.stack([_spd(rng, d)])
    full, efull = O.encode_beam(T, d, Hb, [O.Codebook(C, None, G) for C in Cs], 0, K ** 2)
    narrow, enarrow = O.encode_beam(T, d, Hb, [O.Codebook(C, None, G) for C in Cs], 0, 1)
    assert np.all(enarrow >= efull - 1e-6)
    # seeded with the optimal tuple, the width-1 beam must keep it
    kept, ekept = O.encode_beam(T, d, Hb, [O.Codebook(C, full[s], G) for s, C in enumerate(Cs)],
                                0, 1, keep_if_better=True)
    np.testing.assert_allclose(ekept, efull, rtol=1e-6)
    for s in range(m):
        np.testing.assert_array_equal(kept[s], full[s])


# ---------------------------------------------------------------- O5 init
def test_kmeans_init_strata_distinct_deterministic():
    n, K = 1000, 37
    a = O.kmeans_sample_indices(n, K, 123)
    b = O.kmeans_sample_indices(n, K, 123)
    c = O.kmeans_sample_indices(n, K, 124)
    np.testing.assert_array_equal(a, b)
    assert not np.array_equal(a, c)
    assert len(set(a.tolist())) == K
    for k, v in enumerate(a):
        assert (k * n) // K <= v < ((k + 1) * n) // K
    np.testing.assert_array_equal(O.kmeans_sample_indices(5, 5, 9), np.arange(5))


def test_kmeans_init_takes_sampled_vectors_and_residuals():
    rng = np.random.default_rng(5)
    M, G, d, K = 10, 3, 8, 6
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    idx = O.kmeans_sample_indices(M * G, K, 77)
    C = O.kmeans_init(T, d, G, K, 77)
    for k, v in enumerate(idx):
        i, g = divmod(int(v), G)
        np.testing.assert_array_equal(C[k], T[i, g * d:(g + 1) * d])
    C0 = rng.standard_normal((4, d)).astype(np.float32)
    codes0 = rng.integers(0, 4, (M, G))
    Cr = O.kmeans_init(T, d, G, K, 77, fixed=[O.Codebook(C0, codes0, G)])
    for k, v in enumerate(idx):
        i, g = divmod(int(v), G)
        np.testing.assert_allclose(Cr[k], T[i, g * d:(g + 1) * d] - C0[codes0[i, g]], atol=1e-6)


# ---------------------------------------------------------------- O6 LS update
def test_update_isotropic_is_cluster_mean():
    rng = np.random.default_rng(6)
    M, G, d, K = 60, 2, 8, 7
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    codes = rng.integers(0, K - 1, (M, G))         # codeword K-1 stays empty
    Cold = rng.standard_normal((K, d)).astype(np.float32)
    Hb = np.stack([np.float32(2.0) * np.eye(d, dtype=np.float32)] * G)
    C, counts = O.update_codebook(T, d, Hb, [O.Codebook(Cold, codes, G)], 0)
    V = np.concatenate([T[:, g * d:(g + 1) * d] for g in range(G)])
    code = np.concatenate([codes[:, g] for g in range(G)])
    for k in range(K - 1):
        np.testing.assert_allclose(C[k], V[code == k].astype(np.float64).mean(0), rtol=1e-5,
                                   atol=1e-6)
    np.testing.assert_array_equal(C[K - 1], Cold[K - 1])
    np.testing.assert_array_equal(counts, np.bincount(code, minlength=K))


def test_update_is_a_minimiser_and_single_member_is_exact():
    rng = np.random.default_rng(7)
    M, G, d, K = 40, 3, 8, 5
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    codes = rng.integers(0, K, (M, G))
    codes[0, 0] = K - 1
    codes[(codes == K - 1)] = 0
    codes[0, 0] = K - 1                             # codeword K-1 has exactly one member
    Hb = np.stack([_spd(rng, d) for _ in range(G)])
    Cold = rng.standard_normal((K, d)).astype(np.float32)
    C, counts = O.update_codebook(T, d, Hb, [O.Codebook(Cold, codes, G)], 0)
    assert counts[K - 1] == 1
    np.testing.assert_allclose(C[K - 1], T[0, :d], rtol=1e-5, atol=1e-6)

    def obj(k, c):
        tot = 0.0
        for g in range(G):
            Dg = T[codes[:, g] == k, g * d:(g + 1) * d].astype(np.float64) - c
            L = np.linalg.cholesky(Hb[g].astype(np.float64))
            tot += float((np.linalg.norm(Dg @ L, axis=1) ** 2).sum())
        return tot

    for k in range(K):
        base = obj(k, C[k].astype(np.float64))
        for _ in range(10):
            u = rng.standard_normal(d) * 1e-2
            assert obj(k, C[k] + u) >= base - 1e-9 * max(1.0, base)


def test_update_of_second_codebook_targets_residual():
    rng = np.random.default_rng(8)
    M, G, d = 30, 2, 4
    T = rng.standard_normal((M, G * d)).astype(np.float32)
    C0 = rng.standard_normal((6, d)).astype(np.float32)
    C1 = rng.standard_normal((5, d)).astype(np.float32)
    c0 = rng.integers(0, 6, (M, G))
    c1 = rng.integers(0, 5, (M, G))
    Hb = np.stack([_spd(rng, d) for _ in range(G)])
    a, ca = O.update_codebook(T, d, Hb, [O.Codebook(C0, c0, G), O.Codebook(C1, c1, G)], 1)
    R = T.astype(np.float64).copy()
    for g in range(G):
        R[:, g * d:(g + 1) * d] -= C0[c0[:, g]]
    b, cb = O.update_codebook(R, d, Hb, [O.Codebook(C1, c1, G)], 0)
    np.testing.assert_allclose(a, b, rtol=1e-5, atol=1e-6)
    np.testing.assert_array_equal(ca, cb)


def test_lloyd_objective_non_increasing():
    rng = np.random.default_rng(9)
    M, G, d, K = 64, 4, 8, 16
    T = (0.02 * rng.standard_normal((M, G * d))).astype(np.float32)
    Hb = np.stack([_spd(rng, d) for _ in range(G)])
    C0 = O.kmeans_init(T, d, G, K, 5)
    _, objective = O.lloyd(T, d, Hb, [], C0, G, 8)
    assert all(b <= a * (1 + 1e-9) for a, b in zip(objective, objective[1:]))
    assert objective[-1] < objective[0]


# ---------------------------------------------------------------- O7/O8 importance & reorder
def test_importance_wa_equals_literal_app_a2_sum():
    rng = np.random.default_rng(12)
    n, M, N = 9, 5, 16
    X = rng.standard_normal((n, N)).astype(np.float32)
    W = rng.standard_normal((M, N)).astype(np.float32)
    Wq = (W + 0.1 * rng.standard_normal((M, N))).astype(np.float32)
    _, xsq, _, _ = O.hessian(X, 0.0, 8)
    I = O.importance(W, Wq, xsq, O.MODE_WA, 0)
    lit = np.zeros(N)
    for i in range(N):
        lit[i] = max(0.5 * sum((float(X[k, i]) * (float(W[j, i]) - float(Wq[j, i]))) ** 2
                               for k in range(n)) for j in range(M))
    np.testing.assert_allclose(I * n, lit, rtol=1e-6)            # xsq carries the 1/n
    np.testing.assert_allclose(O.importance(W, Wq, xsq, O.MODE_WONLY, 0),
                               (W.astype(np.float64) ** 2).max(0))


def test_hinv_diag_closed_forms():
    """diag(H^-1) of Eq. (wa): a diagonal H, 2 x 2 blocks, and delta I + u u^T
    (Sherman-Morrison: [H^-1]_ii = 1/delta - u_i^2 / (delta (delta + |u|^2)))."""
    h = np.array([0.5, 2.0, 4.0, 1.25])
    np.testing.assert_allclose(O.hinv_diag(np.diag(h)), 1.0 / h, rtol=1e-14)
    a, b, c = 3.0, -1.2, 2.0
    H = np.kron(np.eye(3), np.array([[a, b], [b, c]]))
    det = a * c - b * b
    np.testing.assert_allclose(O.hinv_diag(H), np.tile([c / det, a / det], 3), rtol=1e-13)
    rng = np.random.default_rng(21)
    u, delta = rng.standard_normal(9), 0.3
    exp = 1.0 / delta - u * u / (delta * (delta + u @ u))
    np.testing.assert_allclose(O.hinv_diag(delta * np.eye(9) + np.outer(u, u)), exp, rtol=1e-12)


def test_hinv_diag_equals_schur_complement():
    """OBS identity: 1 / [H^-1]_ii = H_ii - H_i,r H_r,r^-1 H_r,i (r = every other index), the
    least value of z^T H z over z with z_i = 1; computed by a linear solve on the rest."""
    rng = np.random.default_rng(22)
    N = 12
    X = rng.standard_normal((30, N)) * rng.uniform(0.2, 3.0, N)
    H = X.T @ X / 30 + 0.01 * np.eye(N)
    got = O.hinv_diag(H)
    for i in range(N):
        r = [j for j in range(N) if j != i]
        s = H[i, i] - H[i, r] @ np.linalg.solve(H[np.ix_(r, r)], H[r, i])
        assert abs(1.0 / got[i] - s) <= 1e-10 * s
        z = np.zeros(N)
        z[i] = 1.0
        z[r] = -np.linalg.solve(H[np.ix_(r, r)], H[r, i])
        assert abs(z @ H @ z - s) <= 1e-10 * s


def test_hinv_diag_equals_woodbury_when_tokens_are_fewer_than_channels():
    """H = delta I + X^T X / n with n < N: [H^-1]_ii = (1 - x_i^T (n delta I + X X^T)^-1 x_i)
    / delta (Woodbury), from an n x n system instead of the N x N factor."""
    rng = np.random.default_rng(24)
    n, N, delta = 7, 20, 0.05
    X = rng.standard_normal((n, N)) * rng.uniform(0.3, 2.0, N)
    H = X.T @ X / n + delta * np.eye(N)
    A = n * delta * np.eye(n) + X @ X.T
    q = np.einsum("ki,ki->i", X, np.linalg.solve(A, X))
    np.testing.assert_allclose(O.hinv_diag(H), (1.0 - q) / delta, rtol=1e-10)


def test_importance_eq_wa_is_app_a2_for_uncorrelated_channels():
    """Eq. (wa) with a diagonal X^T X (orthogonal channels, no damping) is the App. A.2 form:
    1 / [H^-1]_ii = H_ii = xsq_i. With correlated channels the two differ."""
    rng = np.random.default_rng(23)
    n, M, N = 24, 6, 16
    Q, _ = np.linalg.qr(rng.standard_normal((n, N)))
    X = (Q * rng.uniform(0.5, 4.0, N)).astype(np.float32)
    W = rng.standard_normal((M, N)).astype(np.float32)
    Wq = (W + 0.1 * rng.standard_normal((M, N))).astype(np.float32)
    H, xsq, _, _ = O.hessian(X, 0.0, 8)
    I_inv = O.importance(W, Wq, xsq, O.MODE_WA_INV, 0, O.hinv_diag(H))
    I_a2 = O.importance(W, Wq, xsq, O.MODE_WA, 0)
    np.testing.assert_allclose(I_inv, I_a2, rtol=1e-4)
    dW = W.astype(np.float64) - Wq
    lit = np.array([max(dW[j, i] ** 2 for j in range(M)) / (2.0 * np.linalg.inv(
        H.astype(np.float64))[i, i]) for i in range(N)])
    np.testing.assert_allclose(I_inv, lit, rtol=1e-5)
    Xc = X + 0.5 * X[:, :1]                          # channel 0 mixed into every channel
    Hc, xc, _, _ = O.hessian(Xc, 0.0, 8)
    assert not np.allclose(O.importance(W, Wq, xc, O.MODE_WA_INV, 0, O.hinv_diag(Hc)),
                           O.importance(W, Wq, xc, O.MODE_WA, 0), rtol=1e-2)
    perm = O.select_reorder_channels(W, 8, Wq, xsq, H, 0.25, O.MODE_WA_INV, 0)[0]
    np.testing.assert_array_equal(perm, np.lexsort((np.arange(N), -I_inv)))


def test_reorder_bijection_roundtrip_and_blocks():
    rng = np.random.default_rng(13)
    M, N, d = 7, 32, 8
    W = rng.standard_normal((M, N)).astype(np.float32)
    X = rng.standard_normal((20, N)).astype(np.float32)
    H, xsq, _, _ = O.hessian(X, 0.01, d)
    Wq = np.round(W * 2) / 2
    perm, I, Ws, Hb, Gc = O.select_reorder_channels(W, d, Wq, xsq, H, 0.1, O.MODE_WA, 0)
    assert sorted(perm.tolist()) == list(range(N))
    assert np.all(np.diff(I[perm].astype(np.float64)) <= 0)
    inv = np.argsort(perm)
    np.testing.assert_array_equal(Ws[:, inv], W)
    Hp = H[np.ix_(perm, perm)]
    for g in range(N // d):
        np.testing.assert_array_equal(Hb[g], Hp[g * d:(g + 1) * d, g * d:(g + 1) * d])
    assert Gc == 1
    # random mode: a seeded permutation, deterministic
    p1 = O.select_reorder_channels(W, d, Wq, xsq, H, 0.1, O.MODE_RANDOM, 5)[0]
    p2 = O.select_reorder_channels(W, d, Wq, xsq, H, 0.1, O.MODE_RANDOM, 5)[0]
    np.testing.assert_array_equal(p1, p2)
    assert sorted(p1.tolist()) == list(range(N))


def test_importance_ties_broken_by_index():
    W = np.ones((3, 16), np.float32)
    perm = O.select_reorder_channels(W, 8, np.zeros_like(W), np.ones(16, np.float32),
                                     np.eye(16, dtype=np.float32), 0.5, O.MODE_WONLY, 0)[0]
    np.testing.assert_array_equal(perm, np.arange(16))


def test_n_crit_groups_closed_form():
    for N, d, lam, gc in _golden("n_crit_groups.txt"):
        assert O.n_crit_groups(int(N), int(d), float(lam)) == int(gc)
    assert O.n_crit_groups(64, 8, 0.0) == 0
    assert O.n_crit_groups(64, 8, 1.0) == 8


def test_outlier_channels_land_in_critical_set():
    cfg = S.C1.with_(kmeans_iters=2)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    d, G = cfg.d, cfg.G
    H, xsq, Hb0, _ = O.hessian(X, cfg.damp_rel, d)
    C0 = O.kmeans_init(W, d, G, cfg.K_base, 1)
    pre, _ = O.lloyd(W, d, Hb0, [], C0, G, cfg.kmeans_iters)
    W_pre = O.reconstruct_error(W, d, Hb0, None, [pre], 0)[0]
    outl = set(S.pick_columns(cfg.seed, cfg.name + "/W/outliers", cfg.N, 8).tolist())
    for mode in (O.MODE_WA, O.MODE_WONLY):
        perm, _, _, _, Gc = O.select_reorder_channels(W, d, W_pre, xsq, H, cfg.crit_frac,
                                                      mode, 0)
        assert outl <= set(perm[:Gc * d].tolist())


# ---------------------------------------------------------------- O10 losses & decode
def test_loss_full_two_routes_and_block_loss_matches_encode():
    rng = np.random.default_rng(14)
    M, N, d, n = 6, 24, 8, 30
    X = rng.standard_normal((n, N)).astype(np.float32)
    W = rng.standard_normal((M, N)).astype(np.float32)
    H, xsq, _, delta = O.hessian(X, 0.05, d)
    perm = rng.permutation(N).astype(np.int32)
    Ws = W[:, perm]
    Hb = np.stack([H[np.ix_(perm[g * d:g * d + d], perm[g * d:g * d + d])] for g in range(3)])
    C0 = rng.standard_normal((5, d)).astype(np.float32)
    C1 = (0.2 * rng.standard_normal((4, d))).astype(np.float32)
    cbs = [O.Codebook(C0, None, 3), O.Codebook(C1, None, 1)]
    codes, verr = O.encode_beam(Ws, d, Hb, cbs, 0, 4)
    cbs = [O.Codebook(C0, codes[0], 3), O.Codebook(C1, codes[1], 1)]
    W_hat, lb, lc, lf = O.reconstruct_error(Ws, d, Hb, perm, cbs, 1, X, float(delta))
    dW = W.astype(np.float64) - W_hat.astype(np.float64)
    tr = float(np.trace(dW @ H.astype(np.float64) @ dW.T))
    assert abs(lf - tr) <= 1e-5 * tr
    assert abs(lb - float(verr.astype(np.float64).sum())) <= 1e-5 * lb
    assert abs(lc - float(verr[:, :1].astype(np.float64).sum())) <= 1e-5 * lc
    # reconstruction of vector (i, g) in the original order is the sum of its codewords
    for i in range(M):
        for g in range(3):
            r = C0[codes[0][i, g]].astype(np.float64)
            if g < 1:
                r = r + C1[codes[1][i, g]]
            np.testing.assert_allclose(W_hat[i, perm[g * d:(g + 1) * d]], r, rtol=1e-6)


def test_codebook_holding_every_vector_gives_zero_loss():
    rng = np.random.default_rng(15)
    M, N, d = 4, 16, 8
    W = rng.standard_normal((M, N)).astype(np.float32)
    C = np.concatenate([W[:, g * d:(g + 1) * d] for g in range(2)])
    Hb = np.stack([_spd(rng, d) for _ in range(2)])
    codes, verr = O.encode_beam(W, d, Hb, [O.Codebook(C, None, 2)], 0, 1)
    np.testing.assert_array_equal(verr, 0)
    W_hat, lb, lc, _ = O.reconstruct_error(W, d, Hb, None, [O.Codebook(C, codes[0], 2)], 0)
    np.testing.assert_array_equal(W_hat, W)
    assert lb == 0.0 and lc == 0.0


# ---------------------------------------------------------------- A16 bit-width (golden)
def test_avg_bits_paper_values():
    for e, d, m, lam, exp, dec, *_ in _golden("avg_bits.txt"):
        v = O.avg_bits(int(e), int(d), int(m), float(lam))
        assert round(v, int(dec)) == pytest.approx(float(exp))


def test_avg_bits_of_base_codebooks_alone_is_sec_3_2_eq_bitwidth():
    """m base codebooks and no extended ones: the App. A.1 count reduces to Sec. 3.2 Eq.
    (bitwidth) for a 4096 x 4096 matrix, n = m e / d + 2^(e - 20) m d; the two 1-bit settings
    Sec. 3.2 names for e = 8 (m = 1, d = 8 and m = 2, d = 16) both come to 1 bit and a
    fraction of a percent."""
    for e, d, m in [(8, 8, 1), (8, 16, 2), (10, 8, 2), (12, 16, 3), (8, 8, 4)]:
        eq = m * e / d + 2.0 ** (e - 20) * m * d
        assert O.avg_bits(e, d, 1, 0.0, n_base=m) == pytest.approx(eq, rel=1e-12)
        assert O.avg_bits(e, d, 1, 0.3, n_base=m) == pytest.approx(eq, rel=1e-12)
    for d, m in [(8, 1), (16, 2)]:
        assert 1.0 < O.avg_bits(8, d, 1, 0.0, n_base=m) < 1.01


# ---------------------------------------------------------------- schedule invariants
def test_schedule_invariants_small():
    """Extended codebooks never raise the critical-channel loss (LS optimality vs c = 0
    start), Lloyd objectives never rise, and one refinement round never raises the loss."""
    cfg = S.LayerConfig("pin_small", 64, 64, 96, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=3, K_base=16, n_ext=2, K_ext=8, crit_frac=0.1, B=4,
                        kmeans_iters=4)
    out = O.quantize_layer(S.gen_W(cfg), S.gen_X(cfg), cfg)
    cl = out["crit_loss_after_ext"]
    assert all(b <= a * (1 + 1e-9) for a, b in zip(cl, cl[1:]))
    ob = out["base_objective"]
    assert all(b <= a * (1 + 1e-9) for a, b in zip(ob, ob[1:]))
    h = out["loss_history"]
    assert h[-1] <= h[0] * (1 + 1e-9)
    assert out["loss_full"] > 0


# ---------------------------------------------------------------- schedule wiring pins
# These restate the per-matrix schedule (Alg. 1, prequantization through the refinement loop)
# by hand on cases whose result has a closed form, so that a wiring slip (a step fed the
# wrong matrix, Hessian blocks, seed, residual or order) fails one of them. They use only
# numpy and the synthetic generator, none of the oracle's step functions.
def _h64(X, damp_rel):
    """H = X^T X / n + delta I in fp64, the undamped diagonal and delta (App. A.2 proxy with
    the damping reading)."""
    X = np.asarray(X, np.float64)
    S_ = X.T @ X / X.shape[0]
    xsq = np.diag(S_).copy()
    delta = float(np.float32(damp_rel)) * xsq.mean()
    return S_ + delta * np.eye(S_.shape[0]), xsq, delta


def _blocks(H, perm, d):
    Hp = H[np.ix_(perm, perm)]
    return [Hp[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(len(perm) // d)]


def _wmean(pairs):
    """argmin_c sum (t - c)^T H (t - c) over (H, t) pairs: (sum H)^-1 sum H t."""
    A = sum(H for H, _ in pairs)
    b = sum(H @ t for H, t in pairs)
    return np.linalg.solve(A, b)


def _seed(seed, phase, cb):
    return int(S.splitmix64(seed, np.array([phase * 1024 + cb]))[0])


def _strata(n, K, seed):
    """One vector index per stratum [floor(k n / K), floor((k+1) n / K))."""
    out = []
    for k in range(K):
        lo, hi = (k * n) // K, ((k + 1) * n) // K
        out.append(lo + int(S.splitmix64(seed, np.array([k]))[0]) % (hi - lo))
    return out


def _nearest(t, C, Hg):
    e = [float((t - c) @ Hg @ (t - c)) for c in np.asarray(C, np.float64)]
    return int(np.argmin(e))


def _importance_perm(W, W_pre, xsq):
    I = 0.5 * xsq * np.max((np.asarray(W, np.float64) - W_pre) ** 2, axis=0)
    return np.array(sorted(range(len(I)), key=lambda j: (-I[j], j)))


def test_schedule_with_one_codeword_per_codebook_is_a_sequence_of_weighted_means():
    """K_base = K_ext = 1: every code is 0, so each Lloyd fit is the H-weighted mean of its
    targets (Sec. 3.1 Eq. kmeans with one cluster) and the schedule is a fixed sequence of
    such means: prequantize in the original order, importance from that reconstruction
    (App. A.2), base on the reordered W with the reordered H blocks, each extended codebook on
    the critical residual of the base and earlier extended codebooks (Sec. 4.3), then one
    refinement round updating base, ext 1, ext 2 in that order with the others fixed."""
    cfg = S.LayerConfig("pin_k1", 6, 32, 48, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=2, K_base=1, n_ext=2, K_ext=1, crit_frac=0.3, B=2,
                        kmeans_iters=2, refine_rounds=1)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = O.quantize_layer(W, X, cfg)
    d, M, N = 8, cfg.M, cfg.N
    G = N // d
    Gc = 2                                             # ceil(0.3 * 32 / 8)
    H, xsq, delta = _h64(X, cfg.damp_rel)
    W64 = W.astype(np.float64)
    vec = lambda A, i, g: A[i, g * d:(g + 1) * d]
    H0 = _blocks(H, np.arange(N), d)
    c_pre = _wmean([(H0[g], vec(W64, i, g)) for i in range(M) for g in range(G)])
    perm = _importance_perm(W, np.tile(c_pre, G)[None, :], xsq)
    Ws = W64[:, perm]
    Hs = _blocks(H, perm, d)
    c_b = _wmean([(Hs[g], vec(Ws, i, g)) for i in range(M) for g in range(G)])
    crit = [(i, g) for i in range(M) for g in range(Gc)]
    c_1 = _wmean([(Hs[g], vec(Ws, i, g) - c_b) for i, g in crit])
    c_2 = _wmean([(Hs[g], vec(Ws, i, g) - c_b - c_1) for i, g in crit])
    # one refinement round: base, then ext 1, then ext 2, each with the others fixed
    c_b = _wmean([(Hs[g], vec(Ws, i, g) - (c_1 + c_2 if g < Gc else 0.0))
                  for i in range(M) for g in range(G)])
    c_1 = _wmean([(Hs[g], vec(Ws, i, g) - c_b - c_2) for i, g in crit])
    c_2 = _wmean([(Hs[g], vec(Ws, i, g) - c_b - c_1) for i, g in crit])

    scale = np.abs(c_pre).max()   # the second extended codeword is ~0 (its residual's
                                  # weighted mean is zero once ext 1 fits it): absolute scale

    def close(a, b):
        np.testing.assert_allclose(np.asarray(a, np.float64).reshape(-1), b, rtol=0,
                                   atol=2e-5 * scale)
    close(out["C_pre"], c_pre)
    np.testing.assert_array_equal(out["perm"], perm)
    assert out["n_crit_groups"] == Gc
    cbs = out["codebooks"]
    close(cbs[0].C, c_b)
    close(cbs[1].C, c_1)
    close(cbs[2].C, c_2)
    rec = np.tile(c_b, G)
    rec[:Gc * d] += np.tile(c_1 + c_2, Gc)
    D = Ws - rec[None, :]
    lb = sum(float(vec(D, i, g) @ Hs[g] @ vec(D, i, g)) for i in range(M) for g in range(G))
    lc = sum(float(vec(D, i, g) @ Hs[g] @ vec(D, i, g)) for i, g in crit)
    Dorig = np.empty_like(D)
    Dorig[:, perm] = D
    lf = float(np.einsum("ij,jk,ik->", Dorig, H, Dorig))
    assert out["loss_block"] == pytest.approx(lb, rel=1e-5)
    assert out["loss_crit"] == pytest.approx(lc, rel=1e-5)
    assert out["loss_full"] == pytest.approx(lf, rel=1e-5)


def test_schedule_without_lloyd_iterations_keeps_the_sampled_codewords():
    """kmeans_iters = 0 and no refinement: each codebook is its k-means initialisation, the
    vectors (or critical residuals) drawn from the strata with that phase's seed, and the
    codes are the arg-min encodes. The prequantize codebook comes from W in the original order
    (phase 1), the base from the reordered W (phase 2, a fresh draw, not the prequantize
    codebook), extended codebook t from the critical residual after the base and the earlier
    extended codebooks (phase 3, codebook t)."""
    cfg = S.LayerConfig("pin_t0", 8, 32, 40, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=2, K_base=8, n_ext=2, K_ext=4, crit_frac=0.3, B=2,
                        kmeans_iters=0, refine_rounds=0, seed=5)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = O.quantize_layer(W, X, cfg)
    d, M, N = 8, cfg.M, cfg.N
    G, Gc = N // d, 2
    H, xsq, _ = _h64(X, cfg.damp_rel)
    W64 = W.astype(np.float64)
    vec = lambda A, v, Gs: A[v // Gs, (v % Gs) * d:(v % Gs + 1) * d]
    H0 = _blocks(H, np.arange(N), d)
    C_pre = np.stack([vec(W64, v, G) for v in _strata(M * G, 8, _seed(5, 1, 0))])
    W_pre = np.concatenate([C_pre[[_nearest(vec(W64, i * G + g, G), C_pre, H0[g])
                                   for i in range(M)]] for g in range(G)], axis=1)
    perm = _importance_perm(W, W_pre, xsq)
    Ws = W64[:, perm]
    Hs = _blocks(H, perm, d)
    C_b = np.stack([vec(Ws, v, G) for v in _strata(M * G, 8, _seed(5, 2, 0))])
    code_b = np.array([[_nearest(vec(Ws, i * G + g, G), C_b, Hs[g]) for g in range(G)]
                       for i in range(M)])
    res = np.stack([vec(Ws, i * G + g, G) - C_b[code_b[i, g]] for i in range(M)
                    for g in range(Gc)])               # critical residual, vector i * Gc + g
    C_e, code_e = [], []
    for t in (1, 2):
        Ct = res[_strata(M * Gc, 4, _seed(5, 3, t))]
        ct = np.array([_nearest(res[v], Ct, Hs[v % Gc]) for v in range(M * Gc)])
        res = res - Ct[ct]
        C_e.append(Ct)
        code_e.append(ct.reshape(M, Gc))
    np.testing.assert_array_equal(out["C_pre"], C_pre.astype(np.float32))
    np.testing.assert_array_equal(out["perm"], perm)
    cbs = out["codebooks"]
    np.testing.assert_array_equal(cbs[0].C, C_b.astype(np.float32))
    np.testing.assert_array_equal(cbs[0].codes, code_b)
    for t in range(2):
        np.testing.assert_allclose(cbs[t + 1].C, C_e[t], rtol=0, atol=1e-7)
        np.testing.assert_array_equal(cbs[t + 1].codes, code_e[t])


def test_schedule_with_two_base_codebooks_of_one_codeword_each():
    """Two base codebooks (Sec. 6.4's m = 2 setting) with one codeword each, one extended
    codebook of one codeword: the second base is the H-weighted mean of the residual of the
    first over every group (which is zero), the extended codebook that of the residual of both
    on the critical groups, and the refinement round updates base 1, base 2, ext 1 in that
    order with the others fixed."""
    _two_base_one_codeword(8)


def test_schedule_with_two_base_codebooks_of_one_codeword_each_at_d16():
    """The same at d = 16, the vector length of Sec. 6.4's m = 2 setting."""
    _two_base_one_codeword(16)


def _two_base_one_codeword(d):
    cfg = S.LayerConfig("pin_m2_k1", 6, 32, 48, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=2, K_base=1, n_ext=1, K_ext=1, crit_frac=0.3, B=2,
                        kmeans_iters=2, refine_rounds=1, n_base=2, d=d)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = O.quantize_layer(W, X, cfg)
    M, N = cfg.M, cfg.N
    G, Gc = N // d, -(-3 * N // (10 * d))             # ceil(0.3 * N / d)
    H, xsq, _ = _h64(X, cfg.damp_rel)
    W64 = W.astype(np.float64)
    vec = lambda A, i, g: A[i, g * d:(g + 1) * d]
    H0 = _blocks(H, np.arange(N), d)
    c_pre = _wmean([(H0[g], vec(W64, i, g)) for i in range(M) for g in range(G)])
    perm = _importance_perm(W, np.tile(c_pre, G)[None, :], xsq)
    Ws = W64[:, perm]
    Hs = _blocks(H, perm, d)
    every = [(i, g) for i in range(M) for g in range(G)]
    crit = [(i, g) for i in range(M) for g in range(Gc)]
    c_1 = _wmean([(Hs[g], vec(Ws, i, g)) for i, g in every])
    c_2 = _wmean([(Hs[g], vec(Ws, i, g) - c_1) for i, g in every])
    c_e = _wmean([(Hs[g], vec(Ws, i, g) - c_1 - c_2) for i, g in crit])
    ext = lambda g: c_e if g < Gc else 0.0
    c_1 = _wmean([(Hs[g], vec(Ws, i, g) - c_2 - ext(g)) for i, g in every])
    c_2 = _wmean([(Hs[g], vec(Ws, i, g) - c_1 - ext(g)) for i, g in every])
    c_e = _wmean([(Hs[g], vec(Ws, i, g) - c_1 - c_2) for i, g in crit])
    scale = np.abs(c_pre).max()
    cbs = out["codebooks"]
    assert len(cbs) == 3 and [cb.G_cov for cb in cbs] == [G, G, Gc]
    for cb, c in zip(cbs, (c_1, c_2, c_e)):
        np.testing.assert_allclose(np.asarray(cb.C, np.float64).reshape(-1), c, rtol=0,
                                   atol=2e-5 * scale)
    rec = np.tile(c_1 + c_2, G)
    rec[:Gc * d] += np.tile(c_e, Gc)
    D = Ws - rec[None, :]
    lb = sum(float(vec(D, i, g) @ Hs[g] @ vec(D, i, g)) for i, g in every)
    assert out["loss_block"] == pytest.approx(lb, rel=1e-5)


def test_schedule_with_two_base_codebooks_without_lloyd_iterations():
    """Two base codebooks, kmeans_iters = 0, no refinement: base 2 is drawn (phase 2,
    codebook 1) from the residual of base 1 over every group and encodes that residual; the
    extended codebook is drawn (phase 3, codebook 1) from the critical residual of both."""
    cfg = S.LayerConfig("pin_m2_t0", 8, 32, 40, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=2, K_base=8, n_ext=1, K_ext=4, crit_frac=0.3, B=2,
                        kmeans_iters=0, refine_rounds=0, seed=7, n_base=2)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = O.quantize_layer(W, X, cfg)
    d, M, N = 8, cfg.M, cfg.N
    G, Gc = N // d, 2
    H, xsq, _ = _h64(X, cfg.damp_rel)
    W64 = W.astype(np.float64)
    vec = lambda A, v, Gs: A[v // Gs, (v % Gs) * d:(v % Gs + 1) * d]
    H0 = _blocks(H, np.arange(N), d)
    C_pre = np.stack([vec(W64, v, G) for v in _strata(M * G, 8, _seed(7, 1, 0))])
    W_pre = np.concatenate([C_pre[[_nearest(vec(W64, i * G + g, G), C_pre, H0[g])
                                   for i in range(M)]] for g in range(G)], axis=1)
    perm = _importance_perm(W, W_pre, xsq)
    Ws = W64[:, perm]
    Hs = _blocks(H, perm, d)
    res = np.stack([vec(Ws, v, G) for v in range(M * G)])      # vector v = i * G + g
    C_b, code_b = [], []
    for b in (0, 1):
        Cb = res[_strata(M * G, 8, _seed(7, 2, b))]
        cb = np.array([_nearest(res[v], Cb, Hs[v % G]) for v in range(M * G)])
        res = res - Cb[cb]
        C_b.append(Cb)
        code_b.append(cb.reshape(M, G))
    rc = np.stack([res[i * G + g] for i in range(M) for g in range(Gc)])
    C_e = rc[_strata(M * Gc, 4, _seed(7, 3, 1))]
    code_e = np.array([_nearest(rc[v], C_e, Hs[v % Gc]) for v in range(M * Gc)])
    np.testing.assert_array_equal(out["perm"], perm)
    cbs = out["codebooks"]
    for b in (0, 1):
        np.testing.assert_allclose(cbs[b].C, C_b[b], rtol=0, atol=1e-7)
        np.testing.assert_array_equal(cbs[b].codes, code_b[b])
    np.testing.assert_allclose(cbs[2].C, C_e, rtol=0, atol=1e-7)
    np.testing.assert_array_equal(cbs[2].codes, code_e.reshape(M, Gc))


def test_schedule_with_a_codeword_per_vector_reconstructs_exactly():
    """K_base equal to the number of vectors: the strata hold one vector each, so the base
    k-means starts from every vector of the reordered W and the reconstruction is exact; the
    extended codebooks then fit a zero residual. Every loss is zero and W_hat equals W."""
    cfg = S.LayerConfig("pin_kall", 4, 32, 40, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=2, K_base=16, n_ext=1, K_ext=2, crit_frac=0.3, B=2,
                        kmeans_iters=2, refine_rounds=1)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = O.quantize_layer(W, X, cfg)
    assert out["loss_block"] == 0.0 and out["loss_crit"] == 0.0
    assert abs(out["loss_full"]) <= 1e-12 * float((W.astype(np.float64) ** 2).sum())
    np.testing.assert_array_equal(out["W_hat"], W)


def test_schedule_puts_a_dominant_channel_first():
    """One input channel whose weights and activations dwarf the rest has the largest App. A.2
    importance, so the reorder puts it first and the critical set is ceil(lambda N / d) whole
    groups."""
    cfg = S.LayerConfig("pin_dom", 16, 64, 64, "plain", "lognormal", 0.3, K_base=4, n_ext=1,
                        K_ext=2, crit_frac=0.05, B=2, kmeans_iters=2, refine_rounds=1)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    W[:, 37] *= 100.0
    X[:, 37] *= 100.0
    out = O.quantize_layer(W, X, cfg)
    assert out["perm"][0] == 37
    assert out["n_crit_groups"] == 1                   # ceil(0.05 * 64 / 8)
    np.testing.assert_array_equal(np.sort(out["perm"]), np.arange(64))


# ---------------------------------------------------------------- NEXT-1 coupled search
def _coupled_case(seed, M=6, G=3, d=4, K=5, n=40):
    rng = np.random.default_rng(seed)
    N = G * d
    X = rng.standard_normal((n, N)) @ rng.standard_normal((N, N)) * 0.4   # correlated channels
    H = X.T @ X / n + 0.05 * np.eye(N)
    W = rng.standard_normal((M, N)).astype(np.float32)
    C = rng.standard_normal((K, d)).astype(np.float32)
    codes = rng.integers(0, K, (M, G))
    return W, H, C, codes, d, G


def _row_loss(w, H, rec):
    D = np.asarray(w, np.float64) - rec
    return float(D @ H @ D)


def test_coupled_sweep_never_raises_the_full_loss():
    W, H, C, codes, d, G = _coupled_case(31)
    cbs = [O.Codebook(C, codes, G)]
    before = O.full_loss(W, H, cbs)
    new, hist = O.coupled_sweep(W, d, H, cbs, 0, sweeps=3)
    seq = [before] + hist
    assert all(b <= a * (1 + 1e-12) for a, b in zip(seq, seq[1:]))
    assert hist[-1] < before
    assert abs(O.full_loss(W, H, [O.Codebook(C, new, G)]) - hist[-1]) <= 1e-9 * hist[-1]


def test_coupled_sweep_with_block_diagonal_H_is_the_plain_encode():
    W, H, C, codes, d, G = _coupled_case(32)
    Hb = np.zeros_like(H)
    for g in range(G):
        Hb[g * d:(g + 1) * d, g * d:(g + 1) * d] = H[g * d:(g + 1) * d, g * d:(g + 1) * d]
    new, _ = O.coupled_sweep(W, d, Hb, [O.Codebook(C, codes, G)], 0)
    blocks = np.stack([Hb[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(G)])
    ref, _ = O.encode_beam(W, d, blocks.astype(np.float32), [O.Codebook(C, None, G)], 0, 1)
    np.testing.assert_array_equal(new, ref[0])


def test_coupled_sweep_fixed_point_is_optimal_per_group_by_brute_force():
    """Swept to a fixed point, no single (row, group) code change lowers the row's full loss,
    evaluated directly as (w - w_enc)^T H (w - w_enc)."""
    W, H, C, codes, d, G = _coupled_case(33)
    cbs = [O.Codebook(C, codes, G)]
    for _ in range(20):
        new, _ = O.coupled_sweep(W, d, H, cbs, 0)
        done = np.array_equal(new, cbs[0].codes)
        cbs = [O.Codebook(C, new, G)]
        if done:
            break
    assert done
    C64 = C.astype(np.float64)
    for i in range(W.shape[0]):
        rec = np.concatenate([C64[new[i, g]] for g in range(G)])
        base = _row_loss(W[i], H, rec)
        for g in range(G):
            for k in range(C.shape[0]):
                trial = rec.copy()
                trial[g * d:(g + 1) * d] = C64[k]
                assert _row_loss(W[i], H, trial) >= base * (1 - 1e-12) - 1e-12


def test_coupled_sweep_between_exhaustive_optimum_and_block_diagonal_start():
    W, H, C, codes, d, G = _coupled_case(34, M=3, G=2, K=4)
    blocks = np.stack([H[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(G)])
    start, _ = O.encode_beam(W, d, blocks.astype(np.float32), [O.Codebook(C, None, G)], 0, 1)
    new, _ = O.coupled_sweep(W, d, H, [O.Codebook(C, start[0], G)], 0, sweeps=4)
    C64 = C.astype(np.float64)
    for i in range(W.shape[0]):
        best = min(_row_loss(W[i], H, np.concatenate([C64[a], C64[b]]))
                   for a in range(4) for b in range(4))
        got = _row_loss(W[i], H, np.concatenate([C64[new[i, 0]], C64[new[i, 1]]]))
        init = _row_loss(W[i], H, np.concatenate([C64[start[0][i, 0]], C64[start[0][i, 1]]]))
        assert best * (1 - 1e-12) <= got <= init * (1 + 1e-12)


def test_coupled_sweep_of_second_codebook_is_the_sweep_on_the_residual():
    W, H, C, codes, d, G = _coupled_case(35)
    rng = np.random.default_rng(36)
    C0 = rng.standard_normal((7, d)).astype(np.float32)
    c0 = rng.integers(0, 7, (W.shape[0], G))
    a, ha = O.coupled_sweep(W, d, H, [O.Codebook(C0, c0, G), O.Codebook(C, codes, G)], 1)
    R = W.astype(np.float64) - np.concatenate([C0[c0[:, g]] for g in range(G)], axis=1)
    b, hb = O.coupled_sweep(R, d, H, [O.Codebook(C, codes, G)], 0)
    np.testing.assert_array_equal(a, b)
    np.testing.assert_allclose(ha, hb, rtol=1e-9)


# ---------------------------------------------------------------- NEXT-3 inference product
def test_lut_matvec_equals_the_reconstructed_matrix_times_the_input():
    """Lookup-table product vs the explicit route: W_hat (reconstruct_error, original order)
    times the inputs by a matrix product."""
    rng = np.random.default_rng(41)
    M, N, d, Gc = 7, 32, 8, 2
    W = rng.standard_normal((M, N)).astype(np.float32)
    perm = rng.permutation(N).astype(np.int32)
    C0 = rng.standard_normal((9, d)).astype(np.float32)
    C1 = (0.3 * rng.standard_normal((5, d))).astype(np.float32)
    cbs = [O.Codebook(C0, rng.integers(0, 9, (M, N // d)), N // d),
           O.Codebook(C1, rng.integers(0, 5, (M, Gc)), Gc)]
    Hb = np.stack([np.eye(d, dtype=np.float32)] * (N // d))
    W_hat = O.reconstruct_error(W[:, perm], d, Hb, perm, cbs, Gc)[0]
    Xin = rng.standard_normal((3, N))
    np.testing.assert_allclose(O.lut_matvec(Xin, perm, cbs, d),
                               Xin @ W_hat.astype(np.float64).T, rtol=1e-6, atol=1e-6)
    # without a permutation the sorted order is the original one
    W_id = O.reconstruct_error(W, d, Hb, None, cbs, Gc)[0]
    np.testing.assert_allclose(O.lut_matvec(Xin, None, cbs, d),
                               Xin @ W_id.astype(np.float64).T, rtol=1e-6, atol=1e-6)
    # a permuted input channel moves with its weight column
    e = np.zeros(N)
    e[perm[5]] = 1.0
    np.testing.assert_allclose(O.lut_matvec(e, perm, cbs, d)[0], W_hat[:, perm[5]], rtol=1e-6)


def test_beam_ties_follow_err_then_parent_rank_then_index():
    """Exact ties (integer codewords, H = I): stage 0 orders equal errors by codeword index;
    the last stage orders equal errors by parent rank, then index."""
    d = 2
    C0 = np.array([[0, 0], [2, 0]], np.float32)       # both at err 1 from t = (1, 0)
    C1 = np.array([[1, 0], [-1, 0]], np.float32)      # (0, 0) and (1, 1) both reach err 0
    T = np.array([[1, 0]], np.float32)
    Hb = np.eye(d, dtype=np.float32)[None]
    for B in (1, 2, 4):
        codes, verr = O.encode_beam(T, d, Hb, [O.Codebook(C0, None, 1),
                                               O.Codebook(C1, None, 1)], 0, B)
        assert (codes[0][0, 0], codes[1][0, 0]) == (0, 0), B
        assert verr[0, 0] == 0.0
    # a single codebook with two equal codewords: the smaller index
    codes, _ = O.encode_beam(T, d, Hb, [O.Codebook(np.array([[1, 1], [1, -1], [1, 1]],
                                                            np.float32), None, 1)], 0, 1)
    assert codes[0][0, 0] == 0
