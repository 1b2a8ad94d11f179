"""CRVQ oracle: a plain, slow fp64 CPU statement of the Hessian-weighted additive-codebook
code search (arXiv 2412.09282, Alg. 1 with Sec. 3.1, Sec. 4.1-4.3 and App. A.1-A.2).

TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
leg may import this module. The CUDA library shares no code with it, and it imports nothing
from the CUDA package.

Arithmetic is numpy float64 throughout; every function that mirrors a C-ABI call rounds its
floating outputs to float32 once, at the end, as the library's outputs are float32.

Data model (shared vocabulary with the C-ABI):
  * W is M x N (rows = output features, columns = input channels, Sec. 3.1). A vector is the
    length-d row segment W[i, g*d:(g+1)*d] (Eq. for S in Sec. 3.1); G = N/d groups.
  * X is n_tok x N (row = token). The paper writes X as N x O and the Hessian proxy as XX^T
    (App. A.2); ours is X^T X, the same matrix.
  * A vector set is a row-major M x (G_sub*d) block of a matrix with leading dimension ldT;
    vector (i, g) is scored with the d x d Hessian block H_blocks[g].
  * A codebook is (C: K x d, codes: M x G_cov int, G_cov): it covers groups g < G_cov of the
    set. The base codebook (each of them, with several, Sec. 6.4) covers every group; the
    extended codebooks cover only the first G_c groups, which hold the reordered critical
    channels (Sec. 4.3, Fig. 2). The
    reconstruction of vector (i, g) is the sum of C_s[codes_s[i, g]] over the codebooks
    that cover g (additive VQ, Sec. 3.1 last paragraph and Sec. 4.3).

Readings where the paper is silent or ambiguous (all listed in the design notes):
  * Vector-to-codeword score is the block-diagonal part of the Alg. 1 loss
    ||WX - W_enc X||^2: err(t, c) = (t - c)^T H_g (t - c). With H_g = cI it is the plain L2
    nearest codeword of Sec. 3.1 Eq. (2)-(3).
  * Importance uses the App. A.2 form I_i = max_j 1/2 sum_k (x_ik dw_ji)^2
    = 1/2 * xsq_i * max_j dw_ji^2 (with xsq the mean of squares, a constant factor 1/n);
    Eq. (wa) in Sec. 4.1 divides by an inverse-Hessian diagonal instead, which the App. A.2
    expansion does not reproduce; the App. A.2 form is the default. Eq. (wa) as printed is
    the mode MODE_WA_INV, with the inverse taken of the damped proxy H (the undamped X^T X is
    singular whenever there are fewer tokens than channels; the factor 1/n scales every I_i
    alike and leaves the order unchanged).
  * Damping: H = X^T X / n + delta I, delta = damp_rel * mean_i xsq_i (the paper has none;
    it keeps the LS codebook solves well posed).
  * k-means init: one vector drawn from each of K equal strata of the vector index range,
    by SplitMix64; empty clusters keep their old codeword.
  * FineTuneCodebook (Alg. 1) is the closed-form least-squares update of one codebook with
    the others fixed, under the same H-weighted objective.
  * BeamSearchOptimize (Alg. 1) is a stage-wise beam over the codebooks that cover a
    vector, in codebook order, keeping the B best partial tuples by (err, parent rank, k).

Beyond the per-matrix schedule (each pinned in the tests):
  * MODE_WA_INV / hinv_diag: Eq. (wa) with the inverse-Hessian diagonal;
  * coupled_sweep / full_loss: code search under the full Alg. 1 loss, cross-group terms
    included (Gauss-Seidel over groups);
  * lut_matvec: the inference product from codes, without forming W_enc.
"""
from __future__ import annotations

import math

import numpy as np

# Importance modes (Sec. 4.1 and Sec. 6.3 / Table 2); MODE_WA_INV is Eq. (wa) as printed.
MODE_WA, MODE_WONLY, MODE_RANDOM, MODE_WA_INV = 0, 1, 2, 3

_GAMMA = 0x9E3779B97F4A7C15
_MASK = 0xFFFFFFFFFFFFFFFF


def splitmix64(stream: int, counter: int) -> int:
    """Output `counter` (0-based) of the SplitMix64 stream `stream` (Steele et al. 2014)."""
    z = (stream + (counter + 1) * _GAMMA) & _MASK
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK
    return z ^ (z >> 31)


def f32(a):
    return np.asarray(a, dtype=np.float64).astype(np.float32)


class Codebook:
    """One codebook of a vector set: K x d codewords, codes (M x G_cov) and its coverage."""

    def __init__(self, C, codes, G_cov):
        self.C = np.asarray(C, dtype=np.float32)
        self.codes = None if codes is None else np.asarray(codes, dtype=np.int64)
        self.G_cov = int(G_cov)

    @property
    def K(self):
        return self.C.shape[0]


# --------------------------------------------------------------------------------------
# S1: Hessian proxy (Alg. 1 "Require: XX^T"; App. A.2)
# --------------------------------------------------------------------------------------
def hessian(X, damp_rel, d):
    """H = X^T X / n + delta I with delta = damp_rel * mean(diag(X^T X / n)).

    Returns (H fp32 N x N, xsq fp32 N = undamped diagonal, H_blocks fp32 (N/d) x d x d in
    the original channel order, delta fp32)."""
    X = np.asarray(X, dtype=np.float64)
    n, N = X.shape
    S = (X.T @ X) / n                        # App. A.2: entries sum_k x_ik x_jk
    xsq = np.diag(S).copy()
    delta = float(np.float32(damp_rel)) * xsq.mean()
    H = S + delta * np.eye(N)
    H32 = f32(H)
    G = N // d
    Hb = np.stack([H32[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(G)]) if G else \
        np.zeros((0, d, d), np.float32)
    return H32, f32(xsq), Hb, np.float32(delta)


# --------------------------------------------------------------------------------------
# S3: channel importance (Sec. 4.1, App. A.2) and reordering (Sec. 4.2)
# --------------------------------------------------------------------------------------
def n_crit_groups(N, d, crit_frac):
    """Critical groups: ceil(lambda*N/d) whole groups, at most N/d (Sec. 4.3 ratio lambda)."""
    lam = float(np.float32(crit_frac))
    return min(N // d, int(math.ceil(lam * N / d - 1e-12))) if lam > 0 else 0


def hinv_diag(H):
    """diag(H^-1) of a symmetric positive definite H (fp64): with the Cholesky factor
    H = L L^T, H^-1 = L^-T L^-1, so [H^-1]_ii = sum_k (L^-1)_ki^2 (the denominator of Eq. (wa),
    Sec. 4.1)."""
    import scipy.linalg
    H = np.asarray(H, dtype=np.float64)
    L = np.linalg.cholesky(H)
    Linv = scipy.linalg.solve_triangular(L, np.eye(H.shape[0]), lower=True)
    return np.sum(Linv * Linv, axis=0)


def importance(W, W_pre, xsq, mode, seed, hinv=None):
    """Per-channel importance I (fp64).

    W-A  (App. A.2): I_i = max_j 1/2 * xsq_i * (w_ji - VQ(w_ji))^2.
    W-only (Sec. 4.1): I_i = max_j w_ji^2.
    random (Table 2): I_i = a 24-bit uniform from SplitMix64(seed, i).
    W-A inverse (Eq. (wa)): I_i = max_j (w_ji - VQ(w_ji))^2 / (2 [H^-1]_ii), hinv = diag(H^-1)."""
    W = np.asarray(W, dtype=np.float64)
    M, N = W.shape
    if mode == MODE_WA:
        dW = W - np.asarray(W_pre, dtype=np.float64)
        return 0.5 * np.asarray(xsq, np.float64) * np.max(dW * dW, axis=0)
    if mode == MODE_WA_INV:
        dW = W - np.asarray(W_pre, dtype=np.float64)
        return np.max(dW * dW, axis=0) / (2.0 * np.asarray(hinv, np.float64))
    if mode == MODE_WONLY:
        return np.max(W * W, axis=0)
    if mode == MODE_RANDOM:
        return np.array([(splitmix64(seed, i) >> 40) * 2.0 ** -24 for i in range(N)])
    raise ValueError(mode)


def select_reorder_channels(W, d, W_pre, xsq, H, crit_frac, mode, seed):
    """Alg. 1 ComputeImportance + ReorderChannels.

    perm sorts channels by importance, descending, ties by original index; perm[new] = old.
    W_sorted[:, p] = W[:, perm[p]]; H_blocks[g][a][b] = H[perm[g d + a], perm[g d + b]].
    Returns (perm int32, importance fp32, W_sorted fp32, H_blocks fp32, n_crit_groups)."""
    W = np.asarray(W, dtype=np.float32)
    M, N = W.shape
    hinv = hinv_diag(H) if mode == MODE_WA_INV else None
    I = importance(W, W_pre, xsq, mode, seed, hinv)
    perm = np.lexsort((np.arange(N), -I)).astype(np.int32)
    Ws = W[:, perm]
    H = np.asarray(H, dtype=np.float32)
    G = N // d
    Hb = np.stack([H[np.ix_(perm[g * d:(g + 1) * d], perm[g * d:(g + 1) * d])]
                   for g in range(G)])
    return perm, f32(I), np.ascontiguousarray(Ws), Hb, n_crit_groups(N, d, crit_frac)


# --------------------------------------------------------------------------------------
# Vector-set helpers
# --------------------------------------------------------------------------------------
def _group(T, g, d):
    return np.asarray(T[:, g * d:(g + 1) * d], dtype=np.float64)


def _fixed_sum(cbs, g, M, d, skip=()):
    """Sum over the codebooks that cover group g (except those in `skip`) of C[code]."""
    acc = np.zeros((M, d))
    for s, cb in enumerate(cbs):
        if s in skip or g >= cb.G_cov:
            continue
        acc += cb.C.astype(np.float64)[cb.codes[:, g]]
    return acc


def _recon(cbs, g, rows):
    """Sum of C_s[codes_s[rows, g]] over the given codebooks that cover group g."""
    acc = 0.0
    for cb in cbs:
        if g < cb.G_cov:
            acc = acc + cb.C.astype(np.float64)[cb.codes[rows, g]]
    return acc


def quad_err(R, C, Hg):
    """err[v, k] = (R_v - C_k)^T Hg (R_v - C_k) in fp64 (Sec. 3.1 score under the Alg. 1 loss)."""
    D = R[:, None, :] - C[None, :, :]
    return np.einsum("vkd,vkd->vk", D @ Hg, D)


# --------------------------------------------------------------------------------------
# k-means init (Eq. kmeans, Sec. 3.1; Alg. 1 KMeansCodebook)
# --------------------------------------------------------------------------------------
def kmeans_sample_indices(n, K, seed):
    """Stratified draw: idx_k = floor(k n / K) + SplitMix64(seed, k) mod stratum size."""
    out = np.empty(K, dtype=np.int64)
    for k in range(K):
        lo = (k * n) // K
        hi = ((k + 1) * n) // K
        out[k] = lo + splitmix64(seed, k) % (hi - lo)
    return out


def kmeans_init(T, d, G_sub, K, seed, fixed=()):
    """Initial codebook: the residuals (w.r.t. the fixed codebooks) of K sampled vectors."""
    T = np.asarray(T, dtype=np.float32)
    M = T.shape[0]
    n = M * G_sub
    if K > n:
        raise ValueError("K exceeds the number of vectors")
    idx = kmeans_sample_indices(n, K, seed)
    C = np.empty((K, d))
    for k, v in enumerate(idx):
        i, g = divmod(int(v), G_sub)
        r = T[i, g * d:(g + 1) * d].astype(np.float64)
        for cb in fixed:
            if g < cb.G_cov:
                r = r - cb.C[cb.codes[i, g]].astype(np.float64)
        C[k] = r
    return f32(C)


# --------------------------------------------------------------------------------------
# Encode / beam search (Sec. 3.1 Eq. (2)-(3); Alg. 1 VectorQuant and BeamSearchOptimize)
# --------------------------------------------------------------------------------------
def encode_beam(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, row_chunk=512):
    """Codes for codebooks n_fixed..n_cb-1 of every vector in the set.

    Target = vector minus the reconstruction of the fixed codebooks 0..n_fixed-1. The
    searched codebooks that cover a vector are taken in order; each stage extends every kept
    partial tuple by every codeword and keeps the B smallest by (err, parent rank, k). The
    result is the best tuple of the last stage. With keep_if_better, the tuple already in the
    searched codebooks' codes is kept when its err is strictly smaller.
    Returns (codes: list of M x G_cov int32 arrays, None for fixed ones; vec_err M x G_sub)."""
    T = np.asarray(T, dtype=np.float32)
    M = T.shape[0]
    G_sub = H_blocks.shape[0]
    out = [None if s < n_fixed else
           (cb.codes.copy() if cb.codes is not None else np.zeros((M, cb.G_cov), np.int64))
           for s, cb in enumerate(cbs)]
    vec_err = np.zeros((M, G_sub))
    for g in range(G_sub):
        Hg = np.asarray(H_blocks[g], dtype=np.float64)
        searched = [s for s in range(n_fixed, len(cbs)) if g < cbs[s].G_cov]
        for r0 in range(0, M, row_chunk):
            rows = slice(r0, min(M, r0 + row_chunk))
            t = _group(T[rows], g, d)
            m = t.shape[0]
            base = t - _recon(cbs[:n_fixed], g, rows)
            res = base[:, None, :]                      # m x Bh x d
            err = quad_err(base, np.zeros((1, d)), Hg)  # m x 1 (no searched codebook)
            codes = np.zeros((m, 1, 0), dtype=np.int64)
            ar = np.arange(m)[:, None]
            for s in searched:
                C = cbs[s].C.astype(np.float64)
                K = C.shape[0]
                Bh = res.shape[1]
                D = res[:, :, None, :] - C[None, None, :, :]          # m x Bh x K x d
                e = np.einsum("mhkd,mhkd->mhk", D @ Hg, D).reshape(m, Bh * K)
                keep = min(B, Bh * K)
                order = np.argsort(e, axis=1, kind="stable")[:, :keep]  # (err, h, k) order
                h, k = order // K, order % K
                res = res[ar, h] - C[k]
                codes = np.concatenate([codes[ar, h], k[:, :, None]], axis=2)
                err = np.take_along_axis(e, order, axis=1)
            best_err = err[:, 0]
            best = codes[:, 0, :]
            if keep_if_better and searched:
                old = np.stack([cbs[s].codes[rows, g] for s in searched], axis=1)
                rec = sum(cbs[s].C.astype(np.float64)[old[:, j]] for j, s in enumerate(searched))
                D = base - rec
                old_err = np.einsum("vd,vd->v", D @ Hg, D)
                use_old = old_err < best_err
                best = np.where(use_old[:, None], old, best)
                best_err = np.where(use_old, old_err, best_err)
            for j, s in enumerate(searched):
                out[s][rows, g] = best[:, j]
            vec_err[rows, g] = best_err
    return [None if o is None else o.astype(np.int32) for o in out], f32(vec_err)


# --------------------------------------------------------------------------------------
# Codebook least-squares update (Alg. 1 KMeansCodebook update step / FineTuneCodebook)
# --------------------------------------------------------------------------------------
def update_codebook(T, d, H_blocks, cbs, which):
    """Codebook `which` re-fitted with all other codebooks fixed.

    Each member v of cluster k has target tau_v = t_v - sum_{s != which} C_s[code_s(v)];
    c_k minimises sum_v (tau_v - c)^T H_{g_v} (tau_v - c), i.e. solves
    (sum_v H_{g_v}) c = sum_v H_{g_v} tau_v. Empty clusters keep their codeword.
    Returns (C_out fp32 K x d, counts int32 K)."""
    T = np.asarray(T, dtype=np.float32)
    M = T.shape[0]
    cw = cbs[which]
    K = cw.K
    A = np.zeros((K, d, d))
    b = np.zeros((K, d))
    counts = np.zeros(K, dtype=np.int64)
    for g in range(cw.G_cov):
        Hg = np.asarray(H_blocks[g], dtype=np.float64)
        tau = _group(T, g, d) - _fixed_sum(cbs, g, M, d, skip=(which,))
        code = cw.codes[:, g]
        c = np.bincount(code, minlength=K)
        counts += c
        A += c[:, None, None] * Hg[None]
        np.add.at(b, code, tau @ Hg)            # Hg symmetric: (Hg tau_v) as a row
    C_out = cw.C.astype(np.float64).copy()
    ne = counts > 0
    if ne.any():
        C_out[ne] = np.linalg.solve(A[ne], b[ne][..., None])[..., 0]
    return f32(C_out), counts.astype(np.int32)


# --------------------------------------------------------------------------------------
# Reconstruction, inverse reorder and losses (Alg. 1 QuantLoss; Sec. 4.3 reverse reorder)
# --------------------------------------------------------------------------------------
# NEXT-3: inference product with the quantized matrix (no W_enc formed)
# --------------------------------------------------------------------------------------
def lut_matvec(Xin, perm, cbs, d):
    """Y = Xin W_hat^T for a batch of inputs Xin (b x N, original channel order), with W_hat
    given by its codes: the inputs are permuted once (x_sorted[p] = x[perm[p]]), each codebook
    s and group g get a lookup table T_s,g[k] = <C_s[k], x_sorted,g>, and
    y_i = sum over the covering codebooks and groups of T_s,g[codes_s[i, g]]."""
    Xin = np.atleast_2d(np.asarray(Xin, dtype=np.float64))
    b, N = Xin.shape
    G = N // d
    Xs = Xin[:, np.asarray(perm)] if perm is not None else Xin
    M = cbs[0].codes.shape[0]
    Y = np.zeros((b, M))
    for cb in cbs:
        C = cb.C.astype(np.float64)
        for g in range(cb.G_cov):
            T = Xs[:, g * d:(g + 1) * d] @ C.T          # b x K lookup table
            Y += T[:, cb.codes[:, g]]
    return Y


# --------------------------------------------------------------------------------------
# NEXT-1: Hessian-coupled code search (the full Alg. 1 loss, cross-group terms included)
# --------------------------------------------------------------------------------------
def full_loss(W_sorted, H_sorted, cbs):
    """tr(dW H dW^T) with dW = W_sorted - decode(cbs) and H in the same (sorted) channel order:
    the Alg. 1 loss ||W X - W_enc X||^2 up to the factor n."""
    W = np.asarray(W_sorted, dtype=np.float64)
    dW = W - decode(W.shape[0], W.shape[1], cbs[0].C.shape[1], cbs)
    return float(np.einsum("ij,jk,ik->", dW, np.asarray(H_sorted, np.float64), dW))


def coupled_sweep(W_sorted, d, H_sorted, cbs, which, sweeps=1):
    """Gauss-Seidel over the groups of codebook `which` under the full loss (others fixed).

    The loss separates over rows. For row i and group g, with every other group fixed,
      L = D_g^T H_gg D_g + 2 D_g^T b_g + const,   b_g = sum_{g' != g} H_gg' D_g',
    where D = w_i - w_enc_i. Writing D_g = t_g - c (t_g: the row's segment minus the other
    codebooks' codewords) and completing the square, the best codeword c minimises
      (t_g + H_gg^-1 b_g - c)^T H_gg (t_g + H_gg^-1 b_g - c),
    the block-diagonal score of Sec. 3.1 / Alg. 1 for a shifted target (ties: smaller index).
    Groups are visited in order, each with the others' current codes, so the loss never rises.
    Returns (new codes of `which` (M x G_cov int64), loss after each group step)."""
    W = np.asarray(W_sorted, dtype=np.float64)
    H = np.asarray(H_sorted, dtype=np.float64)
    M, N = W.shape
    cb = cbs[which]
    C = cb.C.astype(np.float64)
    codes = cb.codes.copy()
    cur = [Codebook(c.C, c.codes, c.G_cov) for c in cbs]
    cur[which] = Codebook(cb.C, codes, cb.G_cov)
    D = W - decode(M, N, d, cur)                      # current error, all rows
    history = []
    for _ in range(sweeps):
        for g in range(cb.G_cov):
            sl = slice(g * d, (g + 1) * d)
            Hgg = H[sl, sl]
            b = D @ H[:, sl] - D[:, sl] @ Hgg         # sum over g' != g of D_g' H_g'g (rows)
            t = D[:, sl] + C[codes[:, g]]             # segment minus the other codebooks
            shift = np.linalg.solve(Hgg, b.T).T       # H_gg^-1 b_g (H symmetric)
            err = quad_err(t + shift, C, Hgg)
            k = np.argmin(err, axis=1)                # first minimum: the smaller index
            codes[:, g] = k
            D[:, sl] = t - C[k]
            history.append(float(np.einsum("ij,jk,ik->", D, H, D)))
    return codes, history


# --------------------------------------------------------------------------------------
def decode(M, N, d, cbs):
    """W_enc in the sorted channel order: sum of the covering codebooks' codewords."""
    G = N // d
    out = np.zeros((M, N))
    for g in range(G):
        out[:, g * d:(g + 1) * d] = _fixed_sum(cbs, g, M, d)
    return out


def reconstruct_error(W_sorted, d, H_blocks, perm, cbs, G_c, X=None, delta=0.0):
    """Returns (W_hat fp32 in the original channel order, loss_block, loss_crit, loss_full).

    loss_block = sum_v (t_v - r_v)^T H_g (t_v - r_v) over all vectors (block-diagonal part of
    the Alg. 1 loss); loss_crit = the same over the critical groups g < G_c; loss_full =
    ||(W - W_hat) X^T||^2 / n + delta ||W - W_hat||^2 = tr(dW H dW^T), the Alg. 1 loss with
    the damped H (None when X is None). perm None means the identity."""
    Ws = np.asarray(W_sorted, dtype=np.float64)
    M, N = Ws.shape
    G = N // d
    Wh = decode(M, N, d, cbs)
    D = Ws - Wh
    lb = 0.0
    lc = 0.0
    for g in range(G):
        Dg = D[:, g * d:(g + 1) * d]
        e = float(np.einsum("vd,vd->", Dg @ np.asarray(H_blocks[g], np.float64), Dg))
        lb += e
        if g < G_c:
            lc += e
    perm = np.arange(N) if perm is None else np.asarray(perm)
    W_hat = np.empty((M, N))
    W_hat[:, perm] = Wh
    lf = None
    if X is not None:
        Dorig = np.empty((M, N))
        Dorig[:, perm] = D
        X64 = np.asarray(X, dtype=np.float64)
        P = Dorig @ X64.T
        lf = float((P * P).sum() / X64.shape[0] + float(delta) * (Dorig * Dorig).sum())
    return f32(W_hat), lb, lc, lf


# --------------------------------------------------------------------------------------
# Average bit-width (Sec. 3.2 Eq. (bitwidth); App. A.1)
# --------------------------------------------------------------------------------------
def avg_bits(e, d, m, lam, M=4096, N=4096, include_perm=False, n_base=1):
    """Bits per weight of an M x N matrix with n_base base and m-1 extended codebooks.

    Codes: e bits per vector for each base codebook on all M N / d vectors (Sec. 3.2 Eq.
    (bitwidth) counts m such codebooks), and for each of the m-1 extended codebooks on the
    lambda fraction of critical vectors (App. A.1); codebooks: n_base + m - 1 of 2^e fp16
    vectors of length d; optional 16-bit reorder index per channel (App. A.1)."""
    nvec = M * N / d
    bits = n_base * nvec * e + (m - 1) * lam * nvec * e + (n_base + m - 1) * (2 ** e) * d * 16
    if include_perm:
        bits += 16 * N
    return bits / (M * N)


# --------------------------------------------------------------------------------------
# S1-S7: one weight matrix through Alg. 1, prequantization through the refinement loop
# --------------------------------------------------------------------------------------
PHASE_PREQUANT, PHASE_BASE, PHASE_EXT, PHASE_RANDOM = 1, 2, 3, 4


def phase_seed(seed, phase, cb):
    return splitmix64(seed, phase * 1024 + cb)


def lloyd(T, d, H_blocks, fixed, C0, G_cov, iters, seed_unused=None):
    """T iterations of (encode, LS update) for the last codebook, then a final encode."""
    cbs = list(fixed) + [Codebook(C0, None, G_cov)]
    j = len(cbs) - 1
    objective = []
    for _ in range(iters):
        codes, verr = encode_beam(T, d, H_blocks, cbs, n_fixed=j, B=1)
        cbs[j] = Codebook(cbs[j].C, codes[j], G_cov)
        objective.append(float(verr.astype(np.float64)[:, :G_cov].sum()))
        C, _ = update_codebook(T, d, H_blocks, cbs, j)
        cbs[j] = Codebook(C, codes[j], G_cov)
    codes, verr = encode_beam(T, d, H_blocks, cbs, n_fixed=j, B=1)
    cbs[j] = Codebook(cbs[j].C, codes[j], G_cov)
    objective.append(float(verr.astype(np.float64)[:, :G_cov].sum()))
    return cbs[j], objective


def quantize_layer(W, X, cfg):
    """The whole per-matrix schedule (Alg. 1, prequantization through the refinement loop)
    with the readings above.

    cfg has attributes d, K_base, n_ext, K_ext, crit_frac, B, kmeans_iters, refine_rounds,
    eps_rel, damp_rel, importance_mode, seed, and optionally n_base (base codebooks, default
    1). Returns a dict of every intermediate result; out["codebooks"] lists the n_base base
    codebooks, then the extended ones."""
    d = cfg.d
    W = np.asarray(W, dtype=np.float32)
    M, N = W.shape
    G = N // d
    out = {}
    # S1
    H, xsq, Hb0, delta = hessian(X, cfg.damp_rel, d)
    out.update(H=H, xsq=xsq, H_blocks_orig=Hb0, delta=delta)
    # S2: prequantize in the original order (Alg. 1, prequantization step)
    C0 = kmeans_init(W, d, G, cfg.K_base, phase_seed(cfg.seed, PHASE_PREQUANT, 0))
    pre, _ = lloyd(W, d, Hb0, [], C0, G, cfg.kmeans_iters)
    W_pre, pre_loss, _, _ = reconstruct_error(W, d, Hb0, None, [pre], 0)
    out.update(C_pre=pre.C, codes_pre=pre.codes, W_pre=W_pre, loss_pre=pre_loss)
    # S3 (Alg. 1, importance and reordering steps)
    perm, I, Ws, Hb, Gc = select_reorder_channels(
        W, d, W_pre, xsq, H, cfg.crit_frac, cfg.importance_mode,
        phase_seed(cfg.seed, PHASE_RANDOM, 0))
    out.update(perm=perm, importance=I, W_sorted=Ws, H_blocks=Hb, n_crit_groups=Gc)
    # S4 (Alg. 1, base codebook steps). With several base codebooks (Sec. 6.4, the m = 2
    # setting) base codebook b covers every group and is fitted on the residual of bases
    # 0..b-1, as the extended loop does on the critical groups; cfg.n_base defaults to one.
    cbs = []
    for b in range(getattr(cfg, "n_base", 1)):
        Cb0 = kmeans_init(Ws, d, G, cfg.K_base, phase_seed(cfg.seed, PHASE_BASE, b), cbs)
        base, obj = lloyd(Ws, d, Hb, cbs, Cb0, G, cfg.kmeans_iters)
        if b == 0:
            out["base_objective"] = obj
        cbs.append(base)
    # S5 (Alg. 1, extended-codebook loop): extended codebooks on the critical residual
    crit_losses = [reconstruct_error(Ws, d, Hb, perm, cbs, Gc)[2]]
    Tc = Ws[:, :Gc * d]
    Hbc = Hb[:Gc]
    for t in range(1, cfg.n_ext + 1):
        fixed = [Codebook(cb.C, cb.codes[:, :Gc], Gc) for cb in cbs]
        Ct0 = kmeans_init(Tc, d, Gc, cfg.K_ext, phase_seed(cfg.seed, PHASE_EXT, t), fixed)
        ext, _ = lloyd(Tc, d, Hbc, fixed, Ct0, Gc, cfg.kmeans_iters)
        cbs.append(Codebook(ext.C, ext.codes, Gc))
        crit_losses.append(reconstruct_error(Ws, d, Hb, perm, cbs, Gc)[2])
    out["crit_loss_after_ext"] = crit_losses
    # S6 (Alg. 1, refinement loop): LS codebook updates + joint beam re-encode
    _, lb, _, _ = reconstruct_error(Ws, d, Hb, perm, cbs, Gc)
    history = [lb]
    for _ in range(cfg.refine_rounds):
        for j in range(len(cbs)):
            C, _ = update_codebook(Ws, d, Hb, cbs, j)
            cbs[j] = Codebook(C, cbs[j].codes, cbs[j].G_cov)
        codes, _ = encode_beam(Ws, d, Hb, cbs, n_fixed=0, B=cfg.B, keep_if_better=True)
        cbs = [Codebook(cb.C, codes[s], cb.G_cov) for s, cb in enumerate(cbs)]
        _, lb, _, _ = reconstruct_error(Ws, d, Hb, perm, cbs, Gc)
        history.append(lb)
        if lb > (1.0 - cfg.eps_rel) * history[-2]:
            break
    out["loss_history"] = history
    # S7
    W_hat, lb, lc, lf = reconstruct_error(Ws, d, Hb, perm, cbs, Gc, X, float(delta))
    out.update(codebooks=cbs, W_hat=W_hat, loss_block=lb, loss_crit=lc, loss_full=lf)
    return out
