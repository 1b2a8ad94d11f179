"""GPU-vs-oracle parity of every C-ABI entry point, called through the ctypes binding on
seeded synthetic inputs. Stepwise: each call gets byte-identical inputs on both sides.

Bars: code indices and permutations bit-exact except fp64 near-ties (relative margin below
1e-6 of err_best + t^T H t, or importance gaps below 1e-6 of max I); codebooks within 1e-4 of
the codebook's max |value|; losses within 1e-4 relative; H within 2e-5 * sqrt(H_aa H_bb)
(3xTF32 tensor-core products accumulated in fp32 over chunks of at most 1024 tokens, chunks
summed in fp32 in chunk order: about 1e-6 typical, under 1e-5 including the accumulator's
rounding bias); reconstructions bit-exact (fp64 sums of fp32 codewords rounded once on both
sides).
"""
import numpy as np
import pytest
import torch

import synthetic as S
from oracle import crvq_oracle as O
from parity_util import (beam_boundary_gap, check_codes_with_ties, dev, host, oracle_cbs)

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook
    from paper_2412_09282_gb300 import build as _build
    _build.build()

D = 8


@pytest.fixture(scope="module")
def c1():
    cfg = S.C1
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    H, xsq, Hb0, delta = O.hessian(X, cfg.damp_rel, D)
    return dict(cfg=cfg, W=W, X=X, H=H, xsq=xsq, Hb0=Hb0, delta=delta)


def _sync():
    P.crvq_sync()


def _cmp_codebook(Cg, Co, tol=1e-4):
    err = np.abs(Cg.astype(np.float64) - Co).max() / max(np.abs(Co).max(), 1e-30)
    assert err <= tol, f"codebook rel err {err}"


# ------------------------------------------------------------------------------ S1 Hessian
@pytest.mark.parametrize("n,N", [(1024, 512), (77, 136), (300, 8), (5, 264), (2500, 264)])
def test_hessian_parity(n, N):
    cfg = S.C1.with_(name=f"hess_{n}_{N}", n_tok=n, N=N)
    X = S.gen_X(cfg)
    H, xsq, Hb, delta = P.crvq_hessian(dev(X), cfg.damp_rel, D)
    _sync()
    Ho, xo, Hbo, do = O.hessian(X, cfg.damp_rel, D)
    Hg = host(H)
    scale = np.sqrt(np.outer(np.diag(Ho), np.diag(Ho)))
    assert np.all(np.abs(Hg - Ho) <= 2e-5 * scale + 1e-30)
    np.testing.assert_allclose(host(xsq), xo, rtol=2e-5)
    assert abs(float(host(delta)[0]) - float(do)) <= 2e-5 * abs(float(do))
    np.testing.assert_array_equal(host(Hb), np.stack(
        [Hg[g * D:(g + 1) * D, g * D:(g + 1) * D] for g in range(N // D)]))
    assert np.array_equal(Hg, Hg.T)


@pytest.mark.parametrize("n,N", [(1024, 512), (77, 136), (300, 8), (2500, 264), (4096, 1032)])
def test_hessian_blocks_equal_dense_blocks(n, N):
    """The blocks-only path (no N x N matrix) returns the dense H's diagonal blocks bit for bit,
    in the stored order and through a channel permutation (1, 3 and 4 token chunks; a ragged
    last 128-channel tile), with the same xsq and delta."""
    cfg = S.C1.with_(name=f"hessb_{n}_{N}", n_tok=n, N=N)
    X = S.gen_X(cfg)
    Xd = dev(X)
    H, xsq, Hb, delta = P.crvq_hessian(Xd, cfg.damp_rel, D)
    Hb2, xsq2, delta2 = P.crvq_hessian_blocks(Xd, cfg.damp_rel, D)
    perm = np.random.default_rng(n + N).permutation(N).astype(np.int32)
    Hb3, xsq3, delta3 = P.crvq_hessian_blocks(Xd, cfg.damp_rel, D, perm=dev(perm))
    _sync()
    Hg = host(H)
    np.testing.assert_array_equal(host(Hb2), host(Hb))
    for a in (xsq2, xsq3):
        np.testing.assert_array_equal(host(a), host(xsq))
    for a in (delta2, delta3):
        np.testing.assert_array_equal(host(a), host(delta))
    want = np.stack([Hg[np.ix_(perm[g * D:(g + 1) * D], perm[g * D:(g + 1) * D])]
                     for g in range(N // D)])
    np.testing.assert_array_equal(host(Hb3), want)


def test_hessian_blocks_reports_out_of_range_channel():
    cfg = S.C1.with_(name="hessb_bad", n_tok=64, N=64)
    X = dev(S.gen_X(cfg))
    perm = np.arange(64, dtype=np.int32)
    perm[5] = 64
    P.crvq_hessian_blocks(X, cfg.damp_rel, D, perm=dev(perm))
    with pytest.raises(P.CrvqError):
        P.crvq_sync()
    P.crvq_hessian_blocks(X, cfg.damp_rel, D)   # the context is still usable
    P.crvq_sync()


# ------------------------------------------------------------------------------ S3 reorder
@pytest.mark.parametrize("mode", [0, 1, 2])
def test_select_reorder_parity(c1, mode):
    W, H, xsq = c1["W"], c1["H"], c1["xsq"]
    W_pre = (np.round(W * 40) / 40).astype(np.float32)
    perm, imp, Ws, Hb, gc = P.crvq_select_reorder_channels(dev(W), D, dev(W_pre), dev(xsq),
                                                           dev(H), 0.02, mode, seed=1234)
    _sync()
    po, io, Wso, Hbo, gco = O.select_reorder_channels(W, D, W_pre, xsq, H, 0.02, mode, 1234)
    assert gc == gco
    pg = host(perm)
    I64 = O.importance(W, W_pre, xsq, mode, 1234)
    np.testing.assert_allclose(host(imp), io, rtol=1e-6)
    diff = np.nonzero(pg != po)[0]
    for p in diff:  # only near-ties may swap
        assert abs(I64[pg[p]] - I64[po[p]]) <= 1e-6 * I64.max()
    assert sorted(pg.tolist()) == list(range(W.shape[1]))
    np.testing.assert_array_equal(host(Ws), W[:, pg])
    Hp = H[np.ix_(pg, pg)]
    np.testing.assert_array_equal(host(Hb), np.stack(
        [Hp[g * D:(g + 1) * D, g * D:(g + 1) * D] for g in range(W.shape[1] // D)]))


# ------------------------------------------------------------------------------ k-means init
def test_kmeans_init_parity(c1):
    W = c1["W"]
    M, N = W.shape
    G = N // D
    Cg = P.crvq_kmeans_init(dev(W), D, G, 256, seed=99)
    _sync()
    np.testing.assert_array_equal(host(Cg), O.kmeans_init(W, D, G, 256, 99))
    # residual init on a 3-group critical slice with a fixed base codebook (bit-exact: fp64
    # residual rounded once on both sides)
    rng = np.random.default_rng(0)
    Cb = (0.02 * rng.standard_normal((256, D))).astype(np.float32)
    codes = rng.integers(0, 256, (M, G)).astype(np.int32)
    Wd = dev(W)
    codes_d = dev(codes)
    fixed = [Codebook(dev(Cb), codes_d[:, :3], 3)]
    Cr = P.crvq_kmeans_init(Wd[:, :3 * D], D, 3, 100, seed=7, fixed=fixed)
    _sync()
    Co = O.kmeans_init(W[:, :3 * D], D, 3, 100, 7, [O.Codebook(Cb, codes[:, :3], 3)])
    np.testing.assert_array_equal(host(Cr), Co)
    # K equal to the number of vectors takes every vector once
    Ca = P.crvq_kmeans_init(Wd[:2, :2 * D], D, 2, 4, seed=3)
    _sync()
    np.testing.assert_array_equal(host(Ca), np.stack([W[0, :8], W[0, 8:16], W[1, :8],
                                                      W[1, 8:16]]))


# ------------------------------------------------------------------------------ encode
def _codebook_for(W, G, K, seed, scale=1.0):
    C = O.kmeans_init(W, D, G, K, seed)
    return (C * np.float32(scale)).astype(np.float32)


@pytest.mark.parametrize("M,K", [(512, 256), (77, 1500), (513, 1), (1, 300), (600, 4100)])
def test_encode_argmin_parity(c1, M, K):
    W = c1["W"][:M] if M <= 512 else np.concatenate([c1["W"], c1["W"][:M - 512] * 1.5])
    W = np.ascontiguousarray(W, dtype=np.float32)
    G = W.shape[1] // D
    Hb = c1["Hb0"]
    C = _codebook_for(W, G, min(K, W.shape[0] * G), 5)
    if C.shape[0] < K:
        C = np.concatenate([C, C[:K - C.shape[0]] * 1.01]).astype(np.float32)
    codes = torch.zeros((W.shape[0], G), dtype=torch.int32, device="cuda")
    cbs = [Codebook(dev(C), codes, G)]
    verr = P.crvq_encode_beam(dev(W), D, dev(Hb), cbs, 0, 1, want_err=True)
    _sync()
    oc, oerr = O.encode_beam(W, D, Hb, [O.Codebook(C, None, G)], 0, 1)
    check_codes_with_ties(W, D, Hb, [O.Codebook(C, None, G)], 0, [host(codes)], oc)
    np.testing.assert_allclose(host(verr), oerr, rtol=1e-5, atol=1e-12)


def test_encode_argmin_exact_duplicate_codewords_tie_to_smaller_index(c1):
    W = c1["W"][:64]
    G = W.shape[1] // D
    C = _codebook_for(W, G, 16, 3)
    C = np.concatenate([C, C]).astype(np.float32)       # every codeword twice
    codes = torch.zeros((64, G), dtype=torch.int32, device="cuda")
    P.crvq_encode_beam(dev(W), D, dev(c1["Hb0"]), [Codebook(dev(C), codes, G)], 0, 1)
    _sync()
    oc, _ = O.encode_beam(W, D, c1["Hb0"], [O.Codebook(C, None, G)], 0, 1)
    np.testing.assert_array_equal(host(codes), oc[0])
    assert host(codes).max() < 16


def test_encode_fixed_codebooks_on_critical_slice(c1):
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G, Gc = N // D, 5
    rng = np.random.default_rng(1)
    Cb = _codebook_for(W, G, 256, 11)
    cb_codes = rng.integers(0, 256, (M, G)).astype(np.int32)
    Ce = (0.3 * _codebook_for(W, G, 64, 12)).astype(np.float32)
    Wd = dev(W)
    base_codes = dev(cb_codes)
    ext_codes = torch.zeros((M, Gc), dtype=torch.int32, device="cuda")
    cbs = [Codebook(dev(Cb), base_codes[:, :Gc], Gc), Codebook(dev(Ce), ext_codes, Gc)]
    verr = P.crvq_encode_beam(Wd[:, :Gc * D], D, dev(Hb[:Gc]), cbs, 1, 1, want_err=True)
    _sync()
    ocbs = [O.Codebook(Cb, cb_codes[:, :Gc], Gc), O.Codebook(Ce, None, Gc)]
    oc, oerr = O.encode_beam(W[:, :Gc * D], D, Hb[:Gc], ocbs, 1, 1)
    check_codes_with_ties(W[:, :Gc * D], D, Hb[:Gc], ocbs, 1, [None, host(ext_codes)], oc)
    np.testing.assert_allclose(host(verr), oerr, rtol=1e-5)


@pytest.mark.parametrize("B", [1, 2, 4, 8, 16])
def test_encode_beam_parity_mixed_coverage(c1, B):
    """Full set: base covers every group, two extended codebooks cover the first Gc groups;
    critical vectors get the 3-stage beam, the others the base arg-min, in one call."""
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G, Gc = N // D, 4
    Cb = _codebook_for(W, G, 256, 21)
    rng = np.random.default_rng(2)
    Ce1 = (0.4 * _codebook_for(W, G, 64, 22)).astype(np.float32)
    Ce2 = (0.15 * _codebook_for(W, G, 32, 23)).astype(np.float32)
    codes = [torch.zeros((M, G), dtype=torch.int32, device="cuda"),
             torch.zeros((M, Gc), dtype=torch.int32, device="cuda"),
             torch.zeros((M, Gc), dtype=torch.int32, device="cuda")]
    cbs = [Codebook(dev(Cb), codes[0], G), Codebook(dev(Ce1), codes[1], Gc),
           Codebook(dev(Ce2), codes[2], Gc)]
    verr = P.crvq_encode_beam(dev(W), D, dev(Hb), cbs, 0, B, want_err=True)
    _sync()
    ocbs = [O.Codebook(Cb, None, G), O.Codebook(Ce1, None, Gc), O.Codebook(Ce2, None, Gc)]
    oc, oerr = O.encode_beam(W, D, Hb, ocbs, 0, B)
    gpu = [host(c) for c in codes]
    # mismatching critical vectors must come from a near-tie inside the oracle's beam
    diff = np.zeros((M, G), bool)
    for s in range(3):
        diff[:, :cbs[s].G_cov] |= gpu[s] != oc[s]
    for i, g in zip(*np.nonzero(diff)):
        Cs = [Cb] + ([Ce1, Ce2] if g < Gc else [])
        gap = beam_boundary_gap(W[i, g * D:(g + 1) * D].astype(np.float64), Hb[g], Cs, B)
        assert gap < 1e-6, f"vector ({i},{g}) differs with beam gap {gap}"
    np.testing.assert_allclose(host(verr)[~diff], oerr[~diff], rtol=1e-5)


def test_encode_keep_if_better(c1):
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G, Gc = N // D, 3
    Cb = _codebook_for(W, G, 128, 31)
    Ce = (0.3 * _codebook_for(W, G, 16, 32)).astype(np.float32)
    ocbs = [O.Codebook(Cb, None, G), O.Codebook(Ce, None, Gc)]
    best, _ = O.encode_beam(W, D, Hb, ocbs, 0, 16)      # a (near) optimal tuple
    # start from the optimal tuple: a width-1 beam must keep it wherever it is better
    codes = [dev(best[0]), dev(best[1])]
    cbs = [Codebook(dev(Cb), codes[0], G), Codebook(dev(Ce), codes[1], Gc)]
    P.crvq_encode_beam(dev(W), D, dev(Hb), cbs, 0, 1, keep_if_better=True)
    _sync()
    oc, _ = O.encode_beam(W, D, Hb, [O.Codebook(Cb, best[0], G), O.Codebook(Ce, best[1], Gc)],
                          0, 1, keep_if_better=True)
    check_codes_with_ties(W, D, Hb, [O.Codebook(Cb, best[0], G), O.Codebook(Ce, best[1], Gc)],
                          0, [host(c) for c in codes], oc)


# ------------------------------------------------------------------------------ update
@pytest.mark.parametrize("which", [0, 1])
def test_update_codebook_parity(c1, which):
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G, Gc = N // D, 6
    rng = np.random.default_rng(3 + which)
    Cb = _codebook_for(W, G, 256, 41)
    Ce = (0.3 * _codebook_for(W, G, 64, 42)).astype(np.float32)
    cb_codes = rng.integers(0, 250, (M, G)).astype(np.int32)    # 250..255 stay empty
    ce_codes = rng.integers(0, 60, (M, Gc)).astype(np.int32)    # 60..63 stay empty
    cbs = [Codebook(dev(Cb), dev(cb_codes), G), Codebook(dev(Ce), dev(ce_codes), Gc)]
    Cg, cnt = P.crvq_update_codebook(dev(W), D, dev(Hb), cbs, which)
    _sync()
    ocbs = [O.Codebook(Cb, cb_codes, G), O.Codebook(Ce, ce_codes, Gc)]
    Co, co = O.update_codebook(W, D, Hb, ocbs, which)
    np.testing.assert_array_equal(host(cnt), co)
    _cmp_codebook(host(Cg), Co.astype(np.float64))
    empty = co == 0
    np.testing.assert_array_equal(host(Cg)[empty], (Cb if which == 0 else Ce)[empty])


def test_update_codebook_in_place_and_large_K(c1):
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G = N // D
    rng = np.random.default_rng(5)
    K = 4096                                            # two radix passes
    C = _codebook_for(W, G, K, 51)
    codes = rng.integers(0, K, (M, G)).astype(np.int32)
    Cd = dev(C)
    cbs = [Codebook(Cd, dev(codes), G)]
    P.crvq_update_codebook(dev(W), D, dev(Hb), cbs, 0, C_out=Cd)
    _sync()
    Co, _ = O.update_codebook(W, D, Hb, [O.Codebook(C, codes, G)], 0)
    _cmp_codebook(host(Cd), Co.astype(np.float64))


def test_update_is_deterministic(c1):
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G = N // D
    rng = np.random.default_rng(6)
    C = _codebook_for(W, G, 256, 61)
    codes = dev(rng.integers(0, 256, (M, G)).astype(np.int32))
    cbs = [Codebook(dev(C), codes, G)]
    a, _ = P.crvq_update_codebook(dev(W), D, dev(Hb), cbs, 0)
    b, _ = P.crvq_update_codebook(dev(W), D, dev(Hb), cbs, 0)
    _sync()
    assert torch.equal(a, b)


# ------------------------------------------------------------------------------ S7 losses
@pytest.mark.parametrize("shape", ["c1", "wide", "ragged"])
def test_reconstruct_error_parity(c1, shape):
    if shape == "c1":
        W, X, H, delta = c1["W"], c1["X"], c1["H"], float(c1["delta"])
    else:
        # wide: N = 2056 channels, the full-loss product over three K chunks; ragged: M = 203
        # rows (not a multiple of the decode's 4 rows per warp), G = 33 groups (a ragged last
        # group slice), n_tok = 77
        M_, N_, n_ = (200, 2056, 300) if shape == "wide" else (203, 264, 77)
        cfg = S.C1.with_(name=f"recon_{shape}", M=M_, N=N_, n_tok=n_)
        W, X = S.gen_W(cfg), S.gen_X(cfg)
        H, _, _, delta = O.hessian(X, cfg.damp_rel, D)
        delta = float(delta)
    M, N = W.shape
    G, Gc = N // D, 2
    rng = np.random.default_rng(7)
    perm = rng.permutation(N).astype(np.int32)
    Ws = np.ascontiguousarray(W[:, perm])
    Hb = np.stack([H[np.ix_(perm[g * D:g * D + D], perm[g * D:g * D + D])] for g in range(G)])
    Cb = _codebook_for(Ws, G, 256, 71)
    Ce = (0.3 * _codebook_for(Ws, G, 32, 72)).astype(np.float32)
    cbc = rng.integers(0, 256, (M, G)).astype(np.int32)
    cec = rng.integers(0, 32, (M, Gc)).astype(np.int32)
    cbs = [Codebook(dev(Cb), dev(cbc), G), Codebook(dev(Ce), dev(cec), Gc)]
    Wh, lb, lc, lf = P.crvq_reconstruct_error(dev(Ws), D, dev(Hb), dev(perm), cbs, Gc,
                                              X=dev(X), damp_delta=delta)
    ocbs = [O.Codebook(Cb, cbc, G), O.Codebook(Ce, cec, Gc)]
    Who, lbo, lco, lfo = O.reconstruct_error(Ws, D, Hb, perm, ocbs, Gc, X, delta)
    np.testing.assert_array_equal(host(Wh), Who)
    assert abs(lb - lbo) <= 1e-4 * lbo
    assert abs(lc - lco) <= 1e-4 * lco
    # the full loss: 3xTF32 products, fp32 accumulation in chunks of 1024 channels summed in
    # order, fp32 sums of squares per row: a few 1e-6 relative
    assert abs(lf - lfo) <= 2e-5 * lfo
    # identity order, no X
    Wh2, lb2, _, lf2 = P.crvq_reconstruct_error(dev(Ws), D, dev(Hb), None, cbs, Gc)
    assert lf2 is None
    np.testing.assert_array_equal(host(Wh2), O.reconstruct_error(Ws, D, Hb, None, ocbs, Gc)[0])
    # identity order with X's columns taken in the sorted order beforehand: the same full loss
    # (the channel sum of the loss product in another order)
    Xs = np.ascontiguousarray(X[:, perm])
    _, lb3, lc3, lf3 = P.crvq_reconstruct_error(dev(Ws), D, dev(Hb), None, cbs, Gc, X=dev(Xs),
                                                damp_delta=delta)
    assert lb3 == lb and lc3 == lc
    assert abs(lf3 - lfo) <= 2e-5 * lfo


# ------------------------------------------------------------------------------ errors
def test_device_index_check_reports_and_recovers(c1):
    W, Hb = c1["W"], c1["Hb0"]
    M, N = W.shape
    G = N // D
    C = _codebook_for(W, G, 16, 81)
    bad = np.zeros((M, G), np.int32)
    bad[3, 4] = 999                                      # out of range: skipped, reported
    with pytest.raises(P.CrvqError) as e:
        P.crvq_update_codebook(dev(W), D, dev(Hb), [Codebook(dev(C), dev(bad), G)], 0)
        P.crvq_sync()
    assert e.value.status == -7
    P.crvq_sync()                                        # the word was cleared
    good = dev(np.zeros((M, G), np.int32))
    P.crvq_encode_beam(dev(W), D, dev(Hb), [Codebook(dev(C), good, G)], 0, 1)
    P.crvq_sync()


@pytest.mark.parametrize("where", ["T", "other_codebook", "H"])
def test_update_reports_a_nan_in_its_inputs(c1, where):
    """A NaN in the targets, in a fixed codebook or in an H block makes the fixed-point scale
    bound non-finite (the maxima keep NaN), and the next crvq_sync reports CRVQ_ERR_NUMERIC
    instead of returning a codebook built from INT_MIN terms with status OK."""
    W, Hb = c1["W"].copy(), c1["Hb0"].copy()
    M, N = W.shape
    G, Gc = N // D, 4
    rng = np.random.default_rng(91)
    Cb = _codebook_for(W, G, 64, 92)
    Ce = (0.3 * _codebook_for(W, G, 16, 93)).astype(np.float32)
    if where == "T":
        W[7, 13] = np.nan
    elif where == "other_codebook":
        Ce[3, 5] = np.nan
    else:
        Hb[2, 4, 4] = np.nan
    cbs = [Codebook(dev(Cb), dev(rng.integers(0, 64, (M, G)).astype(np.int32)), G),
           Codebook(dev(Ce), dev(rng.integers(0, 16, (M, Gc)).astype(np.int32)), Gc)]
    P.crvq_sync()
    with pytest.raises(P.CrvqError) as e:
        P.crvq_update_codebook(dev(W), D, dev(Hb), cbs, 0)
        P.crvq_sync()
    assert e.value.status == -6
    P.crvq_sync()                                        # the word was cleared


def test_invalid_arguments_raise_before_launch(c1):
    W = dev(c1["W"])
    with pytest.raises(P.CrvqError) as e:
        P.crvq_kmeans_init(W[:1, :8], D, 1, 2, seed=0)   # K > #vectors
    assert e.value.status == -1
    with pytest.raises(P.CrvqError) as e:
        P.crvq_hessian(dev(c1["X"]), 0.01, d=16)
    assert e.value.status == -2


# ------------------------------------------------------------------------------ end to end
def _gpu_schedule_with_checks(W, X, cfg):
    """The per-matrix schedule driven call by call through the C ABI, each step checked
    against the oracle fed the GPU's own state (stepwise re-synced parity along the GPU's
    trajectory). Returns the GPU state at the end."""
    d = cfg.d
    M, N = W.shape
    G = N // d
    seed = lambda ph, cb: O.phase_seed(cfg.seed, ph, cb)
    Xd, Wd = dev(X), dev(W)
    H, xsq, Hb0, delta = P.crvq_hessian(Xd, cfg.damp_rel, d)

    def lloyd(T, Hb, fixed, C0, G_cov, Td_np, Hb_np):
        codes = torch.zeros((M, G_cov), dtype=torch.int32, device="cuda")
        cbs = list(fixed) + [Codebook(C0, codes, G_cov)]
        j = len(cbs) - 1
        for it in range(cfg.kmeans_iters + 1):
            P.crvq_encode_beam(T, d, Hb, cbs, j, 1)
            P.crvq_sync()
            ocb = oracle_cbs(cbs)
            oc, _ = O.encode_beam(Td_np, d, Hb_np, [c for c in ocb[:j]] +
                                  [O.Codebook(ocb[j].C, None, G_cov)], j, 1)
            check_codes_with_ties(Td_np, d, Hb_np, ocb[:j] + [O.Codebook(ocb[j].C, None, G_cov)],
                                  j, [None] * j + [host(codes)], oc)
            if it == cfg.kmeans_iters:
                break
            Cn, _ = P.crvq_update_codebook(T, d, Hb, cbs, j)
            P.crvq_sync()
            Co, _ = O.update_codebook(Td_np, d, Hb_np, oracle_cbs(cbs), j)
            _cmp_codebook(host(Cn), Co.astype(np.float64))
            cbs[j] = Codebook(Cn, codes, G_cov)
        return cbs[j]

    # S2 prequantize
    C0 = P.crvq_kmeans_init(Wd, d, G, cfg.K_base, seed(1, 0))
    pre = lloyd(Wd, Hb0, [], C0, G, W, host(Hb0))
    W_pre, _, _, _ = P.crvq_reconstruct_error(Wd, d, Hb0, None, [pre], 0)
    # S3
    perm, imp, Ws, Hb, Gc = P.crvq_select_reorder_channels(
        Wd, d, W_pre, xsq, H, cfg.crit_frac, cfg.importance_mode, seed(4, 0))
    P.crvq_sync()
    po = O.select_reorder_channels(W, d, host(W_pre), host(xsq), host(H), cfg.crit_frac,
                                   cfg.importance_mode, seed(4, 0))
    np.testing.assert_array_equal(host(perm), po[0])
    Ws_np, Hb_np = host(Ws), host(Hb)
    # S4: base codebook b on the residual of bases 0..b-1 over every group
    cbs = []
    for b in range(getattr(cfg, "n_base", 1)):
        Cb0 = P.crvq_kmeans_init(Ws, d, G, cfg.K_base, seed(2, b), fixed=list(cbs))
        cbs.append(lloyd(Ws, Hb, list(cbs), Cb0, G, Ws_np, Hb_np))
    # S5
    crit = Ws[:, :Gc * d]
    for t in range(1, cfg.n_ext + 1):
        fixed = [Codebook(cb.C, cb.codes[:, :Gc], Gc) for cb in cbs]
        Ct0 = P.crvq_kmeans_init(crit, d, Gc, cfg.K_ext, seed(3, t), fixed=fixed)
        ext = lloyd(crit, Hb[:Gc], fixed, Ct0, Gc, Ws_np[:, :Gc * d], Hb_np[:Gc])
        cbs.append(Codebook(ext.C, ext.codes, Gc))
    # S6 (one round)
    for r in range(cfg.refine_rounds):
        for j in range(len(cbs)):
            Cn, _ = P.crvq_update_codebook(Ws, d, Hb, cbs, j)
            P.crvq_sync()
            Co, _ = O.update_codebook(Ws_np, d, Hb_np, oracle_cbs(cbs), j)
            _cmp_codebook(host(Cn), Co.astype(np.float64))
            cbs[j] = Codebook(Cn, cbs[j].codes, cbs[j].G_cov)
        before = oracle_cbs(cbs)
        P.crvq_encode_beam(Ws, d, Hb, cbs, 0, cfg.B, keep_if_better=True)
        P.crvq_sync()
        oc, _ = O.encode_beam(Ws_np, d, Hb_np, before, 0, cfg.B, keep_if_better=True)
        gpu = [host(cb.codes) for cb in cbs]
        diff = np.zeros((M, G), bool)
        for s in range(len(cbs)):
            diff[:, :cbs[s].G_cov] |= gpu[s] != oc[s]
        for i, g in zip(*np.nonzero(diff)):
            Cs = [cb.C for cb in before if g < cb.G_cov]
            gap = beam_boundary_gap(Ws_np[i, g * d:(g + 1) * d].astype(np.float64), Hb_np[g],
                                    Cs, cfg.B)
            assert gap < 1e-6, f"refinement code differs at ({i},{g}) with gap {gap}"
    Wh, lb, lc, lf = P.crvq_reconstruct_error(Ws, d, Hb, perm, cbs, Gc, X=Xd,
                                              damp_delta=float(host(delta)[0]))
    ocb = oracle_cbs(cbs)
    _, lbo, lco, lfo = O.reconstruct_error(Ws_np, d, Hb_np, host(perm), ocb, Gc, X,
                                           float(host(delta)[0]))
    assert abs(lb - lbo) <= 1e-4 * lbo and abs(lc - lco) <= 1e-4 * lco
    assert abs(lf - lfo) <= 1e-4 * lfo
    return dict(perm=host(perm), cbs=[(host(cb.C), host(cb.codes)) for cb in cbs],
                losses=(lb, lc, lf))


@pytest.mark.parametrize("name", ["c1", "small_B8_3ext", "two_base_2ext"])
def test_quantize_layer_matches_resynced_stepwise_schedule(c1, name):
    """Every step of the schedule agrees with the oracle given the GPU's state, and the
    one-call crvq_quantize_layer reproduces that trajectory exactly (same kernels, same
    order; the fused Lloyd statistics equal the standalone update's, bit for bit). The
    two-base case has two base codebooks over every group (Sec. 6.4's m = 2 setting)."""
    if name == "c1":
        cfg, W, X = c1["cfg"], c1["W"], c1["X"]
    else:
        cfg = S.LayerConfig("pin_med", 256, 192, 300, "outlier_cols", "lognormal", 0.5,
                            n_outlier_cols=5, K_base=128, n_ext=3, K_ext=32, crit_frac=0.1,
                            B=8, kmeans_iters=5)
        if name == "two_base_2ext":
            cfg = cfg.with_(n_base=2, K_base=64, n_ext=2, B=4, kmeans_iters=3)
        W, X = S.gen_W(cfg), S.gen_X(cfg)
    ref = _gpu_schedule_with_checks(W, X, cfg)
    out = P.crvq_quantize_layer(dev(W), dev(X), cfg)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(out.perm), ref["perm"])
    nb = cfg.n_base
    C_base = host(out.C_base).reshape(nb, cfg.K_base, cfg.d)
    codes_base = host(out.codes_base).reshape(nb, *ref["cbs"][0][1].shape)
    for b in range(nb):
        np.testing.assert_array_equal(C_base[b], ref["cbs"][b][0])
        np.testing.assert_array_equal(codes_base[b], ref["cbs"][b][1])
    for t in range(cfg.n_ext):
        np.testing.assert_array_equal(host(out.C_ext[t]), ref["cbs"][nb + t][0])
        np.testing.assert_array_equal(host(out.codes_ext[t]), ref["cbs"][nb + t][1])
    lb, lc, lf = ref["losses"]
    assert out.report["loss_block"] == pytest.approx(lb, rel=1e-12)
    assert out.report["loss_full"] == pytest.approx(lf, rel=1e-12)


def test_quantize_layer_c1_independent_oracle_run(c1):
    """The one-call layer against an independent oracle run of the whole schedule. When the
    two trajectories take the same decisions (every final code equal), codebooks and losses
    agree to 1e-4 relative. If they part, the parting decision must be an exempted fp64
    near-tie: the stepwise run along the GPU's trajectory then checks every step against the
    oracle given the GPU's state, and the one-call layer must reproduce that trajectory."""
    cfg = c1["cfg"]
    W, X = c1["W"], c1["X"]
    out = P.crvq_quantize_layer(dev(W), dev(X), cfg)
    torch.cuda.synchronize()
    ref = O.quantize_layer(W, X, cfg)
    np.testing.assert_array_equal(host(out.perm), ref["perm"])
    cbs = ref["codebooks"]
    gpu_codes = [host(out.codes_base)] + [host(out.codes_ext[t]) for t in range(cfg.n_ext)]
    if all(np.array_equal(g, cb.codes) for g, cb in zip(gpu_codes, cbs)):
        _cmp_codebook(host(out.C_base), cbs[0].C.astype(np.float64))
        for t in range(cfg.n_ext):
            _cmp_codebook(host(out.C_ext[t]), cbs[t + 1].C.astype(np.float64))
        for key in ("loss_block", "loss_crit", "loss_full", "loss_pre"):
            assert abs(out.report[key] - ref[key]) <= 1e-4 * abs(ref[key]), key
    else:
        stepwise = _gpu_schedule_with_checks(W, X, cfg)
        np.testing.assert_array_equal(host(out.codes_base), stepwise["cbs"][0][1])
        np.testing.assert_array_equal(host(out.C_base), stepwise["cbs"][0][0])


def test_quantize_layer_host_buffers_match_device(c1):
    cfg = c1["cfg"].with_(kmeans_iters=3)
    a = P.crvq_quantize_layer(dev(c1["W"]), dev(c1["X"]), cfg)
    torch.cuda.synchronize()
    Wh = torch.from_numpy(c1["W"]).pin_memory()
    Xh = torch.from_numpy(c1["X"]).pin_memory()
    b = P.crvq_quantize_layer(Wh, Xh, cfg)
    assert b.perm.device.type == "cpu"
    np.testing.assert_array_equal(host(a.perm), b.perm.numpy())
    np.testing.assert_array_equal(host(a.codes_base), b.codes_base.numpy())
    np.testing.assert_array_equal(host(a.C_ext), b.C_ext.numpy())
    assert a.report["loss_full"] == b.report["loss_full"]


def test_quantize_layer_two_base_codebooks_host_direct_and_graph_agree(c1, monkeypatch):
    """Two base codebooks: the graph replay on device buffers, the staged host-buffer call and
    the direct (uncaptured) run give the same outputs bit for bit, and each base codebook's
    codes stay in range with every group covered."""
    cfg = c1["cfg"].with_(kmeans_iters=2, n_base=2, K_base=64)
    a = P.crvq_quantize_layer(dev(c1["W"]), dev(c1["X"]), cfg)
    torch.cuda.synchronize()
    Wh = torch.from_numpy(c1["W"]).pin_memory()
    Xh = torch.from_numpy(c1["X"]).pin_memory()
    b = P.crvq_quantize_layer(Wh, Xh, cfg)
    monkeypatch.setenv("CRVQ_GRAPHS", "0")
    c = P.crvq_quantize_layer(dev(c1["W"]), dev(c1["X"]), cfg)
    torch.cuda.synchronize()
    M, N = c1["W"].shape
    assert tuple(a.C_base.shape) == (2, 64, cfg.d)
    assert tuple(a.codes_base.shape) == (2, M, N // cfg.d)
    codes = host(a.codes_base)
    assert codes.min() >= 0 and codes.max() < 64
    for k in ("perm", "C_base", "codes_base", "C_ext", "codes_ext", "W_hat"):
        ref = host(getattr(a, k))
        np.testing.assert_array_equal(ref, getattr(b, k).numpy(), err_msg=k)
        np.testing.assert_array_equal(ref, host(getattr(c, k)), err_msg=k)
    for k in ("loss_block", "loss_crit", "loss_full", "loss_pre"):
        assert a.report[k] == b.report[k] == c.report[k], k


def test_quantize_layer_graph_replay_matches_direct_run(c1, monkeypatch):
    """With device buffers the layer is captured into a CUDA graph on the first call and
    replayed on later ones: a replay equals the direct (uncaptured) run bit for bit, also after
    the contents of W change in place, and counts the same launches."""
    cfg = c1["cfg"].with_(kmeans_iters=3)
    W = dev(c1["W"])
    X = dev(c1["X"])
    first = P.crvq_quantize_layer(W, X, cfg)                     # captured
    n0 = P.crvq_launch_count()
    again = P.crvq_quantize_layer(W, X, cfg, out=first)          # replayed
    torch.cuda.synchronize()
    n_graph = P.crvq_launch_count() - n0
    W.mul_(1.5)                                                  # same pointer, new values
    replay = P.crvq_quantize_layer(W, X, cfg, out=again)
    torch.cuda.synchronize()
    got = {k: host(getattr(replay, k)).copy() for k in ("perm", "C_base", "codes_base",
                                                          "C_ext", "codes_ext", "W_hat")}
    rep = dict(replay.report)
    monkeypatch.setenv("CRVQ_GRAPHS", "0")
    n1 = P.crvq_launch_count()
    direct = P.crvq_quantize_layer(W, X, cfg)
    torch.cuda.synchronize()
    assert P.crvq_launch_count() - n1 == n_graph
    for k, v in got.items():
        np.testing.assert_array_equal(v, host(getattr(direct, k)), err_msg=k)
    for k in ("loss_block", "loss_crit", "loss_full", "loss_pre", "scores", "flagged"):
        assert rep[k] == direct.report[k], k
