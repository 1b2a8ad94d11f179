"""The inference product from codes (App. "Inference Speed", Table speed) through the C ABI,
against the fp64 oracle's lookup-table product (O.lut_matvec, pinned on the CPU against the
explicit route W_hat x).

Bar: |y_gpu - y_oracle| <= 1e-5 * sum over the terms of |<c, x>|, the sum taken with |C| and
|x| (fp32 arithmetic: each codeword-input product is an 8-term FMA chain, a warp adds 32 group
terms in a 5-level tree, the slices are added in order, so the rounding error is below about
(8 + 5 + slices) * 2^-24 of that sum).
"""
import numpy as np
import pytest
import torch

from oracle import crvq_oracle as O
from parity_util import dev, host

pytestmark = pytest.mark.gpu

D = 8


def _case(seed, M, N, Ks, Gcs):
    rng = np.random.default_rng(seed)
    G = N // D
    perm = rng.permutation(N).astype(np.int32)
    cbs = []
    for K, Gc in zip(Ks, Gcs):
        C = (rng.standard_normal((K, D)) * (0.02 if not cbs else 0.005)).astype(np.float32)
        codes = rng.integers(0, K, (M, Gc)).astype(np.int32)
        cbs.append(O.Codebook(C, codes, Gc))
    return perm, cbs, G


def _check(Xin, perm, cbs, M):
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook
    gcbs = [Codebook(dev(cb.C), dev(cb.codes.astype(np.int32)), cb.G_cov) for cb in cbs]
    Y = P.crvq_lut_matvec(dev(Xin), None if perm is None else dev(perm), gcbs, M)
    P.crvq_sync()
    ref = O.lut_matvec(Xin, perm, cbs, D)
    scale = O.lut_matvec(np.abs(Xin), perm,
                         [O.Codebook(np.abs(cb.C), cb.codes, cb.G_cov) for cb in cbs], D)
    err = np.abs(host(Y).astype(np.float64) - ref)
    assert np.all(err <= 1e-5 * scale + 1e-30), float((err / scale).max())
    return Y


@pytest.mark.parametrize("b", [1, 3, 8])
def test_lut_matvec_ragged_shapes_with_extended_codebooks(b):
    """203 rows, 33 groups (two slices, the second with one group), a base codebook over every
    group and two extended codebooks on the first 3 groups, shared-memory tables."""
    M, N = 203, 264
    perm, cbs, G = _case(1, M, N, [256, 32, 7], [33, 3, 3])
    X = np.random.default_rng(2).standard_normal((b, N)).astype(np.float32)
    _check(X, perm, cbs, M)


def test_lut_matvec_large_codebook_uses_direct_codeword_products():
    """K = 4096: the slice's tables would not fit in shared memory, so the kernel dots the
    codewords directly; identity order."""
    M, N = 77, 520
    _, cbs, G = _case(3, M, N, [4096, 256], [65, 6])
    X = np.random.default_rng(4).standard_normal((2, N)).astype(np.float32)
    _check(X, None, cbs, M)


def test_lut_matvec_equals_the_reconstruction_times_the_input():
    """On a quantized layer's own outputs: the product from codes equals W_hat x with W_hat
    from crvq_quantize_layer (both fp32; W_hat rounded once per element)."""
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook
    import synthetic as S
    cfg = S.C1
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = P.crvq_quantize_layer(dev(W), dev(X), cfg)
    P.crvq_sync()
    G, Gc = cfg.N // D, out.report["n_crit_groups"]
    cbs = [Codebook(out.C_base, out.codes_base, G)] + \
        [Codebook(out.C_ext[t].contiguous(), out.codes_ext[t], Gc) for t in range(cfg.n_ext)]
    xin = X[:4]
    Y = P.crvq_lut_matvec(dev(xin), out.perm, cbs, cfg.M)
    P.crvq_sync()
    ref = xin.astype(np.float64) @ host(out.W_hat).astype(np.float64).T
    scale = np.abs(xin).astype(np.float64) @ np.abs(host(out.W_hat)).astype(np.float64).T
    assert np.all(np.abs(host(Y) - ref) <= 1e-5 * scale)
    # the same through the oracle on the layer's codes
    ocbs = [O.Codebook(host(cb.C), host(cb.codes), cb.G_cov) for cb in cbs]
    _check(xin, host(out.perm), ocbs, cfg.M)


def test_lut_matvec_llama_gate_proj_shape_sampled():
    """The decoder block's gate_proj shape (11008 x 4096, 512 groups = 16 slices; base K = 256
    and two extended codebooks on 11 groups), one input, every row against the oracle."""
    M, N = 11008, 4096
    perm, cbs, G = _case(5, M, N, [256, 256, 256], [512, 11, 11])
    X = np.random.default_rng(6).standard_normal((1, N)).astype(np.float32)
    _check(X, perm, cbs, M)


def test_lut_matvec_is_deterministic_and_reports_bad_codes():
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook
    M, N = 64, 256
    perm, cbs, G = _case(7, M, N, [256], [32])
    X = dev(np.random.default_rng(8).standard_normal((2, N)).astype(np.float32))
    codes = dev(cbs[0].codes.astype(np.int32))
    gcbs = [Codebook(dev(cbs[0].C), codes, G)]
    a = P.crvq_lut_matvec(X, dev(perm), gcbs, M)
    b = P.crvq_lut_matvec(X, dev(perm), gcbs, M)
    P.crvq_sync()
    assert torch.equal(a, b)
    codes[3, 5] = 256                                        # out of range: skipped, reported
    P.crvq_lut_matvec(X, dev(perm), gcbs, M)
    with pytest.raises(P.CrvqError) as e:
        P.crvq_sync()
    assert e.value.status == -7
    P.crvq_sync()
    with pytest.raises(P.CrvqError) as e:                    # more than 8 inputs
        P.crvq_lut_matvec(dev(np.zeros((9, N), np.float32)), dev(perm), gcbs, M)
    assert e.value.status == -2
