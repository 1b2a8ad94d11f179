"""The beam stage on the tensor cores (beam_tc_kernel) keeps exactly the lists of the SIMT
stage (beam_stage_kernel): its tensor-core scores only filter the candidates, which are scored
again with the SIMT stage's fp32 chain and inserted in the same order with the same rule. With
CRVQ_BEAM_TC=0 every stage runs on the SIMT kernel; the codes and the vectors' errors of the
two runs must be equal bit for bit (beam widths 1, 2, 4, 8: lists of 2 to 9 entries; one and
two 128-codeword chunks; partial coverage by the extended codebooks)."""
import os

import numpy as np
import pytest
import torch

from parity_util import dev, host

pytestmark = pytest.mark.gpu

D = 8


def _case(seed, M, G, Gc, Ks):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((512, G * D)) * rng.lognormal(0.0, 0.5, G * D)
    H = X.T @ X / 512 + 0.01 * np.eye(G * D)
    Hb = np.stack([H[g * D:(g + 1) * D, g * D:(g + 1) * D] for g in range(G)]).astype(np.float32)
    W = (0.02 * rng.standard_normal((M, G * D))).astype(np.float32)
    Cs = [(0.02 * rng.standard_normal((Ks[0], D))).astype(np.float32)]
    for j, K in enumerate(Ks[1:]):
        Cs.append((0.02 * 0.4 ** (j + 1) * rng.standard_normal((K, D))).astype(np.float32))
    return W, Hb, Cs


def _run(W, Hb, Cs, G, Gc, B):
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook
    M = W.shape[0]
    covs = [G] + [Gc] * (len(Cs) - 1)
    codes = [torch.zeros((M, c), dtype=torch.int32, device="cuda") for c in covs]
    cbs = [Codebook(dev(C), cd, c) for C, cd, c in zip(Cs, codes, covs)]
    verr = P.crvq_encode_beam(dev(W), D, dev(Hb), cbs, 0, B, want_err=True)
    P.crvq_sync()
    return [host(c).copy() for c in codes], host(verr).copy()


@pytest.mark.parametrize("B", [1, 2, 4, 8])
@pytest.mark.parametrize("shape", [(640, 24, 7, (256, 256, 256)), (300, 16, 16, (96, 200))])
def test_tensor_core_beam_equals_simt_beam(B, shape):
    M, G, Gc, Ks = shape
    W, Hb, Cs = _case(B * 7 + G, M, G, Gc, Ks)
    old = os.environ.get("CRVQ_BEAM_TC")
    try:
        os.environ["CRVQ_BEAM_TC"] = "0"
        simt_codes, simt_err = _run(W, Hb, Cs, G, Gc, B)
        os.environ["CRVQ_BEAM_TC"] = "1"
        tc_codes, tc_err = _run(W, Hb, Cs, G, Gc, B)
    finally:
        if old is None:
            os.environ.pop("CRVQ_BEAM_TC", None)
        else:
            os.environ["CRVQ_BEAM_TC"] = old
    for a, b in zip(simt_codes, tc_codes):
        np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(simt_err, tc_err)
