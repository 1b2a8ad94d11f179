"""The reorder-strategy / lambda / m settings of the synthetic ablation (Table 2, Sec. 6.3-6.4)
through crvq_quantize_layer, end to end against independent oracle runs: each importance mode
(random, W-only, W-A in the App. A.2 form and as Eq. (wa) with the inverse-Hessian diagonal),
a larger critical ratio with three extended codebooks, and two base codebooks with three
extended ones (Sec. 6.4's m = 2 setting). When the
final codes agree the losses agree to 1e-4; the channel order always agrees exactly."""
import numpy as np
import pytest
import torch

import synthetic as S
from oracle import crvq_oracle as O
from parity_util import dev, host

pytestmark = pytest.mark.gpu


def _cmp(out, ref, cfg):
    np.testing.assert_array_equal(host(out.perm), ref["perm"])
    cbs = ref["codebooks"]
    M, G = cfg.M, cfg.N // cfg.d
    gpu = list(host(out.codes_base).reshape(cfg.n_base, M, G)) + \
        [host(out.codes_ext[t]) for t in range(cfg.n_ext)]
    assert len(gpu) == len(cbs)
    same = all(np.array_equal(g, cb.codes) for g, cb in zip(gpu, cbs))
    if same:
        for key in ("loss_block", "loss_crit", "loss_full", "loss_pre"):
            assert abs(out.report[key] - ref[key]) <= 1e-4 * abs(ref[key]), key
    return same


@pytest.mark.parametrize("mode,lam,n_ext,n_base", [(2, 0.02, 1, 1), (1, 0.02, 1, 1),
                                                   (0, 0.02, 1, 1), (3, 0.02, 1, 1),
                                                   (0, 0.10, 3, 1), (0, 0.10, 3, 2)])
def test_sweep_settings_match_independent_oracle_runs(mode, lam, n_ext, n_base):
    import paper_2412_09282_gb300 as P
    cfg = S.LayerConfig("sweep_small", 192, 256, 384, "outlier_cols", "lognormal", 0.5,
                        n_outlier_cols=4, K_base=64, n_ext=n_ext, K_ext=32, crit_frac=lam,
                        B=4, kmeans_iters=4, importance_mode=mode, n_base=n_base)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    out = P.crvq_quantize_layer(dev(W), dev(X), cfg)
    P.crvq_sync()
    ref = O.quantize_layer(W, X, cfg)
    assert out.report["n_crit_groups"] == ref["n_crit_groups"]
    _cmp(out, ref, cfg)
    # the critical loss never rises with each extended codebook (before the refinement)
    cl = ref["crit_loss_after_ext"]
    assert all(b <= a * (1 + 1e-9) for a, b in zip(cl, cl[1:]))
