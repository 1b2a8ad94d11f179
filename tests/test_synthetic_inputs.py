"""The synthetic stand-ins follow their stated recipes (the workloads' shapes and value
distributions): seeded and reproducible row by row, N(0, 0.02^2) weights with the configured
outlier columns, bf16-rounded heavy-tailed columns for the q_proj workload, SwiGLU-like sparse
activations for down_proj, LogNormal channel scales. Small row samples only (CPU, seconds)."""
import numpy as np

import synthetic as S


def _rows(cfg, n=64):
    return np.arange(n)


def test_row_subsets_regenerate_the_same_values():
    cfg = S.C1
    full = S.gen_W(cfg)
    part = S.gen_W(cfg, np.array([3, 100, 511]))
    np.testing.assert_array_equal(part, full[[3, 100, 511]])
    Xf = S.gen_X(cfg)
    np.testing.assert_array_equal(S.gen_X(cfg, np.array([0, 999])), Xf[[0, 999]])


def test_plain_weights_are_n0_002():
    W = S.gen_W(S.C3, _rows(S.C3, 32)).astype(np.float64)
    assert abs(W.mean()) < 2e-4
    assert abs(W.std() - 0.02) < 2e-4


def test_outlier_columns_are_ten_times_larger():
    cfg = S.C1
    W = S.gen_W(cfg).astype(np.float64)
    col_std = W.std(axis=0)
    big = np.sort(np.argsort(col_std)[-cfg.n_outlier_cols:])
    assert np.all(col_std[big] > 0.15) and np.median(col_std) < 0.03
    assert np.allclose(np.median(col_std[big]) / np.median(col_std), 10.0, rtol=0.15)


def test_q_proj_weights_are_bf16_with_heavy_tailed_columns():
    cfg = S.C2
    W = S.gen_W(cfg, _rows(cfg, 256))
    bits = W.view(np.uint32)
    assert np.all(bits & 0xFFFF == 0)  # every value is a bf16 number
    Wd = W.astype(np.float64)
    kurt = ((Wd - Wd.mean(0)) ** 4).mean(0) / Wd.var(0) ** 2
    heavy = np.argsort(kurt)[-cfg.n_outlier_cols:]
    assert np.median(kurt[heavy]) > 6.0          # Student t (nu = 3) columns
    assert abs(np.median(kurt) - 3.0) < 0.6      # the rest Gaussian


def test_swiglu_activations_are_seventy_percent_near_zero():
    cfg = S.C3
    X = S.gen_X(cfg, np.arange(16)).astype(np.float64)
    scale = np.exp(cfg.x_sigma * 3.0)  # a generous bound on the channel scales
    small = np.abs(X) < 1e-3 * 6.0 * scale
    assert abs(small.mean() - 0.7) < 0.02


def test_channel_scales_are_lognormal():
    cfg = S.C4
    X = S.gen_X(cfg, np.arange(512)).astype(np.float64)
    log_std = np.log(X.std(axis=0))
    # log of a LogNormal(0, sigma) scale times the unit normal's std (1)
    assert abs(log_std.std() - cfg.x_sigma) < 0.05
    assert abs(log_std.mean()) < 0.05


def test_block_matrices_share_their_calibration_input():
    layers = S.C5
    tags = {L.name.split("/")[-1]: L.x_tag for L in layers}
    assert len({tags[n] for n in ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj",
                                  "up_proj")}) == 1
    assert tags["down_proj"] != tags["q_proj"]
    q, k = layers[0], layers[1]
    np.testing.assert_array_equal(S.gen_X(q, np.arange(2)), S.gen_X(k, np.arange(2)))
