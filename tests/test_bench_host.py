"""Host-side logic of bench.py on the CPU: the score count that the CPU baseline's rate
divides by is the number of (hypothesis, codeword) pairs the schedule actually scores; the
oracle pool; the assignment of a block's matrices to streams; the sweep's bit-widths."""
import numpy as np
import pytest


@pytest.mark.parametrize("n_base", [1, 2])
def test_schedule_scores_counts_what_the_schedule_scores(monkeypatch, n_base):
    """bench.schedule_scores (the CPU baseline's numerator) against the pairs the oracle's
    schedule actually scores: every encode call is counted from its arguments (per group, each
    searched stage scores parents x K pairs per vector, parents = min(B, parents x K))."""
    import bench
    from oracle import crvq_oracle as O
    import synthetic as S
    cfg = S.LayerConfig("count", 16, 64, 32, "plain", "lognormal", 0.5, K_base=8, n_ext=2,
                        K_ext=4, crit_frac=0.1, B=2, kmeans_iters=2, n_base=n_base)
    counted = []
    orig = O.encode_beam

    def counting(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        M = np.asarray(T).shape[0]
        total = 0
        for g in range(np.asarray(H_blocks).shape[0]):
            parents = 1
            for s in range(n_fixed, len(cbs)):
                if g < cbs[s].G_cov:
                    K = cbs[s].C.shape[0]
                    total += M * parents * K
                    parents = min(B, parents * K)
        counted.append(total)
        return orig(T, d, H_blocks, cbs, n_fixed, B, keep_if_better, **kw)

    monkeypatch.setattr(O, "encode_beam", counting)
    O.quantize_layer(S.gen_W(cfg), S.gen_X(cfg), cfg)
    assert sum(counted) == bench.schedule_scores(cfg, cfg.M, cfg.N)


def test_oracle_pool_runs_one_sample_per_core_and_counts_their_scores():
    """The all-cores CPU baseline: worker processes (spawn) each run the oracle's whole
    schedule on their own rows; the rate counts every worker's scores over the common span."""
    import bench
    import synthetic as S
    cfg = S.LayerConfig("pool", 32, 64, 32, "plain", "lognormal", 0.5, K_base=8, n_ext=1,
                        K_ext=4, crit_frac=0.1, B=2, kmeans_iters=1)
    assert bench.rows_needed(cfg) == 4                   # K_ext = 4 over one critical group
    pool = bench.OraclePool(cfg, 2)
    try:
        rate, wall, cores, desc = pool.run(0.05)
    finally:
        pool.close()
    rows = pool.rows_for(0.05)
    assert cores == 2 and wall > 0
    assert abs(rate * wall - 2 * bench.schedule_scores(cfg, rows, cfg.N)) <= 1e-6 * rate * wall
    assert "2 row blocks" in desc


def test_lanes_cover_every_matrix_once_largest_first():
    import bench
    import synthetic as S
    sizes = [c.M * c.N for c in S.C5]
    for streams in (1, 2, 3, 4, 7, 12):
        lanes = bench.assign_lanes(sizes, streams)
        assert len(lanes) == min(streams, len(sizes))
        assert sorted(j for lane in lanes for j in lane) == list(range(len(sizes)))
        loads = [sum(sizes[j] for j in lane) for lane in lanes]
        # greedy longest-first: no lane exceeds the lightest by more than one matrix
        assert max(loads) - min(loads) <= max(sizes)
        for lane in lanes:  # each lane runs its largest matrix first
            assert [sizes[j] for j in lane] == sorted((sizes[j] for j in lane), reverse=True)
    # the block's three 11008 x 4096 / 4096 x 11008 matrices go to different lanes with 3
    big = [j for j, s in enumerate(sizes) if s == max(sizes)]
    lanes = bench.assign_lanes(sizes, 3)
    assert sorted(lane[0] for lane in lanes) == sorted(big)
    assert bench.assign_lanes([5], 3) == [[0]]


def test_sweep_bit_width_with_two_base_codebooks_follows_eq_bitwidth():
    """With no extended codebooks (lambda = 0) and no reorder index the setting is plain
    additive VQ, and Sec. 3.2 Eq. (bitwidth) for a 4096 x 4096 matrix gives
    n = m e / d + 2^(e - 20) m d (m = 2, e = 8, d = 8: 2 + 2^-12 * 16); the reorder index adds
    16 bits per channel (App. A.1)."""
    import bench
    import synthetic as S
    import paper_2412_09282_gb300 as P
    try:
        P.crvq_version()
    except (ImportError, OSError):
        pytest.skip("libcrvq.so not built")
    cfg = S.LayerConfig("bits", 4096, 4096, 8, "plain", "lognormal", 0.5, K_base=256, n_ext=0,
                        crit_frac=0.0, n_base=2)
    perm_bits = 16 * 4096 / 4096 ** 2
    assert bench.avg_bits_of(P, cfg) == pytest.approx(2 * 8 / 8 + 2 ** -12 * 2 * 8 + perm_bits,
                                                      rel=1e-12)
    cfg3 = cfg.with_(n_ext=3, crit_frac=0.02)
    one = bench.avg_bits_of(P, cfg3.with_(n_base=1))
    assert bench.avg_bits_of(P, cfg3) == pytest.approx(one + 1 + 2 ** -12 * 8, rel=1e-12)
