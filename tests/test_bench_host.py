"""Host-side logic of bench.py on the CPU: the score count that the CPU baseline's rate
divides by is the number of (hypothesis, codeword) pairs the schedule actually scores."""
import numpy as np


def test_schedule_scores_counts_what_the_schedule_scores(monkeypatch):
    """bench.schedule_scores (the CPU baseline's numerator) against the pairs the oracle's
    schedule actually scores: every encode call is counted from its arguments (per group, each
    searched stage scores parents x K pairs per vector, parents = min(B, parents x K))."""
    import bench
    from oracle import crvq_oracle as O
    import synthetic as S
    cfg = S.LayerConfig("count", 16, 64, 32, "plain", "lognormal", 0.5, K_base=8, n_ext=2,
                        K_ext=4, crit_frac=0.1, B=2, kmeans_iters=2)
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
