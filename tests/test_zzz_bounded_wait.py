"""Failure detection of the bounded device waits, made on purpose without a fault.

Every spin-wait in the library's kernels (mbarrier phases of the tensor-core pipelines) gives
up after 2 s of %globaltimer, records ERRBIT_TIMEOUT in the device error word and lets the
kernel exit, so the context stays usable; the host learns of it at the next crvq_sync. The
self-test entry waits on an mbarrier that nothing arrives on, with that same wait. This file
is collected last so that a failure here does not hide the other tests' results.
"""
import time

import numpy as np
import pytest
import torch

import synthetic as S
from oracle import crvq_oracle as O

pytestmark = pytest.mark.gpu


def test_a_wait_that_runs_out_reports_timeout_and_leaves_the_context_usable():
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300.api import CrvqError

    torch.cuda.synchronize()
    P.crvq_sync()                                    # nothing pending beforehand
    t0 = time.perf_counter()
    P.crvq_selftest_bounded_wait()
    with pytest.raises(CrvqError) as e:
        P.crvq_sync()
    waited = time.perf_counter() - t0
    assert e.value.status == -5                      # CRVQ_ERR_TIMEOUT
    assert 1.5 < waited < 30.0                       # the 2 s bound, not a hang
    P.crvq_sync()                                    # the report was cleared

    # the context still computes: S1 on a small case against the oracle
    cfg = S.C1
    X = S.gen_X(cfg)[:512]
    H, xsq, Hb, delta = P.crvq_hessian(torch.from_numpy(X).cuda(), cfg.damp_rel, 8)
    P.crvq_sync()
    H_o, xsq_o, Hb_o, delta_o = O.hessian(X, cfg.damp_rel, 8)
    scale = np.sqrt(np.outer(np.diag(H_o), np.diag(H_o)))
    assert np.all(np.abs(H.cpu().numpy() - H_o) <= 2e-5 * scale + 1e-30)


def test_non_finite_input_is_reported_and_leaves_the_context_usable():
    """A NaN in W is reported by the layer call (the column maxima flag it; the vector whose
    target is NaN has no finite score and its exact decision reports it), not turned into a
    fault: every index the kernels derive from data is range-checked."""
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300.api import CrvqError

    cfg = S.C1.with_(kmeans_iters=2)
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    Wn = W.copy()
    Wn[3, 17] = np.nan
    torch.cuda.synchronize()
    P.crvq_sync()
    with pytest.raises(CrvqError) as e:
        P.crvq_quantize_layer(torch.from_numpy(Wn).cuda(), torch.from_numpy(X).cuda(), cfg)
        P.crvq_sync()
    assert e.value.status in (-6, -7)                # NUMERIC (or DEVICE for a refused index)
    P.crvq_sync()                                    # the report was cleared
    out = P.crvq_quantize_layer(torch.from_numpy(W).cuda(), torch.from_numpy(X).cuda(), cfg)
    P.crvq_sync()
    assert np.isfinite(out.report["loss_full"]) and out.report["loss_full"] > 0
