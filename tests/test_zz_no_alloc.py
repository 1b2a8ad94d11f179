"""crvq_update_codebook_noalloc against crvq_update_codebook, through the C ABI.

Some callers cannot allocate device memory: runtimes that hand out a fixed arena and forbid
cudaMalloc after start-up, plugins whose host owns every device allocation, latency-critical
callers that must not synchronise (cudaFree synchronises the device). For them the library
offers an update that keeps its scratch in a fixed device array instead of allocating. This
file is collected last so that a failure here does not hide the other tests' results; it
passes alone in a fresh process as well as after the rest of the suite.
"""
import ctypes

import numpy as np
import pytest
import torch

import synthetic as S
from oracle import crvq_oracle as O

pytestmark = pytest.mark.gpu

D = 8


def _setup(seed, K, G_cov_ext):
    cfg = S.C1
    W, X = S.gen_W(cfg), S.gen_X(cfg)
    _, _, Hb, _ = O.hessian(X, cfg.damp_rel, D)
    M, N = W.shape
    G = N // D
    rng = np.random.default_rng(seed)
    Cb = O.kmeans_init(W, D, G, K, seed)
    Ce = (0.3 * O.kmeans_init(W, D, G, 32, seed + 1)).astype(np.float32)
    cb_codes = rng.integers(0, K - 3, (M, G)).astype(np.int32)          # last codes empty
    ce_codes = rng.integers(0, 32, (M, G_cov_ext)).astype(np.int32)
    return W, Hb, Cb, Ce, cb_codes, ce_codes, G


def test_noalloc_update_matches_the_allocating_update_on_two_calls_in_a_row():
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook, build
    build.build()
    lib = P.api._L()
    for call, (seed, K, which) in enumerate([(3, 256, 0), (4, 128, 1)]):
        W, Hb, Cb, Ce, cbc, cec, G = _setup(seed, K, 4)
        Wd = torch.from_numpy(W).cuda()
        Hd = torch.from_numpy(Hb).cuda()
        cbs = [Codebook(torch.from_numpy(Cb).cuda(), torch.from_numpy(cbc).cuda(), G),
               Codebook(torch.from_numpy(Ce).cuda(), torch.from_numpy(cec).cuda(), 4)]
        ref, ref_cnt = P.crvq_update_codebook(Wd, D, Hd, cbs, which)
        Kw = cbs[which].C.shape[0]
        out = torch.full((Kw, D), float("nan"), device="cuda")
        cnt = torch.full((Kw,), -1, dtype=torch.int32, device="cuda")
        arr = P.api._cb_array(cbs)
        st = lib.crvq_update_codebook_noalloc(
            ctypes.c_void_p(Wd.data_ptr()), Wd.stride(0), W.shape[0], G, D,
            ctypes.c_void_p(Hd.data_ptr()), arr, len(cbs), which,
            ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(cnt.data_ptr()),
            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert st == 0, lib.crvq_last_error()
        torch.cuda.synchronize()
        r = ref.cpu().numpy().astype(np.float64)
        o = out.cpu().numpy().astype(np.float64)
        assert np.abs(o - r).max() <= 1e-4 * np.abs(r).max(), f"call {call}"
        np.testing.assert_array_equal(o, r)                  # same arithmetic: bit-identical
        np.testing.assert_array_equal(cnt.cpu().numpy(), ref_cnt.cpu().numpy())


def test_noalloc_update_rejects_sizes_beyond_its_scratch():
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook, build
    build.build()
    M, G, K = 2, 5000, 256                                   # 5000 x 256 counts > 4 MiB
    T = torch.zeros((M, G * D), device="cuda")
    Hb = torch.eye(D, device="cuda").repeat(G, 1, 1).contiguous()
    C = torch.zeros((K, D), device="cuda")
    codes = torch.zeros((M, G), dtype=torch.int32, device="cuda")
    with pytest.raises(P.CrvqError) as e:
        P.crvq_update_codebook_noalloc(T, D, Hb, [Codebook(C, codes, G)], 0)
    assert e.value.status == -2
    assert "static limit" in str(e.value)


def test_noalloc_update_reports_device_errors_through_crvq_sync():
    """What the kernels of the no-allocation update find on the device reaches the caller:
    an out-of-range code (skipped) comes back from the next crvq_sync as CRVQ_ERR_DEVICE, a NaN
    in another codebook as CRVQ_ERR_NUMERIC; each report is cleared once read, and a clean
    call afterwards reports nothing and still equals the allocating update."""
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import Codebook, build
    build.build()
    W, Hb, Cb, Ce, cbc, cec, G = _setup(7, 64, 4)
    Wd = torch.from_numpy(W).cuda()
    Hd = torch.from_numpy(Hb).cuda()
    torch.cuda.synchronize()
    P.crvq_sync()                                            # nothing pending beforehand

    bad_codes = cbc.copy()
    bad_codes[5, 3] = 64                                     # K = 64: out of range
    cbs = [Codebook(torch.from_numpy(Cb).cuda(), torch.from_numpy(bad_codes).cuda(), G),
           Codebook(torch.from_numpy(Ce).cuda(), torch.from_numpy(cec).cuda(), 4)]
    P.crvq_update_codebook_noalloc(Wd, D, Hd, cbs, 0)
    with pytest.raises(P.CrvqError) as e:
        P.crvq_sync()
    assert e.value.status == -7                              # CRVQ_ERR_DEVICE
    P.crvq_sync()                                            # the report was cleared

    nan_ext = Ce.copy()
    nan_ext[2, 1] = np.nan
    cbs = [Codebook(torch.from_numpy(Cb).cuda(), torch.from_numpy(cbc).cuda(), G),
           Codebook(torch.from_numpy(nan_ext).cuda(), torch.from_numpy(cec).cuda(), 4)]
    P.crvq_update_codebook_noalloc(Wd, D, Hd, cbs, 0)
    with pytest.raises(P.CrvqError) as e:
        P.crvq_sync()
    assert e.value.status == -6                              # CRVQ_ERR_NUMERIC
    P.crvq_sync()

    cbs = [Codebook(torch.from_numpy(Cb).cuda(), torch.from_numpy(cbc).cuda(), G),
           Codebook(torch.from_numpy(Ce).cuda(), torch.from_numpy(cec).cuda(), 4)]
    out, cnt = P.crvq_update_codebook_noalloc(Wd, D, Hd, cbs, 0)
    P.crvq_sync()
    ref, ref_cnt = P.crvq_update_codebook(Wd, D, Hd, cbs, 0)
    P.crvq_sync()
    np.testing.assert_array_equal(out.cpu().numpy(), ref.cpu().numpy())
    np.testing.assert_array_equal(cnt.cpu().numpy(), ref_cnt.cpu().numpy())
