"""Layers quantized at once from several host threads, each on its own stream, give the same
results bit for bit as one after another: the library replays each layer's captured graph on
the caller's stream without holding its cache lock, and a host-buffer call takes staging
buffers no other running call uses. Every kernel is deterministic, so any race between the
concurrent layers would show as a difference."""
import threading

import numpy as np
import pytest
import torch

import synthetic as S
from parity_util import host

pytestmark = pytest.mark.gpu

FIELDS = ("perm", "C_base", "codes_base", "C_ext", "codes_ext", "W_hat")


def _snapshot(out):
    snap = {f: host(getattr(out, f)).copy() for f in FIELDS if getattr(out, f) is not None}
    snap["losses"] = tuple(out.report[k] for k in ("loss_pre", "loss_block", "loss_crit",
                                                   "loss_full"))
    return snap


def _same(a, b):
    for k in a:
        if k == "losses":
            assert a[k] == b[k]
        else:
            np.testing.assert_array_equal(a[k], b[k], err_msg=k)


@pytest.mark.parametrize("on_host", [False, True])
def test_concurrent_layers_equal_sequential(on_host):
    import paper_2412_09282_gb300 as P
    cfgs = [S.C1.with_(name=f"conc_{j}", seed=S.C1.seed + 17 * j) for j in range(3)]
    data = []
    for cfg in cfgs:
        W = torch.from_numpy(S.gen_W(cfg))
        X = torch.from_numpy(S.gen_X(cfg))
        if on_host:
            data.append((W.pin_memory(), X.pin_memory()))
        else:
            data.append((W.cuda(), X.cuda()))
    ref = []
    for (W, X), cfg in zip(data, cfgs):
        ref.append(_snapshot(P.crvq_quantize_layer(W, X, cfg, device=torch.device("cuda"))))
    torch.cuda.synchronize()

    got = [None] * len(cfgs)
    errors = []

    def lane(j, s):
        try:
            with torch.cuda.stream(s):
                W, X = data[j]
                out = None
                for _ in range(2):  # the first call captures the layer's graph, the second replays it
                    out = P.crvq_quantize_layer(W, X, cfgs[j], out=out, stream=s,
                                                device=torch.device("cuda"))
                got[j] = _snapshot(out)
        except Exception as e:  # reported on the main thread
            errors.append(e)

    streams = [torch.cuda.Stream() for _ in cfgs]
    threads = [threading.Thread(target=lane, args=(j, s)) for j, s in enumerate(streams)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    P.crvq_sync()
    assert not errors, errors
    for j in range(len(cfgs)):
        _same(ref[j], got[j])
