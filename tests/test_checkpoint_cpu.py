"""Checkpoint / resume of layer-by-layer quantization (paper_2412_09282_gb300.checkpoint),
on the CPU with a stand-in quantizer: which matrices a run computes and which it loads, what
invalidates a stored result, and that a crash never leaves a partial file behind."""
import json
import os

import numpy as np
import pytest
import torch

import synthetic as S
from paper_2412_09282_gb300 import checkpoint as CK
from paper_2412_09282_gb300.api import LayerOutputs

CFG = S.LayerConfig("ck", 16, 32, 24, "plain", "lognormal", 0.5, K_base=8, n_ext=1, K_ext=4,
                    crit_frac=0.25, B=2, kmeans_iters=2)


class FakeQuantizer:
    """Deterministic outputs of the right shapes and dtypes, a function of W and the seed;
    counts its calls and can fail on the n-th."""

    def __init__(self, fail_at=None):
        self.calls = []
        self.fail_at = fail_at

    def __call__(self, W, X, cfg):
        self.calls.append(cfg.name)
        if self.fail_at is not None and len(self.calls) == self.fail_at:
            raise RuntimeError("quantizer failed")
        M, N = W.shape
        G, Gc = N // cfg.d, 1
        rng = np.random.default_rng(int(W.abs().sum().item() * 1e6) % 2**32 + cfg.seed)
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
        return LayerOutputs(
            perm=t(rng.permutation(N).astype(np.int32)),
            C_base=t(rng.standard_normal((cfg.K_base, cfg.d)).astype(np.float32)),
            codes_base=t(rng.integers(0, cfg.K_base, (M, G)).astype(np.int32)),
            C_ext=t(rng.standard_normal((cfg.n_ext, cfg.K_ext, cfg.d)).astype(np.float32)),
            codes_ext=t(rng.integers(0, cfg.K_ext, (cfg.n_ext, M, Gc)).astype(np.int32)),
            W_hat=None, importance=t(rng.random(N).astype(np.float32)),
            report={"loss_block": float(rng.random()), "loss_crit": 0.5, "loss_full": 1.5,
                    "scores": 1e6, "flagged": 3, "n_crit_groups": Gc})


def _layers(n=3, seed_shift=0):
    out = []
    for k in range(n):
        cfg = CFG.with_(name=f"m{k}", seed=k + seed_shift)
        out.append((f"m{k}", torch.from_numpy(S.gen_W(cfg)), torch.from_numpy(S.gen_X(cfg)), cfg))
    return out


def _same(a, b):
    for k in CK.ARRAYS:
        np.testing.assert_array_equal(np.asarray(getattr(a, k)), np.asarray(getattr(b, k)))
    assert a.report == pytest.approx(b.report)


def test_second_run_loads_everything_and_returns_the_same_results(tmp_path):
    q1 = FakeQuantizer()
    r1 = CK.quantize_layers(_layers(), str(tmp_path), q1)
    assert q1.calls == ["m0", "m1", "m2"]
    q2 = FakeQuantizer()
    r2 = CK.quantize_layers(_layers(), str(tmp_path), q2)
    assert q2.calls == []
    for k in r1:
        _same(r1[k], r2[k])
    log = [json.loads(l) for l in open(tmp_path / "log.jsonl")]
    assert [r["source"] for r in log] == ["computed"] * 3 + ["loaded"] * 3
    assert all("loss_block" in r and "scores" in r for r in log)


def test_resume_after_a_crash_recomputes_only_the_unfinished_matrices(tmp_path):
    with pytest.raises(RuntimeError):
        CK.quantize_layers(_layers(4), str(tmp_path), FakeQuantizer(fail_at=3))
    assert sorted(os.listdir(tmp_path)) == ["log.jsonl", "m0.npz", "m1.npz"]  # no partial file
    q = FakeQuantizer()
    CK.quantize_layers(_layers(4), str(tmp_path), q)
    assert q.calls == ["m2", "m3"]


def test_changed_inputs_or_configuration_invalidate_the_stored_result(tmp_path):
    CK.quantize_layers(_layers(), str(tmp_path), FakeQuantizer())
    layers = _layers()
    name, W, X, cfg = layers[1]
    layers[1] = (name, W, X, cfg.with_(B=cfg.B + 1))             # configuration changed
    name, W, X, cfg = layers[2]
    W2 = W.clone()
    W2[0, 0] += 1.0                                               # one weight changed
    layers[2] = (name, W2, X, cfg)
    q = FakeQuantizer()
    CK.quantize_layers(layers, str(tmp_path), q)
    assert q.calls == ["m1", "m2"]
    # renaming the configuration alone keeps the result (the name is not an input)
    name, W, X, cfg = _layers()[0]
    assert CK.fingerprint(W, X, cfg) == CK.fingerprint(W, X, cfg.with_(name="other"))


def test_corrupt_or_truncated_files_are_recomputed(tmp_path):
    CK.quantize_layers(_layers(), str(tmp_path), FakeQuantizer())
    p0, p1 = tmp_path / "m0.npz", tmp_path / "m1.npz"
    p0.write_bytes(p0.read_bytes()[: len(p0.read_bytes()) // 2])  # truncated
    raw = bytearray(p1.read_bytes())
    # flip one byte inside the stored codes (the zip entries are stored, not compressed)
    with np.load(p1) as z:
        needle = np.ascontiguousarray(z["codes_base"]).tobytes()[:64]
    at = bytes(raw).find(needle)
    assert at > 0
    raw[at + 5] ^= 0x01
    p1.write_bytes(bytes(raw))
    # a well-formed file whose arrays no longer match the checksum it carries
    p2 = tmp_path / "m2.npz"
    with np.load(p2) as z:
        parts = {k: np.array(z[k]) for k in z.files}
    parts["C_base"][0, 0] += 1.0
    with open(p2, "wb") as f:
        np.savez(f, **parts)
    assert CK.load(str(p0)) is None and CK.load(str(p1)) is None and CK.load(str(p2)) is None
    q = FakeQuantizer()
    CK.quantize_layers(_layers(), str(tmp_path), q)
    assert q.calls == ["m0", "m1", "m2"]
    for p in (p0, p1, p2):
        assert CK.load(str(p)) is not None


def test_names_must_be_plain_file_names(tmp_path):
    name, W, X, cfg = _layers(1)[0]
    for bad in ("", "../x", "a/b", ".hidden"):
        with pytest.raises(ValueError):
            CK.quantize_layers([(bad, W, X, cfg)], str(tmp_path), FakeQuantizer())
