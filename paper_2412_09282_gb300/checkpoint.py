"""Layer-by-layer quantization with checkpoint and resume.

CRVQ quantizes the linear layers of a model one after another (Alg. 1, outer loop; Sec. 4.4),
so every finished matrix is a natural checkpoint. `quantize_layers` runs a sequence of
matrices through a quantizer (crvq_quantize_layer by default) and writes each result to
`<out_dir>/<name>.npz` as soon as it is done: the permutation, the codebooks, the codes, the
importance and the report, but not W_hat, which the codes and codebooks reproduce. Each file
is written under a temporary name and renamed, so a crash leaves either the old file or the
new one, never a partial file. Each file carries:
  * a fingerprint of what produced it: the configuration, the shapes and a digest of W and X;
  * a SHA-256 checksum of its arrays.
A later run with the same out_dir loads every matrix whose file verifies and whose
fingerprint matches, and quantizes only the others. One JSON line per matrix goes to
`<out_dir>/log.jsonl`: its name, whether it was computed or loaded, the wall time, the
losses and the number of scored pairs.

Host-side bookkeeping only: every step of the method runs in the library's kernels.
"""
from __future__ import annotations

import dataclasses
import hashlib
import json
import os
import time
import zipfile
from typing import Callable, Iterable

import numpy as np

ARRAYS = ("perm", "C_base", "codes_base", "C_ext", "codes_ext", "importance")
FORMAT = 1


def _host(t) -> np.ndarray:
    """A tensor or array as a contiguous host numpy array."""
    if hasattr(t, "detach"):
        t = t.detach()
        if t.device.type != "cpu":
            t = t.cpu()
        t = t.numpy()
    return np.ascontiguousarray(t)


def _tensor_digest(t) -> str:
    """SHA-256 of a tensor's bytes (copied to the host once)."""
    a = _host(t)
    h = hashlib.sha256()
    h.update(str(a.dtype).encode())
    h.update(repr(a.shape).encode())
    h.update(memoryview(a).cast("B"))
    return h.hexdigest()


def fingerprint(W, X, cfg) -> str:
    """What a stored result depends on: the configuration, the shapes and the bytes of W and X.

    Every field of the configuration takes part except its name, so renaming a layer keeps the
    stored result, and any other change invalidates it."""
    if dataclasses.is_dataclass(cfg):
        fields = {f.name: getattr(cfg, f.name) for f in dataclasses.fields(cfg)}
    else:
        fields = dict(vars(cfg))
    fields.pop("name", None)
    doc = {"format": FORMAT, "cfg": {k: repr(v) for k, v in sorted(fields.items())},
           "W": _tensor_digest(W), "X": _tensor_digest(X)}
    return hashlib.sha256(json.dumps(doc, sort_keys=True).encode()).hexdigest()


def _arrays_checksum(arrays: dict) -> str:
    h = hashlib.sha256()
    for k in ARRAYS:
        a = arrays[k]
        h.update(k.encode())
        h.update(str(a.dtype).encode())
        h.update(repr(a.shape).encode())
        h.update(memoryview(np.ascontiguousarray(a)).cast("B"))
    return h.hexdigest()


def save(path: str, outputs, fp: str) -> None:
    """Writes one matrix's result to `path` atomically (temporary file, then rename)."""
    arrays = {k: _host(getattr(outputs, k)) for k in ARRAYS}
    meta = {"format": FORMAT, "fingerprint": fp, "checksum": _arrays_checksum(arrays),
            "report": {k: (float(v) if isinstance(v, float) else int(v))
                       for k, v in outputs.report.items()}}
    tmp = f"{path}.tmp.{os.getpid()}"
    try:
        with open(tmp, "wb") as f:
            np.savez(f, meta=np.array(json.dumps(meta)), **arrays)
            f.flush()
            os.fsync(f.fileno())
        os.replace(tmp, path)
    finally:
        if os.path.exists(tmp):
            os.remove(tmp)


def load(path: str, fp: str | None = None):
    """The stored result at `path` as a LayerOutputs of host tensors (W_hat None), or None when
    the file is missing, unreadable, fails its checksum, or was made from other inputs
    (fingerprint differs from `fp`)."""
    import torch
    from .api import LayerOutputs
    if not os.path.exists(path):
        return None
    try:
        with np.load(path, allow_pickle=False) as z:
            meta = json.loads(str(z["meta"]))
            arrays = {k: np.array(z[k]) for k in ARRAYS}
    except (OSError, ValueError, KeyError, EOFError, zipfile.BadZipFile):
        return None
    if meta.get("format") != FORMAT or meta.get("checksum") != _arrays_checksum(arrays):
        return None
    if fp is not None and meta.get("fingerprint") != fp:
        return None
    t = {k: torch.from_numpy(v) for k, v in arrays.items()}
    return LayerOutputs(perm=t["perm"], C_base=t["C_base"], codes_base=t["codes_base"],
                        C_ext=t["C_ext"], codes_ext=t["codes_ext"], W_hat=None,
                        importance=t["importance"], report=dict(meta["report"]))


def quantize_layers(layers: Iterable, out_dir: str,
                    quantize: Callable | None = None, log: bool = True) -> dict:
    """Quantizes (name, W, X, cfg) items in order, resuming from `out_dir`.

    A matrix whose stored file verifies and matches its inputs is loaded instead of
    quantized. `quantize(W, X, cfg)` defaults to crvq_quantize_layer without W_hat. Returns
    {name: LayerOutputs}, with device tensors for computed matrices and host tensors for
    loaded ones."""
    if quantize is None:
        from .api import crvq_quantize_layer

        def quantize(W, X, cfg):
            return crvq_quantize_layer(W, X, cfg, want_W_hat=False)
    os.makedirs(out_dir, exist_ok=True)
    results = {}
    for name, W, X, cfg in layers:
        if not name or os.sep in name or name.startswith("."):
            raise ValueError(f"layer name {name!r} is not a plain file name")
        path = os.path.join(out_dir, f"{name}.npz")
        t0 = time.perf_counter()
        fp = fingerprint(W, X, cfg)
        out = load(path, fp)
        source = "loaded"
        if out is None:
            out = quantize(W, X, cfg)
            save(path, out, fp)
            source = "computed"
        results[name] = out
        if log:
            rec = {"name": name, "source": source, "seconds": time.perf_counter() - t0}
            rec.update({k: out.report[k] for k in ("loss_block", "loss_crit", "loss_full",
                                                   "scores") if k in out.report})
            with open(os.path.join(out_dir, "log.jsonl"), "a") as f:
                f.write(json.dumps(rec) + "\n")
    return results
