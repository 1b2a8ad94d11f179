"""Seeded synthetic inputs for the CRVQ code-search path (weights W and calibration X).

This module only draws random numbers and shapes them into the workload's matrices; it
holds none of the quantization method's arithmetic. Both the fp64 oracle (tests) and the
CUDA path (tests, bench) take their inputs from here, so the two see byte-identical data.

Random numbers come from SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014) used as a counter-based generator: output i of stream s is
mix64(s + (i+1)*0x9E3779B97F4A7C15). Uniforms take the top 53 bits; normals use the cosine
branch of Box-Muller on two uniforms. Element e of a tensor always uses counters derived from
e, so any row subset of a matrix can be regenerated on its own.

The shapes follow the paper's experimental models (LLaMA-2 7B/70B layers, 4096-token
calibration sequences, Sec. 5.1); the paper's real weights and Red_Pajama calibration text are
not available, so these seeded stand-ins replace them.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix64(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64(stream: int, counters: np.ndarray) -> np.ndarray:
    """Outputs number `counters` (0-based) of the SplitMix64 stream seeded with `stream`."""
    c = np.asarray(counters, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(stream & 0xFFFFFFFFFFFFFFFF) + (c + np.uint64(1)) * _GAMMA
    return _mix64(z)


def stream_key(seed: int, tag: str) -> int:
    """A 64-bit stream id for (seed, tag): FNV-1a of the tag, mixed with the seed."""
    h = 0xCBF29CE484222325
    for b in tag.encode():
        h = ((h ^ b) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return int(_mix64(np.array([(h ^ (seed * 0x9E3779B97F4A7C15)) & 0xFFFFFFFFFFFFFFFF],
                               dtype=np.uint64))[0])


def uniform(stream: int, counters: np.ndarray) -> np.ndarray:
    """U[0,1) doubles with 53 random bits."""
    return (splitmix64(stream, counters) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def normal(stream: int, idx: np.ndarray) -> np.ndarray:
    """Standard normals; element e uses uniforms 2e and 2e+1 of the stream (Box-Muller)."""
    e = np.asarray(idx, dtype=np.uint64)
    u1 = uniform(stream, e * np.uint64(2))
    u2 = uniform(stream, e * np.uint64(2) + np.uint64(1))
    return np.sqrt(-2.0 * np.log1p(-u1)) * np.cos(2.0 * np.pi * u2)


def _matrix_normals(stream: int, rows: np.ndarray, ncols: int) -> np.ndarray:
    rows = np.asarray(rows, dtype=np.int64)
    idx = (rows[:, None].astype(np.uint64) * np.uint64(ncols)
           + np.arange(ncols, dtype=np.uint64)[None, :])
    return normal(stream, idx)


def pick_columns(seed: int, tag: str, N: int, count: int) -> np.ndarray:
    """`count` distinct columns: the ones with the smallest hash keys, returned sorted."""
    keys = splitmix64(stream_key(seed, tag), np.arange(N))
    return np.sort(np.argsort(keys, kind="stable")[:count])


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even), returned as fp32."""
    b = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (b >> np.uint64(16)) & np.uint64(1)
    b = (b + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)
    return b.astype(np.uint32).view(np.float32)


@dataclass(frozen=True)
class LayerConfig:
    """One weight matrix to quantize and the CRVQ hyper-parameters (Alg. 1 inputs)."""
    name: str
    M: int                    # output rows
    N: int                    # input channels
    n_tok: int                # calibration tokens (rows of X)
    w_kind: str               # "plain" | "outlier_cols" | "heavy_bf16"
    x_kind: str               # "lognormal" | "swiglu"
    x_sigma: float = 0.5      # LogNormal(0, x_sigma) channel scales of X
    n_outlier_cols: int = 0   # columns of W that are enlarged or heavy-tailed
    d: int = 8
    K_base: int = 256
    n_ext: int = 1
    K_ext: int = 256
    crit_frac: float = 0.02
    B: int = 8
    kmeans_iters: int = 10
    refine_rounds: int = 1
    eps_rel: float = 1e-3
    damp_rel: float = 0.01
    importance_mode: int = 0  # 0 = W-A (App. A.2), 1 = W-only, 2 = random
    seed: int = 0
    x_tag: str = ""           # layers that share X use the same tag
    n_base: int = 1           # base codebooks over every group (Sec. 6.4's m = 2 setting)

    @property
    def G(self) -> int:
        return self.N // self.d

    def with_(self, **kw) -> "LayerConfig":
        return dataclasses.replace(self, **kw)


def _by_row_chunks(fn, n_rows: int, chunk: int = 2048) -> np.ndarray:
    """fn(rows) over row chunks on a thread pool (numpy releases the GIL in its loops). The
    generators are counter-based, so every element depends only on its own indices and the
    chunked result equals the one-shot one."""
    if n_rows <= chunk:
        return fn(np.arange(n_rows))
    parts = [np.arange(r0, min(n_rows, r0 + chunk)) for r0 in range(0, n_rows, chunk)]
    workers = min(len(parts), os.cpu_count() or 1, 16)
    with ThreadPoolExecutor(max_workers=workers) as ex:
        return np.ascontiguousarray(np.concatenate(list(ex.map(fn, parts)), axis=0))


def gen_W(cfg: LayerConfig, rows: np.ndarray | None = None) -> np.ndarray:
    """Weights: N(0, 0.02^2), with the configured outlier columns; fp32 M x N (or a row subset)."""
    if rows is None:
        return _by_row_chunks(lambda r: gen_W(cfg, r), cfg.M)
    rows = np.asarray(rows)
    s = stream_key(cfg.seed, cfg.name + "/W")
    W = 0.02 * _matrix_normals(s, rows, cfg.N)
    if cfg.w_kind == "outlier_cols":
        cols = pick_columns(cfg.seed, cfg.name + "/W/outliers", cfg.N, cfg.n_outlier_cols)
        W[:, cols] *= 10.0
    elif cfg.w_kind == "heavy_bf16":
        cols = pick_columns(cfg.seed, cfg.name + "/W/heavy", cfg.N, cfg.n_outlier_cols)
        sub = np.arange(len(cols))
        z = [_matrix_normals(stream_key(cfg.seed, cfg.name + f"/W/t{j}"), rows, len(cols))
             for j in range(4)]
        chi2 = (z[1] ** 2 + z[2] ** 2 + z[3] ** 2) / 3.0
        W[:, cols[sub]] = 0.02 * z[0] / np.sqrt(chi2)
    elif cfg.w_kind != "plain":
        raise ValueError(cfg.w_kind)
    W = W.astype(np.float32)
    if cfg.w_kind == "heavy_bf16":
        W = round_to_bf16(W)
    return np.ascontiguousarray(W)


def gen_X(cfg: LayerConfig, rows: np.ndarray | None = None) -> np.ndarray:
    """Calibration activations: n_tok x N fp32, row = token, per-channel LogNormal scales."""
    if rows is None:
        return _by_row_chunks(lambda r: gen_X(cfg, r), cfg.n_tok)
    rows = np.asarray(rows)
    tag = cfg.x_tag or cfg.name
    s_scale = stream_key(cfg.seed, tag + "/X/scale")
    scale = np.exp(cfg.x_sigma * normal(s_scale, np.arange(cfg.N)))
    X = _matrix_normals(stream_key(cfg.seed, tag + "/X"), rows, cfg.N) * scale[None, :]
    if cfg.x_kind == "swiglu":
        # 30% of activations active, the rest shrunk by 1e-3 (SwiGLU-like sparsity).
        rr = np.asarray(rows, dtype=np.int64)
        idx = rr[:, None].astype(np.uint64) * np.uint64(cfg.N) + np.arange(cfg.N, dtype=np.uint64)
        u = uniform(stream_key(cfg.seed, tag + "/X/gate"), idx)
        X = np.where(u < 0.3, X, 1e-3 * X)
    elif cfg.x_kind != "lognormal":
        raise ValueError(cfg.x_kind)
    return np.ascontiguousarray(X.astype(np.float32))


# The five workloads. C1 is small enough for the oracle end to end; C2 (a LLaMA-2-7B q_proj)
# is the headline workload; C3-C5 are the larger LLaMA-shaped cases.
C1 = LayerConfig("c1_512x512", 512, 512, 1024, "outlier_cols", "lognormal", 0.5,
                 n_outlier_cols=8, n_ext=2, B=4)
C2 = LayerConfig("c2_q_proj_4096x4096", 4096, 4096, 4096, "heavy_bf16", "lognormal", 0.5,
                 n_outlier_cols=41, n_ext=1, B=8)
C3 = LayerConfig("c3_down_proj_4096x11008", 4096, 11008, 4096, "plain", "swiglu", 0.5,
                 K_base=65536, n_ext=1, crit_frac=0.01, B=8)
C4 = LayerConfig("c4_up_proj_28672x8192", 28672, 8192, 2048, "plain", "lognormal", 0.7,
                 n_ext=4, crit_frac=0.05, B=8)


def _c5_layers() -> list[LayerConfig]:
    base = dict(n_ext=2, crit_frac=0.02, B=8, w_kind="outlier_cols")
    out = []
    for nm, M, N in [("q_proj", 4096, 4096), ("k_proj", 4096, 4096), ("v_proj", 4096, 4096),
                     ("o_proj", 4096, 4096), ("gate_proj", 11008, 4096),
                     ("up_proj", 11008, 4096), ("down_proj", 4096, 11008)]:
        if nm == "down_proj":
            out.append(LayerConfig("c5_block/" + nm, M, N, 4096, x_kind="swiglu", x_sigma=0.5,
                                   n_outlier_cols=N // 100, x_tag="c5_block/X_down", **base))
        else:
            out.append(LayerConfig("c5_block/" + nm, M, N, 4096, x_kind="lognormal",
                                   x_sigma=0.5, n_outlier_cols=N // 100,
                                   x_tag="c5_block/X_attn_mlp", **base))
    return out


C5 = _c5_layers()

CONFIGS = {"c1": C1, "c2": C2, "c3": C3, "c4": C4}
