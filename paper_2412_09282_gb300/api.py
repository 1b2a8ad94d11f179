"""Python binding of libcrvq with the C names (argument marshalling only).

Tensors are torch CUDA tensors (fp32 / int32). Each call enqueues on the current torch
stream of the tensors' device unless `stream` is given. Outputs that are not passed in are
allocated with torch.empty on the same device. Errors raise CrvqError with the library's
message.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

import torch

from . import _lib

IMPORTANCE_WA, IMPORTANCE_W_ONLY, IMPORTANCE_RANDOM, IMPORTANCE_WA_INV = 0, 1, 2, 3
STATUS = {0: "OK", -1: "INVALID_ARG", -2: "UNSUPPORTED", -3: "CUDA", -4: "NOMEM",
          -5: "TIMEOUT", -6: "NUMERIC", -7: "DEVICE"}


class CrvqError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"crvq status {status} ({STATUS.get(status, '?')}): {msg}")
        self.status = status


def library_path() -> str:
    return _lib.LIB_PATH


def _L():
    return _lib.load()


def _check(st: int):
    if st != 0:
        raise CrvqError(st, _L().crvq_last_error().decode())


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream, device):
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return C.c_void_p(stream.cuda_stream)


def _need(t: torch.Tensor, dtype, name):
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.device.type != "cuda":
        raise TypeError(f"{name} must be a CUDA tensor")


def _rowmajor(t: torch.Tensor, name):
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError(f"{name} must be a 2-D tensor with unit column stride")


@dataclass
class Codebook:
    """C: K x d codewords; codes: M x G_cov int32 view (row stride = ld) or None; G_cov."""
    C: torch.Tensor
    codes: torch.Tensor | None
    G_cov: int

    def to_c(self) -> _lib.crvq_codebook:
        _need(self.C, torch.float32, "codebook C")
        if not self.C.is_contiguous():
            raise ValueError("codebook C must be contiguous")
        ld = 0
        if self.codes is not None:
            _need(self.codes, torch.int32, "codes")
            _rowmajor(self.codes, "codes")
            ld = self.codes.stride(0) if self.codes.shape[0] > 1 else max(self.G_cov, 1)
        return _lib.crvq_codebook(self.C.data_ptr(), int(self.C.shape[0]), 0,
                                  None if self.codes is None else self.codes.data_ptr(),
                                  int(ld), int(self.G_cov))


def _cb_array(cbs):
    arr = (_lib.crvq_codebook * max(1, len(cbs)))()
    for i, cb in enumerate(cbs):
        arr[i] = cb.to_c()
    return arr


def crvq_version() -> str:
    return _L().crvq_version().decode()


def crvq_sync(stream=None, device=None):
    dev = device if device is not None else torch.cuda.current_device()
    _check(_L().crvq_sync(_stream(stream, dev)))


def crvq_selftest_bounded_wait(stream=None, device=None):
    """Enqueue the bounded-wait self-test: the next crvq_sync raises CRVQ_ERR_TIMEOUT."""
    dev = device if device is not None else torch.cuda.current_device()
    _check(_L().crvq_selftest_bounded_wait(_stream(stream, dev)))


def crvq_profile_begin():
    """Start bracketing every library kernel launch with CUDA events."""
    _check(_L().crvq_profile_begin())


def crvq_profile_filter(prefix=None):
    """Profile only kernels whose name starts with `prefix` (None: every kernel)."""
    _check(_L().crvq_profile_filter(None if not prefix else prefix.encode()))


def crvq_profile_end() -> list[dict]:
    """Stop profiling; per kernel name: launches, summed event ms, summed algorithmic units."""
    arr = (_lib.crvq_kernel_stat * 64)()
    n = C.c_int32(0)
    _check(_L().crvq_profile_end(arr, 64, C.byref(n)))
    return [dict(name=arr[i].name.decode(), launches=int(arr[i].launches), ms=arr[i].ms,
                 units=arr[i].units) for i in range(n.value)]


def crvq_launch_count() -> int:
    return int(_L().crvq_launch_count())


def crvq_avg_bits(e, d, m, lam, M=4096, N=4096, include_perm=False) -> float:
    return float(_L().crvq_avg_bits(e, d, m, lam, M, N, int(bool(include_perm))))


def crvq_avg_bits_bases(e, d, n_base, n_ext, lam, M=4096, N=4096, include_perm=False) -> float:
    return float(_L().crvq_avg_bits_bases(e, d, n_base, n_ext, lam, M, N,
                                          int(bool(include_perm))))


def crvq_n_crit_groups(N, d, crit_frac) -> int:
    return int(_L().crvq_n_crit_groups(N, d, crit_frac))


def crvq_hessian(X, damp_rel, d=8, H=None, xsq=None, H_blocks=None, delta=None, stream=None):
    """S1: returns (H, xsq, H_blocks in the original order, delta[1])."""
    _need(X, torch.float32, "X")
    X = X.contiguous()
    n, N = X.shape
    dev = X.device
    H = torch.empty((N, N), device=dev, dtype=torch.float32) if H is None else H
    xsq = torch.empty(N, device=dev, dtype=torch.float32) if xsq is None else xsq
    if H_blocks is None:
        H_blocks = torch.empty((N // d, d, d), device=dev, dtype=torch.float32)
    delta = torch.empty(1, device=dev, dtype=torch.float32) if delta is None else delta
    _check(_L().crvq_hessian(_ptr(X), n, N, d, float(damp_rel), _ptr(H), _ptr(xsq),
                             _ptr(H_blocks), _ptr(delta), _stream(stream, dev)))
    return H, xsq, H_blocks, delta


def crvq_hessian_blocks(X, damp_rel, d=8, perm=None, xsq=None, delta=None, H_blocks=None,
                        stream=None):
    """S1 / S3 blocks only: returns (H_blocks in the order perm (None: stored order), xsq,
    delta[1]) without forming the dense N x N H."""
    _need(X, torch.float32, "X")
    X = X.contiguous()
    n, N = X.shape
    dev = X.device
    if perm is not None:
        _need(perm, torch.int32, "perm")
    xsq = torch.empty(N, device=dev, dtype=torch.float32) if xsq is None else xsq
    delta = torch.empty(1, device=dev, dtype=torch.float32) if delta is None else delta
    if H_blocks is None:
        H_blocks = torch.empty((N // d, d, d), device=dev, dtype=torch.float32)
    _check(_L().crvq_hessian_blocks(_ptr(X), n, N, d, float(damp_rel),
                                    _ptr(perm), _ptr(xsq),
                                    _ptr(delta), _ptr(H_blocks), _stream(stream, dev)))
    return H_blocks, xsq, delta


def crvq_hessian_inverse_diag(H, hinv=None, stream=None):
    """[H^-1]_ii (fp64, length N) of a symmetric positive definite N x N H (device, fp32)."""
    _need(H, torch.float32, "H")
    H = H.contiguous()
    N = H.shape[0]
    hinv = torch.empty(N, device=H.device, dtype=torch.float64) if hinv is None else hinv
    _check(_L().crvq_hessian_inverse_diag(_ptr(H), N, _ptr(hinv), _stream(stream, H.device)))
    return hinv


def crvq_select_reorder_channels(W, d, W_pre, xsq, H, crit_frac, mode=IMPORTANCE_WA, seed=0,
                                 stream=None):
    """S3: returns (perm, importance, W_sorted, H_blocks, n_crit_groups)."""
    _need(W, torch.float32, "W")
    W = W.contiguous()
    M, N = W.shape
    dev = W.device
    perm = torch.empty(N, device=dev, dtype=torch.int32)
    imp = torch.empty(N, device=dev, dtype=torch.float32)
    Ws = torch.empty_like(W)
    Hb = torch.empty((N // d, d, d), device=dev, dtype=torch.float32)
    gc = C.c_int64(0)
    _check(_L().crvq_select_reorder_channels(
        _ptr(W), M, N, d, _ptr(None if W_pre is None else W_pre.contiguous()),
        _ptr(xsq), _ptr(H.contiguous()), float(crit_frac), int(mode), int(seed) & (2**64 - 1),
        _ptr(perm), _ptr(imp), _ptr(Ws), _ptr(Hb), C.byref(gc), _stream(stream, dev)))
    return perm, imp, Ws, Hb, int(gc.value)


def crvq_kmeans_init(T, d, G_sub, K, seed, fixed=(), C_out=None, stream=None):
    """Initial codebook of K codewords drawn from the vector set T (M x G_sub*d view)."""
    _need(T, torch.float32, "T")
    _rowmajor(T, "T")
    M = T.shape[0]
    dev = T.device
    C_out = torch.empty((K, d), device=dev, dtype=torch.float32) if C_out is None else C_out
    arr = _cb_array(fixed)
    _check(_L().crvq_kmeans_init(_ptr(T), T.stride(0), M, G_sub, d, arr, len(fixed), K,
                                 int(seed) & (2**64 - 1), _ptr(C_out), _stream(stream, dev)))
    return C_out


def crvq_encode_beam(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, vec_err=None,
                     want_err=False, stream=None):
    """Writes the codes of codebooks n_fixed.. of `cbs` in place; returns vec_err or None."""
    _need(T, torch.float32, "T")
    _rowmajor(T, "T")
    M = T.shape[0]
    G_sub = H_blocks.shape[0]
    dev = T.device
    if want_err and vec_err is None:
        vec_err = torch.empty((M, G_sub), device=dev, dtype=torch.float32)
    arr = _cb_array(cbs)
    _check(_L().crvq_encode_beam(_ptr(T), T.stride(0), M, G_sub, d, _ptr(H_blocks), arr,
                                 len(cbs), n_fixed, B, int(bool(keep_if_better)), _ptr(vec_err),
                                 _stream(stream, dev)))
    return vec_err


def crvq_update_codebook(T, d, H_blocks, cbs, which, C_out=None, counts=None, stream=None):
    """Returns (C_out, counts): the least-squares refit of codebook `which`."""
    _need(T, torch.float32, "T")
    _rowmajor(T, "T")
    M = T.shape[0]
    G_sub = H_blocks.shape[0]
    dev = T.device
    K = cbs[which].C.shape[0]
    C_out = torch.empty((K, d), device=dev, dtype=torch.float32) if C_out is None else C_out
    counts = torch.empty(K, device=dev, dtype=torch.int32) if counts is None else counts
    arr = _cb_array(cbs)
    _check(_L().crvq_update_codebook(_ptr(T), T.stride(0), M, G_sub, d, _ptr(H_blocks), arr,
                                     len(cbs), which, _ptr(C_out), _ptr(counts),
                                     _stream(stream, dev)))
    return C_out, counts


def crvq_update_codebook_noalloc(T, d, H_blocks, cbs, which, C_out=None, counts=None,
                                 stream=None):
    """crvq_update_codebook without device allocation inside the library: its scratch is a
    fixed 4 MiB device array (see include/crvq.h). Outputs not passed in are allocated here,
    by torch, before the call."""
    _need(T, torch.float32, "T")
    _rowmajor(T, "T")
    M = T.shape[0]
    G_sub = H_blocks.shape[0]
    dev = T.device
    K = cbs[which].C.shape[0]
    C_out = torch.empty((K, d), device=dev, dtype=torch.float32) if C_out is None else C_out
    counts = torch.empty(K, device=dev, dtype=torch.int32) if counts is None else counts
    arr = _cb_array(cbs)
    _check(_L().crvq_update_codebook_noalloc(_ptr(T), T.stride(0), M, G_sub, d, _ptr(H_blocks),
                                             arr, len(cbs), which, _ptr(C_out), _ptr(counts),
                                             _stream(stream, dev)))
    return C_out, counts


def crvq_coupled_sweep(W_sorted, H_sorted, cbs, which, sweeps=1, d=8, want_loss=True,
                       stream=None):
    """Gauss-Seidel sweeps of codebook `which` under the full loss (codes rewritten in place);
    returns the loss before and after each sweep (a list), or None. Synchronizes when the
    losses are requested."""
    _need(W_sorted, torch.float32, "W_sorted")
    _rowmajor(W_sorted, "W_sorted")
    _need(H_sorted, torch.float32, "H_sorted")
    M, N = W_sorted.shape
    arr = _cb_array(cbs)
    loss = (C.c_double * (sweeps + 1))() if want_loss else None
    _check(_L().crvq_coupled_sweep(_ptr(W_sorted), M, N, d, _ptr(H_sorted.contiguous()), arr,
                                   len(cbs), which, sweeps, loss,
                                   _stream(stream, W_sorted.device)))
    return list(loss) if want_loss else None


def crvq_lut_matvec(X_in, perm, cbs, M, d=8, Y=None, stream=None):
    """Y = X_in W_hat^T (b x M) from the codes of `cbs`, X_in b x N in the original channel
    order (a 1-D input is one row); perm None is the identity order."""
    _need(X_in, torch.float32, "X_in")
    X2 = X_in.unsqueeze(0) if X_in.dim() == 1 else X_in
    _rowmajor(X2, "X_in")
    b, N = X2.shape
    dev = X2.device
    Y = torch.empty((b, M), device=dev, dtype=torch.float32) if Y is None else Y
    arr = _cb_array(cbs)
    _check(_L().crvq_lut_matvec(_ptr(X2), X2.stride(0), b, N, d, _ptr(perm), arr, len(cbs), M,
                                _ptr(Y), Y.stride(0), _stream(stream, dev)))
    return Y


def crvq_reconstruct_error(W_sorted, d, H_blocks, perm, cbs, n_crit_groups, X=None,
                           damp_delta=0.0, want_W_hat=True, stream=None):
    """Returns (W_hat or None, loss_block, loss_crit, loss_full). Synchronizes the stream."""
    _need(W_sorted, torch.float32, "W_sorted")
    W_sorted = W_sorted.contiguous()
    M, N = W_sorted.shape
    dev = W_sorted.device
    W_hat = torch.empty_like(W_sorted) if want_W_hat else None
    losses = (C.c_double * 3)()
    arr = _cb_array(cbs)
    Xc = None if X is None else X.contiguous()
    _check(_L().crvq_reconstruct_error(_ptr(W_sorted), M, N, d, _ptr(H_blocks), _ptr(perm), arr,
                                       len(cbs), int(n_crit_groups), _ptr(Xc),
                                       0 if Xc is None else Xc.shape[0], float(damp_delta),
                                       _ptr(W_hat), C.cast(losses, _lib.c_f64p),
                                       _stream(stream, dev)))
    return W_hat, losses[0], losses[1], (None if X is None else losses[2])


@dataclass
class LayerOutputs:
    perm: object
    C_base: object
    codes_base: object
    C_ext: object
    codes_ext: object
    W_hat: object
    importance: object
    report: dict


def _cfg_struct(cfg) -> _lib.crvq_config:
    return _lib.crvq_config(cfg.d, cfg.K_base, cfg.n_ext, cfg.K_ext, cfg.crit_frac, cfg.B,
                            cfg.kmeans_iters, cfg.refine_rounds, cfg.eps_rel, cfg.damp_rel,
                            cfg.importance_mode, getattr(cfg, "n_base", 1),
                            int(cfg.seed) & (2**64 - 1))


def crvq_quantize_layer(W, X, cfg, want_W_hat=True, out=None, stream=None, device=None):
    """Alg. 1, prequantization through the refinement loop, for one matrix. W, X: torch
    tensors on the GPU, or pinned/pageable CPU tensors (then the library stages them and the
    outputs are CPU tensors). With cfg.n_base > 1 base codebooks, C_base and codes_base gain a
    leading axis of that length."""
    M, N = W.shape
    n_tok = X.shape[0]
    d = cfg.d
    G = N // d
    Gc = crvq_n_crit_groups(N, d, cfg.crit_frac)
    on_dev = W.device.type == "cuda"
    dev = W.device if on_dev else torch.device("cpu")
    pin = (not on_dev) and W.is_pinned()

    def alloc(shape, dtype):
        return torch.empty(shape, dtype=dtype, device=dev, pin_memory=pin)

    n_base = getattr(cfg, "n_base", 1)
    lead = (n_base,) if n_base > 1 else ()

    if out is None:
        out = LayerOutputs(
            perm=alloc((N,), torch.int32), C_base=alloc(lead + (cfg.K_base, d), torch.float32),
            codes_base=alloc(lead + (M, G), torch.int32),
            C_ext=alloc((max(cfg.n_ext, 0), cfg.K_ext, d), torch.float32),
            codes_ext=alloc((max(cfg.n_ext, 0), M, Gc), torch.int32),
            W_hat=alloc((M, N), torch.float32) if want_W_hat else None,
            importance=alloc((N,), torch.float32), report={})
    o = _lib.crvq_layer_outputs(out.perm.data_ptr(), out.C_base.data_ptr(),
                                out.codes_base.data_ptr(),
                                out.C_ext.data_ptr() if cfg.n_ext else None,
                                out.codes_ext.data_ptr() if cfg.n_ext else None,
                                None if out.W_hat is None else out.W_hat.data_ptr(),
                                out.importance.data_ptr())
    rep = _lib.crvq_layer_report()
    c = _cfg_struct(cfg)
    cuda_dev = W.device if on_dev else (device if device is not None else
                                        torch.device("cuda", torch.cuda.current_device()))
    Wc = W if W.is_contiguous() else W.contiguous()
    Xc = X if X.is_contiguous() else X.contiguous()
    _check(_L().crvq_quantize_layer(_ptr(Wc), _ptr(Xc), M, N, n_tok, C.byref(c), C.byref(o),
                                    C.byref(rep), _stream(stream, cuda_dev)))
    out.report = {f: getattr(rep, f) for f, _ in _lib.crvq_layer_report._fields_ if f != "_pad"}
    return out
