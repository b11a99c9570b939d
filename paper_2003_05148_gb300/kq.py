"""Thin Python binding of libkq (include/kq.h): argument marshalling only.

Each function has the name of the C entry point it calls, takes CUDA tensors
(PyTorch supplies device memory and the current stream) and passes their device
pointers through ctypes. Every step of the computation runs in libkq's CUDA
kernels; there is no CPU path, and loading fails loudly when libkq.so has not
been built.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from .build import LIB

KQ_OK = 0
STATUS_NAMES = {0: "KQ_OK", 1: "KQ_ERR_INVALID_ARG", 2: "KQ_ERR_ALIGNMENT", 3: "KQ_ERR_NONFINITE",
                4: "KQ_ERR_CUDA", 5: "KQ_ERR_DEVICE_CHECK", 6: "KQ_ERR_WORKSPACE", 7: "KQ_ERR_TIMEOUT"}
FLAG_NONFINITE, FLAG_INDEX_RANGE, FLAG_CODE_RANGE, FLAG_TIMEOUT = 0x1, 0x2, 0x4, 0x8
STOP_ON_STABLE, FIT_PRUNE = 0x1, 0x2  # kq_fit_codebook flags
TEST_SKIP_ARRIVAL, TEST_STOP_TILE_STREAM = 0x1, 0x2  # kq_test_inject_wait_fault faults

EXPORTS = ["kq_status_string", "kq_abi_version", "kq_kernel_launches", "kq_workspace_bytes", "kq_device_status", "kq_init_codebook",
           "kq_assign", "kq_update_centroids", "kq_fit_codebook", "kq_quantize_codebook_6bit", "kq_reconstruct",
           "kq_compression_report", "kq_conventional_ratio", "kq_assign_noalloc", "kq_quantize_scalars_6bit",
           "kq_codebook_grad_step", "kq_levels_grad_step", "kq_search_codebook_size", "kq_quantize_reconstruct",
           "kq_seed_indices", "kq_trace_start", "kq_trace_stop", "kq_trace_count", "kq_trace_get",
           "kq_test_inject_wait_fault", "kq_fit_layers", "kq_fit_prune_stats"]


class KQError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)}")


class LayerJob(ctypes.Structure):
    """kq_layer_job (include/kq.h): one layer of kq_fit_layers."""
    _fields_ = [("W", ctypes.c_void_p), ("n", ctypes.c_int64), ("K", ctypes.c_int32), ("sel", ctypes.c_void_p),
                ("C", ctypes.c_void_p), ("idx", ctypes.c_void_p), ("counts", ctypes.c_void_p),
                ("objective", ctypes.c_void_p), ("levels", ctypes.c_void_p), ("codes", ctypes.c_void_p),
                ("W_out", ctypes.c_void_p), ("ws", ctypes.c_void_p), ("ws_bytes", ctypes.c_size_t)]


class Report(ctypes.Structure):
    _fields_ = [("index_bits", ctypes.c_int64), ("codebook_bits", ctypes.c_int64), ("total_bits", ctypes.c_int64),
                ("beta", ctypes.c_double), ("ratio_kq", ctypes.c_double), ("ratio_con_1bit", ctypes.c_double)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libkq.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"libkq.so is not built ({LIB}); run paper_2003_05148_gb300.build.build()")
        L = ctypes.CDLL(LIB)
        P, i64, i32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_size_t
        sig = {
            "kq_status_string": ([ctypes.c_int], ctypes.c_char_p),
            "kq_abi_version": ([], i32),
            "kq_kernel_launches": ([], ctypes.c_uint64),
            "kq_trace_start": ([i32], ctypes.c_int),
            "kq_trace_stop": ([], ctypes.c_int),
            "kq_trace_count": ([], i32),
            "kq_test_inject_wait_fault": ([P, sz, ctypes.c_uint32, ctypes.c_uint32, P], ctypes.c_int),
            "kq_trace_get": ([i32, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_float)], ctypes.c_int),
            "kq_workspace_bytes": ([i64, i32], sz),
            "kq_device_status": ([P, sz, P, P], ctypes.c_int),
            "kq_fit_prune_stats": ([P, sz, P, P, P], ctypes.c_int),
            "kq_init_codebook": ([P, i64, P, i32, P, P, sz, P], ctypes.c_int),
            "kq_assign": ([P, i64, P, i32, P, P, P, P, sz, P], ctypes.c_int),
            "kq_update_centroids": ([P, i64, P, i32, P, P, P, P, sz, P], ctypes.c_int),
            "kq_fit_codebook": ([P, i64, i32, P, i32, i32, P, P, P, P, P, P, sz, P], ctypes.c_int),
            "kq_quantize_codebook_6bit": ([P, i32, P, i32, P, P, P, P, sz, P], ctypes.c_int),
            "kq_reconstruct": ([P, i64, P, i32, P, P, P, P, sz, P], ctypes.c_int),
            "kq_compression_report": ([i64, i32, i32, i32, ctypes.POINTER(Report)], ctypes.c_int),
            "kq_seed_indices": ([i64, i32, ctypes.c_uint64, P], ctypes.c_int),
            "kq_conventional_ratio": ([i64, i32, i32, i32, i32, ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
            "kq_assign_noalloc": ([P, i64, P, i32, P, P, P], ctypes.c_int),
            "kq_quantize_scalars_6bit": ([P, i64, i32, P, P, P, P, sz, P], ctypes.c_int),
            "kq_codebook_grad_step": ([P, i64, P, i32, ctypes.c_float, P, P, P, P, sz, P], ctypes.c_int),
            "kq_levels_grad_step": ([P, i64, P, i32, P, ctypes.c_float, P, P, P, P, sz, P], ctypes.c_int),
            "kq_quantize_reconstruct": ([P, i64, P, i32, P, P, P, P, sz, P], ctypes.c_int),
            "kq_search_codebook_size": ([P, i64, P, i32, ctypes.c_double, ctypes.c_double, i32, i32, P, P, P,
                                         P, P, P, P, P, P, sz, P], ctypes.c_int),
            "kq_fit_layers": ([ctypes.POINTER(LayerJob), i32, i32, i32, i32, P], ctypes.c_int),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _check(fn: str, status: int) -> None:
    if status != KQ_OK:
        raise KQError(fn, status)


def _dev(t: Optional[torch.Tensor], name: str, dtype: torch.dtype):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or t.device.type != "cuda":
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must have dtype {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


class _Call:
    """Marshalling for one call of an entry point that takes device memory: every
    tensor must live on one CUDA device; the call runs with that device current
    (the library reads the current device for its SM count and launches there) and
    on that device's current stream unless a stream of the same device is given."""

    def __init__(self, fn: str):
        self.fn = fn
        self.device = None

    def ptr(self, t: Optional[torch.Tensor], name: str, dtype: torch.dtype):
        p = _dev(t, name, dtype)
        if t is not None:
            if self.device is None:
                self.device = t.device
            elif t.device != self.device:
                raise ValueError(f"{self.fn}: {name} is on {t.device}, other arguments on {self.device}")
        return p

    def stream(self, stream) -> ctypes.c_void_p:
        if self.device is None:
            raise ValueError(f"{self.fn}: no device tensor given")
        s = torch.cuda.current_stream(self.device) if stream is None else stream
        if s.device != self.device:
            raise ValueError(f"{self.fn}: the stream is on {s.device}, the tensors on {self.device}")
        return ctypes.c_void_p(s.cuda_stream)

    def __call__(self, *args) -> None:
        with torch.cuda.device(self.device):
            _check(self.fn, getattr(lib(), self.fn)(*args))


def _rows(W: torch.Tensor) -> int:
    if W.numel() % 9:
        raise ValueError("kernel tensors must hold a multiple of 9 floats (3x3 kernels)")
    return W.numel() // 9


def kq_status_string(status: int) -> str:
    return lib().kq_status_string(status).decode()


def kq_abi_version() -> int:
    return lib().kq_abi_version()


def kq_kernel_launches() -> int:
    return int(lib().kq_kernel_launches())


def kq_trace_start(capacity: int) -> None:
    """Start a kernel trace of up to `capacity` launches (events on the current device)."""
    _check("kq_trace_start", lib().kq_trace_start(capacity))


def kq_trace_stop() -> None:
    _check("kq_trace_stop", lib().kq_trace_stop())


def kq_trace_read() -> list:
    """[(kernel name, device ms)] of every launch the current trace recorded, in launch order."""
    out = []
    name = ctypes.c_char_p()
    ms = ctypes.c_float()
    for i in range(lib().kq_trace_count()):
        _check("kq_trace_get", lib().kq_trace_get(i, ctypes.byref(name), ctypes.byref(ms)))
        out.append((name.value.decode(), ms.value))
    return out


def kq_workspace_bytes(n: int, K: int) -> int:
    return int(lib().kq_workspace_bytes(n, K))


def workspace(n: int, K: int, device=None) -> torch.Tensor:
    """Zero-filled workspace of kq_workspace_bytes(n, K) bytes on the device."""
    nbytes = kq_workspace_bytes(n, K)
    if nbytes == 0:
        raise ValueError(f"unsupported sizes n={n}, K={K}")
    return torch.zeros(nbytes, dtype=torch.uint8, device=device or "cuda")


def kq_device_status(ws: torch.Tensor, stream=None):
    """(status, flags): read and clear the sticky device status word (synchronises the stream)."""
    flags = ctypes.c_uint32(0)
    c = _Call("kq_device_status")
    ptr = c.ptr(ws, "ws", torch.uint8)
    with torch.cuda.device(c.device):
        st = lib().kq_device_status(ptr, ws.numel(), c.stream(stream), ctypes.byref(flags))
    return st, flags.value


def kq_fit_prune_stats(ws, stream=None):
    """(tiles_run, tiles_all): the (block, tile) pairs the last pruned fit on `ws` processed,
    and those its assignments hold in all (synchronises the stream)."""
    run, total = ctypes.c_uint64(0), ctypes.c_uint64(0)
    c = _Call("kq_fit_prune_stats")
    c(c.ptr(ws, "ws", torch.uint8), ws.numel(), ctypes.byref(run), ctypes.byref(total), c.stream(stream))
    return run.value, total.value


def kq_test_inject_wait_fault(ws, faults: int, wait_limit: int, stream=None) -> None:
    """Failure-detection test hook: later calls on `ws` meet bounded waits that run out."""
    c = _Call("kq_test_inject_wait_fault")
    c(c.ptr(ws, "ws", torch.uint8), ws.numel(), faults, wait_limit, c.stream(stream))


def kq_init_codebook(W, sel, C0, ws, stream=None) -> None:
    c = _Call("kq_init_codebook")
    c(
        c.ptr(W, "W", torch.float32), _rows(W), c.ptr(sel, "sel", torch.int64), sel.numel(),
        c.ptr(C0, "C0", torch.float32), c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_assign(W, C, idx, dist, ws, hint=None, stream=None) -> None:
    c = _Call("kq_assign")
    c(
        c.ptr(W, "W", torch.float32), _rows(W), c.ptr(C, "C", torch.float32), _rows(C),
        c.ptr(hint, "hint", torch.int32), c.ptr(idx, "idx", torch.int32), c.ptr(dist, "dist", torch.float32),
        c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_update_centroids(W, idx, C_prev, C_next, counts, ws, stream=None) -> None:
    c = _Call("kq_update_centroids")
    c(
        c.ptr(W, "W", torch.float32), _rows(W), c.ptr(idx, "idx", torch.int32), _rows(C_prev),
        c.ptr(C_prev, "C_prev", torch.float32), c.ptr(C_next, "C_next", torch.float32),
        c.ptr(counts, "counts", torch.int32), c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_fit_codebook(W, C_init, iters, C_out, idx, counts, objective, ws, stream=None, flags: int = 0) -> int:
    """Returns the number of codebook updates performed (iters unless STOP_ON_STABLE stopped early)."""
    run = ctypes.c_int32(0)
    c = _Call("kq_fit_codebook")
    c(
        c.ptr(W, "W", torch.float32), _rows(W), _rows(C_init), c.ptr(C_init, "C_init", torch.float32), iters, flags,
        c.ptr(C_out, "C_out", torch.float32), c.ptr(idx, "idx", torch.int32), c.ptr(counts, "counts", torch.int32),
        c.ptr(objective, "objective", torch.float64), ctypes.byref(run), c.ptr(ws, "ws", torch.uint8), ws.numel(),
        c.stream(stream))
    return run.value


def kq_fit_layers(jobs, iters: int, level_iters: int = 100, flags: int = 0, stream=None) -> None:
    """All layers of a network in one call (kq_layer_job per layer). Each job is a
    dict with tensors W, C, idx, counts, ws and optionally sel, objective, levels,
    codes, W_out (absent or None: not given); all on one device."""
    c = _Call("kq_fit_layers")
    arr = (LayerJob * len(jobs))()
    for i, j in enumerate(jobs):
        g = j.get
        arr[i] = LayerJob(
            c.ptr(j["W"], "W", torch.float32), _rows(j["W"]), _rows(j["C"]), c.ptr(g("sel"), "sel", torch.int64),
            c.ptr(j["C"], "C", torch.float32), c.ptr(j["idx"], "idx", torch.int32),
            c.ptr(j["counts"], "counts", torch.int32), c.ptr(g("objective"), "objective", torch.float64),
            c.ptr(g("levels"), "levels", torch.float32), c.ptr(g("codes"), "codes", torch.uint8),
            c.ptr(g("W_out"), "W_out", torch.float32), c.ptr(j["ws"], "ws", torch.uint8), j["ws"].numel())
    c(arr, len(jobs), iters, level_iters, flags, c.stream(stream))


def kq_quantize_codebook_6bit(C, counts, max_iters, levels, codes, iters_run, ws, stream=None) -> None:
    c = _Call("kq_quantize_codebook_6bit")
    c(
        c.ptr(C, "C", torch.float32), _rows(C), c.ptr(counts, "counts", torch.int32), max_iters,
        c.ptr(levels, "levels", torch.float32), c.ptr(codes, "codes", torch.uint8),
        c.ptr(iters_run, "iters_run", torch.int32), c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_quantize_scalars_6bit(v, max_iters, levels, codes, iters_run, ws, stream=None) -> None:
    c = _Call("kq_quantize_scalars_6bit")
    c(
        c.ptr(v, "v", torch.float32), v.numel(), max_iters, c.ptr(levels, "levels", torch.float32),
        c.ptr(codes, "codes", torch.uint8), c.ptr(iters_run, "iters_run", torch.int32), c.ptr(ws, "ws", torch.uint8),
        ws.numel(), c.stream(stream))


def kq_codebook_grad_step(G, idx, lr: float, C, C_next, counts, ws, stream=None) -> None:
    c = _Call("kq_codebook_grad_step")
    c(
        c.ptr(G, "G", torch.float32), _rows(G), c.ptr(idx, "idx", torch.int32), _rows(C), float(lr),
        c.ptr(C, "C", torch.float32), c.ptr(C_next, "C_next", torch.float32), c.ptr(counts, "counts", torch.int32),
        c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_levels_grad_step(G, idx, codes, lr: float, levels, levels_next, counts, ws, stream=None) -> None:
    c = _Call("kq_levels_grad_step")
    c(
        c.ptr(G, "G", torch.float32), _rows(G), c.ptr(idx, "idx", torch.int32), codes.numel() // 9,
        c.ptr(codes, "codes", torch.uint8), float(lr), c.ptr(levels, "levels", torch.float32),
        c.ptr(levels_next, "levels_next", torch.float32), c.ptr(counts, "counts", torch.int64),
        c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_search_codebook_size(W, sel, alpha: float, r: float, max_steps: int, lloyd_iters: int, C_out, idx, counts,
                            ws, stream=None):
    """Returns (K, e(K), trace [(size, e)]); C_out / idx / counts hold the fit of size K."""
    k = ctypes.c_int32(0)
    err = ctypes.c_double(0.0)
    steps = ctypes.c_int32(0)
    tK = (ctypes.c_int32 * (max_steps + 1))()
    tE = (ctypes.c_double * (max_steps + 1))()
    c = _Call("kq_search_codebook_size")
    c(
        c.ptr(W, "W", torch.float32), _rows(W), c.ptr(sel, "sel", torch.int64), sel.numel(), float(alpha), float(r),
        max_steps, lloyd_iters, c.ptr(C_out, "C_out", torch.float32), c.ptr(idx, "idx", torch.int32),
        c.ptr(counts, "counts", torch.int32), ctypes.byref(k), ctypes.byref(err), tK, tE, ctypes.byref(steps),
        c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))
    return k.value, err.value, [(tK[i], tE[i]) for i in range(steps.value + 1)]


def kq_quantize_reconstruct(idx, C, levels, codes, W_out, ws, stream=None) -> None:
    c = _Call("kq_quantize_reconstruct")
    c(
        c.ptr(idx, "idx", torch.int32), idx.numel(), c.ptr(C, "C", torch.float32), _rows(C),
        c.ptr(levels, "levels", torch.float32), c.ptr(codes, "codes", torch.uint8), c.ptr(W_out, "W_out", torch.float32),
        c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_reconstruct(idx, C, codes, levels, W_out, ws, K: Optional[int] = None, stream=None) -> None:
    K = _rows(C) if C is not None else codes.numel() // 9 if K is None else K
    c = _Call("kq_reconstruct")
    c(
        c.ptr(idx, "idx", torch.int32), idx.numel(), c.ptr(C, "C", torch.float32), K,
        c.ptr(codes, "codes", torch.uint8), c.ptr(levels, "levels", torch.float32),
        c.ptr(W_out, "W_out", torch.float32), c.ptr(ws, "ws", torch.uint8), ws.numel(), c.stream(stream))


def kq_compression_report(n: int, k: int, omega: int = 3, b_c: int = 32) -> dict:
    r = Report()
    _check("kq_compression_report", lib().kq_compression_report(n, k, omega, b_c, ctypes.byref(r)))
    return {f: getattr(r, f) for f, _ in Report._fields_}


def kq_seed_indices(n: int, K: int, seed: int) -> torch.Tensor:
    """K distinct row numbers in [0, n) (int64, host): the seeded draw that initialises a codebook."""
    out = torch.empty(K, dtype=torch.int64)
    _check("kq_seed_indices", lib().kq_seed_indices(n, K, seed & 0xFFFFFFFFFFFFFFFF, out.data_ptr()))
    return out


def kq_conventional_ratio(n: int, omega: int, u: int, b_1: int, b_fp: int = 32) -> float:
    out = ctypes.c_double(0.0)
    _check("kq_conventional_ratio", lib().kq_conventional_ratio(n, omega, u, b_1, b_fp, ctypes.byref(out)))
    return out.value


def kq_assign_noalloc(W, C, idx, dist, stream=None) -> None:
    """kq_assign without a workspace, for callers that cannot allocate device memory."""
    c = _Call("kq_assign_noalloc")
    c(
        c.ptr(W, "W", torch.float32), _rows(W), c.ptr(C, "C", torch.float32), _rows(C),
        c.ptr(idx, "idx", torch.int32), c.ptr(dist, "dist", torch.float32), c.stream(stream))
