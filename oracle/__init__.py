"""CPU oracle for the Kernel Quantization hot path (arXiv 2003.05148).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` are the only callers. The CUDA library never imports,
links or runs anything here, and nothing here imports the CUDA library.

The compute-heavy steps live in ``kq_oracle.c`` (plain C, built with
``-ffp-contract=off`` so that only the ``fmaf`` calls written in the source fuse);
this module loads it with ctypes and adds the storage accounting of Eq. 4-7,
which is exact integer / rational arithmetic done here in Python.

Parity pins for every function are in ``tests/test_oracle.py``.
"""
from __future__ import annotations

import ctypes
import math
import dataclasses
import os
import subprocess
from fractions import Fraction
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libkq_oracle.so")
_CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-pthread"]

D = 9
LEVELS = 64


def build(force: bool = False) -> str:
    """Compile kq_oracle.c into oracle/_build/libkq_oracle.so (gcc)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        compile_library(_SRC, tmp)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def _bind(lib):
    """Declare the C signatures on a loaded oracle library and return it."""
    if True:
        P = ctypes.c_void_p
        i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        lib.kqo_assign.argtypes = [P, i64, P, i32, P, P, P, P, i32]
        lib.kqo_assign.restype = None
        lib.kqo_update.argtypes = [P, i64, P, i32, P, P, P]
        lib.kqo_update.restype = None
        lib.kqo_objective.argtypes = [P, i64]
        lib.kqo_objective.restype = f64
        lib.kqo_fit.argtypes = [P, i64, i32, P, i32, P, P, P, P, i32]
        lib.kqo_fit.restype = i32
        lib.kqo_level_scale.argtypes = [P, i32, P]
        lib.kqo_level_scale.restype = i32
        lib.kqo_level_fit.argtypes = [P, i32, P, i32, P, P]
        lib.kqo_level_fit.restype = i32
        lib.kqo_reconstruct.argtypes = [P, i64, P, P, P, P]
        lib.kqo_reconstruct.restype = None
        lib.kqo_encode.argtypes = [P, i64, P, P]
        lib.kqo_encode.restype = None
        lib.kqo_gather_rows.argtypes = [P, P, i32, P]
        lib.kqo_gather_rows.restype = None
        lib.kqo_level_fit_scalars.argtypes = [P, i64, i32, P, P]
        lib.kqo_level_fit_scalars.restype = i32
        lib.kqo_codebook_grad_step.argtypes = [P, i64, P, i32, ctypes.c_float, P, P, P]
        lib.kqo_codebook_grad_step.restype = None
        lib.kqo_levels_grad_step.argtypes = [P, i64, P, i32, P, ctypes.c_float, P, P, P]
        lib.kqo_levels_grad_step.restype = None
    return lib


def compile_library(src: str, out: str) -> str:
    """Compile an oracle C source (this one, or a test's modified copy) to `out`."""
    subprocess.run(["gcc", *_CFLAGS, src, "-o", out, "-lm"], check=True)
    return out


def _load():
    global _lib
    if _lib is None:
        _lib = _bind(ctypes.CDLL(build()))
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def default_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:  # pragma: no cover
        return max(1, os.cpu_count() or 1)


def assign(W, C, threads: int = 1, gap: bool = False):
    """Eq. 1 assignment (Sec. 3.1). Returns (idx int32, dist fp32[, d1, d2 fp64]).

    idx_i = argmin_k d(W_i, C_k) with the fp32 direct-form distance and the
    lowest index on ties. With ``gap`` also the fp64 best and second-best
    distances of every row, for judging how close each decision was.
    """
    W, C = _f32(W).reshape(-1, D), _f32(C).reshape(-1, D)
    n, K = W.shape[0], C.shape[0]
    idx = np.empty(n, np.int32)
    dist = np.empty(n, np.float32)
    d1 = np.empty(n, np.float64) if gap else None
    d2 = np.empty(n, np.float64) if gap else None
    _load().kqo_assign(_ptr(W), n, _ptr(C), K, _ptr(idx), _ptr(dist), _ptr(d1), _ptr(d2), threads)
    return (idx, dist, d1, d2) if gap else (idx, dist)


def update(W, idx, C_prev):
    """Eq. 1 centroid step (Sec. 3.1): (C_next fp32 (K, 9), counts int32 (K,))."""
    W, C_prev, idx = _f32(W).reshape(-1, D), _f32(C_prev).reshape(-1, D), _i32(idx)
    K = C_prev.shape[0]
    C_next = np.empty_like(C_prev)
    counts = np.empty(K, np.int32)
    _load().kqo_update(_ptr(W), W.shape[0], _ptr(idx), K, _ptr(C_prev), _ptr(C_next), _ptr(counts))
    return C_next, counts


def objective(dist) -> float:
    """Eq. 1 objective: fp64 sum of per-kernel distances in ascending order."""
    dist = _f32(dist)
    return float(_load().kqo_objective(_ptr(dist), dist.shape[0]))


def fit(W, C_init, iters: int, threads: int = 1):
    """k-means of Eq. 1 for a fixed number of iterations.

    Returns (C_T, idx_T, counts_T, objective[0..T]).
    """
    W, C0 = _f32(W).reshape(-1, D), _f32(C_init).reshape(-1, D)
    n, K = W.shape[0], C0.shape[0]
    C = np.empty_like(C0)
    idx = np.empty(n, np.int32)
    counts = np.empty(K, np.int32)
    obj = np.empty(iters + 1, np.float64)
    _load().kqo_fit(_ptr(W), n, K, _ptr(C0), iters, _ptr(C), _ptr(idx), _ptr(counts), _ptr(obj), threads)
    return C, idx, counts, obj


def level_scale(C, counts) -> int:
    """Exponent S of the fixed-point scale 2^S used for the exact level sums."""
    C, counts = _f32(C).reshape(-1, D), _i32(counts)
    return int(_load().kqo_level_scale(_ptr(C), C.shape[0], _ptr(counts)))


def level_fit(C, counts, max_iters: int = 100):
    """Sec. 3.2 6-bit codebook quantisation: (levels fp32 (64,), codes uint8 (K, 9), updates)."""
    C, counts = _f32(C).reshape(-1, D), _i32(counts)
    K = C.shape[0]
    levels = np.empty(LEVELS, np.float32)
    codes = np.empty((K, D), np.uint8)
    it = _load().kqo_level_fit(_ptr(C), K, _ptr(counts), max_iters, _ptr(levels), _ptr(codes))
    return levels, codes, int(it)


def level_fit_scalars(values, max_iters: int = 100):
    """Sec. 3.2 6-bit quantisation of a fully-connected layer (every scalar weighted 1).

    Returns (levels fp32 (64,), codes uint8 (m,), updates)."""
    v = _f32(values).reshape(-1)
    levels = np.empty(LEVELS, np.float32)
    codes = np.empty(v.shape[0], np.uint8)
    it = _load().kqo_level_fit_scalars(_ptr(v), v.shape[0], max_iters, _ptr(levels), _ptr(codes))
    return levels, codes, int(it)


def codebook_grad_step(G, idx, C, lr: float):
    """Eq. 2 (Sec. 3.1): c_k - lr * mean of the gradients of S_k. Returns (C_next, counts)."""
    G, C, idx = _f32(G).reshape(-1, D), _f32(C).reshape(-1, D), _i32(idx)
    K = C.shape[0]
    C_next = np.empty_like(C)
    counts = np.empty(K, np.int32)
    _load().kqo_codebook_grad_step(_ptr(G), G.shape[0], _ptr(idx), K, float(lr), _ptr(C), _ptr(C_next), _ptr(counts))
    return C_next, counts


def levels_grad_step(G, idx, codes, levels, lr: float):
    """Sec. 3.2 retraining of the 6-bit levels with averaged gradients.

    Returns (levels_next fp32 (64,), counts int64 (64,))."""
    G, idx, levels = _f32(G).reshape(-1, D), _i32(idx), _f32(levels)
    codes = np.ascontiguousarray(codes, dtype=np.uint8).reshape(-1, D)
    nxt = np.empty(LEVELS, np.float32)
    counts = np.empty(LEVELS, np.int64)
    _load().kqo_levels_grad_step(_ptr(G), G.shape[0], _ptr(idx), codes.shape[0], _ptr(codes), float(lr),
                                 _ptr(levels), _ptr(nxt), _ptr(counts))
    return nxt, counts


def encode(values, levels):
    """Sec. 3.2 encode: nearest of the 64 levels by fp32 |v - level|, lower index on ties."""
    v, levels = _f32(values).reshape(-1), _f32(levels)
    codes = np.empty(v.shape[0], np.uint8)
    _load().kqo_encode(_ptr(v), v.shape[0], _ptr(levels), _ptr(codes))
    return codes


def reconstruct(idx, C, codes=None, levels=None):
    """Sec. 3.2 testing phase: W' (n, 9) from kernel indices and the (decoded) codebook."""
    idx, C = _i32(idx), _f32(C).reshape(-1, D)
    out = np.empty((idx.shape[0], D), np.float32)
    if codes is not None:
        codes = np.ascontiguousarray(codes, dtype=np.uint8).reshape(-1, D)
        levels = _f32(levels)
    _load().kqo_reconstruct(_ptr(idx), idx.shape[0], _ptr(C), _ptr(codes), _ptr(levels), _ptr(out))
    return out


def gather_rows(W, sel):
    """Codeword initialisation: C_0[j] = W[sel[j]] (every sel[j] a row of W)."""
    W = _f32(W).reshape(-1, D)
    sel = np.ascontiguousarray(sel, dtype=np.int64)
    if sel.size and (sel.min() < 0 or sel.max() >= W.shape[0]):
        raise ValueError(f"row index outside [0, {W.shape[0]})")
    C0 = np.empty((sel.shape[0], D), np.float32)
    _load().kqo_gather_rows(_ptr(W), _ptr(sel), sel.shape[0], _ptr(C0))
    return C0


# ---------------------------------------------------------------------------
# Algorithm 1 (Sec. 3.1): adaptive codebook size by binary search, Eq. 3.
# ---------------------------------------------------------------------------

def initial_size(n: int, alpha: float) -> int:
    """N_init = alpha * n (Algorithm 1), rounded down and kept in [1, n]."""
    return max(1, min(n, int(math.floor(alpha * n))))


def target_accuracy(a_ori: float, a_base: float, r: float) -> float:
    """Eq. 3: A_target = A_base - (A_ori - A_base) * r."""
    return a_base - (a_ori - a_base) * r


def bisect_codebook_size(n: int, alpha: float, r: float, max_steps: int, accuracy_of, a_ori: float):
    """Algorithm 1's search for one layer, with the accuracy test supplied by the caller.

    accuracy_of(K) quantises the layer with K entries and returns its accuracy.
    B_upper starts at N_init, B_lower at 0; each step tests N_curr = floor((B_upper +
    B_lower) / 2) and moves B_upper there if the accuracy beats A_target (Eq. 3),
    else B_lower. The search stops after max_steps tests, when the interval cannot
    be split any more, or when a test lands exactly on A_target. Returns
    (K, trace): K = B_upper, the smallest tested size that beats the target (N_init
    when none does), and trace = [(size, accuracy)] starting with (N_init, A_base).
    """
    n_init = initial_size(n, alpha)
    a_base = accuracy_of(n_init)
    a_target = target_accuracy(a_ori, a_base, r)
    b_up, b_lo = n_init, 0
    trace = [(n_init, a_base)]
    steps = 0
    while steps < max_steps and b_up - b_lo > 1:
        steps += 1
        k = (b_up + b_lo) // 2
        a = accuracy_of(k)
        trace.append((k, a))
        if a > a_target:
            b_up = k
        else:
            b_lo = k
        if a == a_target:
            break
    return b_up, trace


def search_codebook_size(W, sel, alpha: float, r: float, max_steps: int, lloyd_iters: int, threads: int = 1):
    """Algorithm 1 with the reconstruction-error proxy: accuracy A(K) = -e(K), where
    e(K) = sqrt(J_K / J_0) is the relative l2 error of kernel-level quantisation with K
    entries (J_K: Eq. 1 objective after `lloyd_iters` updates from C_0 = W[sel[:K]];
    J_0 = sum of |W_i|^2, the objective against the zero codeword) and A_ori = 0.

    Returns (K, trace [(size, error)])."""
    W = _f32(W).reshape(-1, D)
    sel = np.ascontiguousarray(sel, dtype=np.int64)
    n = W.shape[0]
    _, d0 = assign(W, np.zeros((1, D), np.float32), threads=threads)
    J0 = objective(d0)

    def accuracy_of(k):
        _, _, _, obj = fit(W, gather_rows(W, sel[:k]), lloyd_iters, threads=threads)
        return -math.sqrt(obj[-1] / J0) if J0 > 0 else 0.0

    k, trace = bisect_codebook_size(n, alpha, r, max_steps, accuracy_of, 0.0)
    return k, [(size, -a) for size, a in trace]


# ---------------------------------------------------------------------------
# Storage accounting, Sec. 3.2-3.3 and Sec. 4.1 (Eq. 4-7). Exact arithmetic.
# ---------------------------------------------------------------------------

def ceil_log2(k: int) -> int:
    """ceil(log2 k) for an integer k >= 1, by integer bit length (k = 1 -> 0)."""
    if k < 1:
        raise ValueError("codebook size must be >= 1")
    return (k - 1).bit_length()


@dataclasses.dataclass(frozen=True)
class Report:
    index_bits: int
    codebook_bits: int
    total_bits: int
    beta: Fraction  # Eq. 7, bits per parameter
    ratio_kq: Fraction  # Eq. 6, C_KQ


def report(n: int, k: int, omega: int = 3, b_c: int = 32, b_fp: int = 32) -> Report:
    """Eq. 4 (B), Eq. 6 (C_KQ) and Eq. 7 (beta) for one layer.

    B = k * omega^2 * b_c + n * ceil(log2 k); beta = B / (n omega^2);
    C_KQ = n omega^2 b_FP / B. b_c = 32 for kernel-level only (K), 6 after
    codebook quantisation (K+C); the 64-entry level table is not counted.
    """
    idx_bits = n * ceil_log2(k)
    cb_bits = k * omega * omega * b_c
    total = idx_bits + cb_bits
    return Report(idx_bits, cb_bits, total, Fraction(total, n * omega * omega),
                  Fraction(n * omega * omega * b_fp, total))


def ratio_conventional(n: int, omega: int, u: int, b_1: int, b_fp: int = 32) -> Fraction:
    """Eq. 5: C_con = n omega^2 b_FP / (u b_1 + n omega^2 ceil(log2 u))."""
    return Fraction(n * omega * omega * b_fp, u * b_1 + n * omega * omega * ceil_log2(u))
