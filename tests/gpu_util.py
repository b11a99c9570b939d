"""Helpers for the GPU parity tests: device setup, calls through the C ABI binding,
and the comparison rules (the tolerances are written here, once)."""
import numpy as np
import torch

import oracle
from paper_2003_05148_gb300 import build, kq

# Centroids: |gpu - oracle| <= 1e-5 * max_j |oracle_kj| per codeword (inf-norm relative).
CENTROID_RTOL = 1e-5
# Indices may differ only where the oracle's fp64 best and second-best distances
# are closer than this, relative to the best.
TIE_RTOL = 1e-6

_ready = False


def dev():
    global _ready
    if not _ready:
        build.build()
        kq.lib()
        _ready = True
    return torch.device("cuda:0")


def to_dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def gpu_assign(W, C, with_dist=True, hint=None):
    n, K = W.shape[0], C.shape[0]
    Wd, Cd = to_dev(W), to_dev(C)
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    dist = torch.empty(n, dtype=torch.float32, device=dev()) if with_dist else None
    ws = kq.workspace(n, K, dev())
    kq.kq_assign(Wd, Cd, idx, dist, ws, hint=None if hint is None else to_dev(hint.astype(np.int32)))
    st, flags = kq.kq_device_status(ws)
    return idx.cpu().numpy(), (dist.cpu().numpy() if with_dist else None), st, flags


def gpu_assign_cuda_cores(W, C):
    """The same assignment through kq_assign_noalloc, which always runs the
    CUDA-core kernel (kq_assign picks the kernel by size)."""
    n = W.shape[0]
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    dist = torch.empty(n, dtype=torch.float32, device=dev())
    kq.kq_assign_noalloc(to_dev(W), to_dev(C), idx, dist)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), dist.cpu().numpy()


def gpu_update(W, idx, C_prev):
    n, K = W.shape[0], C_prev.shape[0]
    Wd, idxd, Cp = to_dev(W), to_dev(idx.astype(np.int32)), to_dev(C_prev)
    Cn = torch.empty_like(Cp)
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    ws = kq.workspace(n, K, dev())
    kq.kq_update_centroids(Wd, idxd, Cp, Cn, counts, ws)
    st, flags = kq.kq_device_status(ws)
    return Cn.cpu().numpy(), counts.cpu().numpy(), st, flags


def gpu_quantize(C, counts, max_iters=100):
    K = C.shape[0]
    Cd, cd = to_dev(C), to_dev(counts.astype(np.int32))
    levels = torch.empty(64, dtype=torch.float32, device=dev())
    codes = torch.empty(K, 9, dtype=torch.uint8, device=dev())
    it = torch.zeros(1, dtype=torch.int32, device=dev())
    ws = kq.workspace(K, K, dev())
    kq.kq_quantize_codebook_6bit(Cd, cd, max_iters, levels, codes, it, ws)
    st, flags = kq.kq_device_status(ws)
    return levels.cpu().numpy(), codes.cpu().numpy(), int(it.item()), st, flags


def gpu_reconstruct(idx, C, codes=None, levels=None):
    n, K = idx.shape[0], C.shape[0]
    Wr = torch.empty(n, 9, dtype=torch.float32, device=dev())
    ws = kq.workspace(n, K, dev())
    kq.kq_reconstruct(to_dev(idx.astype(np.int32)), to_dev(C), None if codes is None else to_dev(codes),
                      None if levels is None else to_dev(levels), Wr, ws)
    st, flags = kq.kq_device_status(ws)
    return Wr.cpu().numpy(), st, flags


def check_indices(W, C, idx_gpu, idx_ref, rows=None):
    """Bit-exact indices, except rows whose oracle fp64 gap is below TIE_RTOL
    (there the GPU's choice must itself be within that gap of the best)."""
    bad = np.nonzero(idx_gpu != idx_ref)[0]
    if bad.size == 0:
        return 0
    Wb = W[bad] if rows is None else W[rows[bad]]
    _, _, d1, d2 = oracle.assign(Wb, C, gap=True)
    gap = (d2 - d1) / np.maximum(d1, 1e-300)
    assert np.all(gap < TIE_RTOL), f"{bad.size} index mismatches, min fp64 gap {gap.min():.3g}"
    cg = C[idx_gpu[bad]].astype(np.float64)
    dg = ((Wb.astype(np.float64) - cg) ** 2).sum(axis=1)
    assert np.all(dg - d1 <= TIE_RTOL * np.maximum(d1, 1e-300))
    return bad.size


def check_centroids(C_gpu, C_ref):
    scale = np.abs(C_ref).max(axis=1, keepdims=True).astype(np.float64)
    err = np.abs(C_gpu.astype(np.float64) - C_ref.astype(np.float64))
    ok = err <= CENTROID_RTOL * scale
    assert ok.all(), f"{(~ok).sum()} centroid entries off, worst rel {(err / np.maximum(scale, 1e-300)).max():.3g}"


def bits_equal(a, b):
    a, b = np.ascontiguousarray(a), np.ascontiguousarray(b)
    return a.shape == b.shape and np.array_equal(a.view(np.uint8), b.view(np.uint8))
