"""GPU parity of the retraining steps (Eq. 2 for the codebook, Sec. 3.2 for the
6-bit levels) and of the 6-bit quantisation of fully-connected weights, each
against the CPU oracle on the same seeded inputs."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import bits_equal, dev, gpu_quantize, to_dev
from paper_2003_05148_gb300 import kq

pytestmark = pytest.mark.gpu


def gpu_quantize_scalars(v, max_iters=100):
    m = v.shape[0]
    levels = torch.empty(64, dtype=torch.float32, device=dev())
    codes = torch.empty(m, dtype=torch.uint8, device=dev())
    it = torch.zeros(1, dtype=torch.int32, device=dev())
    ws = torch.zeros(4096, dtype=torch.uint8, device=dev())
    kq.kq_quantize_scalars_6bit(to_dev(v), max_iters, levels, codes, it, ws)
    st, flags = kq.kq_device_status(ws)
    return levels.cpu().numpy(), codes.cpu().numpy(), int(it.item()), st, flags


def gpu_codebook_grad_step(G, idx, C, lr):
    n, K = G.shape[0], C.shape[0]
    Cn = torch.empty(K, 9, dtype=torch.float32, device=dev())
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    ws = kq.workspace(n, K, dev())
    kq.kq_codebook_grad_step(to_dev(G), to_dev(idx.astype(np.int32)), lr, to_dev(C), Cn, counts, ws)
    st, flags = kq.kq_device_status(ws)
    return Cn.cpu().numpy(), counts.cpu().numpy(), st, flags


def gpu_levels_grad_step(G, idx, codes, levels, lr):
    nxt = torch.empty(64, dtype=torch.float32, device=dev())
    counts = torch.empty(64, dtype=torch.int64, device=dev())
    ws = torch.zeros(4096, dtype=torch.uint8, device=dev())
    kq.kq_levels_grad_step(to_dev(G), to_dev(idx.astype(np.int32)), to_dev(codes), lr, to_dev(levels), nxt, counts,
                           ws)
    st, flags = kq.kq_device_status(ws)
    return nxt.cpu().numpy(), counts.cpu().numpy(), st, flags


def _check_step(got, C, mean, lr, gmax):
    """got = C - lr * mean within the rounding of the exact fixed-point mean (relative
    1e-5 of the row's largest mean, floor 1e-9 of max|G|), the step and the result."""
    mean = mean.astype(np.float64).reshape(C.shape[0], -1)
    C64 = C.astype(np.float64).reshape(mean.shape)
    scale = np.abs(mean).max(axis=1, keepdims=True)
    tol = abs(lr) * (1e-5 * scale + 1e-9 * gmax) + 2.0 ** -23 * (np.abs(C64) + abs(lr) * np.abs(mean))
    err = np.abs(got.astype(np.float64).reshape(mean.shape) - (C64 - lr * mean))
    assert (err <= tol).all(), f"{(err > tol).sum()} entries off, worst {(err / np.maximum(tol, 1e-300)).max():.3g}x tol"


# --------------------------------------------------------------------------- 6-bit quantisation of FC weights

def _fc_weights(m, seed, fan_in=4096):
    # He-scaled Gaussian, the initialisation of a fully-connected layer
    return (synth.random_kernels((m + 8) // 9, 9, seed, float(np.sqrt(2.0 / fan_in))).reshape(-1)[:m]).copy()


@pytest.mark.parametrize("m,seed", [(1, 1), (5, 2), (63, 3), (64, 4), (1000, 5), (100003, 6), (1000003, 7)])
def test_quantize_scalars_matches_oracle(m, seed):
    v = _fc_weights(m, seed)
    lv_g, cd_g, it_g, st, _ = gpu_quantize_scalars(v)
    lv_r, cd_r, it_r = oracle.level_fit_scalars(v)
    assert st == 0
    assert bits_equal(lv_g, lv_r) and np.array_equal(cd_g, cd_r) and it_g == it_r


@pytest.mark.parametrize("case", ["midpoint_ties", "tight_range", "tight_range_iterated", "constant", "two_values",
                                  "huge_range", "subnormal"])
def test_quantize_scalars_ties_and_duplicate_levels(case):
    iters = 100
    if case == "midpoint_ties":
        # linspace(0, 63) levels are the integers; k + 0.5 is equidistant from two
        v = np.concatenate([np.arange(64), np.arange(63) + 0.5, [0.5, 62.5, 31.0]]).astype(np.float32)
        iters = 0
    elif case in ("tight_range", "tight_range_iterated"):
        # 8 ulps of range: the 64 initial levels collapse onto 9 values (duplicates)
        v = (np.float32(1.0) + np.arange(4000) % 9 * np.float32(2.0 ** -23)).astype(np.float32)
        iters = 0 if case == "tight_range" else 10
    elif case == "constant":
        v = np.full(777, 0.125, np.float32)
    elif case == "two_values":
        v = np.where(np.arange(1001) % 3 == 0, -2.0, 5.0).astype(np.float32)
    elif case == "huge_range":
        v = _fc_weights(5000, 11) * np.float32(1e37)
    else:
        v = _fc_weights(5000, 12) * np.float32(1e-38)
    lv_g, cd_g, it_g, st, _ = gpu_quantize_scalars(v, iters)
    lv_r, cd_r, it_r = oracle.level_fit_scalars(v, iters)
    assert st == 0
    assert bits_equal(lv_g, lv_r) and np.array_equal(cd_g, cd_r) and it_g == it_r


def test_quantize_scalars_is_unit_weight_codebook_quantize():
    v = _fc_weights(9 * 20000, 13)
    lv1, cd1, it1, st1, _ = gpu_quantize_scalars(v)
    lv2, cd2, it2, st2, _ = gpu_quantize(v.reshape(-1, 9), np.ones(20000, np.int32))
    assert st1 == 0 and st2 == 0
    assert bits_equal(lv1, lv2) and np.array_equal(cd1, cd2.reshape(-1)) and it1 == it2


def test_quantize_scalars_full_fc_layer_properties():
    # VGG-16 fc7 (4096 x 4096): too large for the oracle's 64-way scan within seconds;
    # check what holds at any size: sorted levels, every sampled scalar at its
    # nearest level (fp32 |v - level|, lower index on ties), levels equal to the
    # means of their scalars.
    m = 4096 * 4096
    v = _fc_weights(m, 14)
    lv, cd, it, st, _ = gpu_quantize_scalars(v)
    assert st == 0 and 0 < it <= 100
    assert np.all(np.diff(lv) >= 0)
    rows = synth.below(synth.stream_key(15, 3), 20000, m)
    assert np.array_equal(cd[rows], oracle.encode(v[rows], lv))
    sums = np.bincount(cd, weights=v.astype(np.float64), minlength=64)
    cnt = np.bincount(cd, minlength=64)
    used = cnt > 0
    if it < 100:  # converged: every used level is the mean of its scalars
        assert np.allclose(lv[used], sums[used] / cnt[used], rtol=1e-6, atol=1e-9 * np.abs(v).max())


def test_quantize_scalars_nonfinite_flagged():
    v = _fc_weights(1000, 16)
    v[17] = np.inf
    _, _, _, st, flags = gpu_quantize_scalars(v)
    assert st == 3 and flags & kq.FLAG_NONFINITE


# --------------------------------------------------------------------------- Eq. 2: codebook step

@pytest.mark.parametrize("n,K,lr", [(1, 1, 0.5), (4096, 16, 0.01), (100003, 1000, 0.1), (4194304, 65536, 0.05)])
def test_codebook_grad_step(n, K, lr):
    G = synth.random_kernels(n, 9, n + 1, 0.01)
    C = synth.random_kernels(K, 9, n + 2, 0.05)
    idx = synth.below(synth.stream_key(n + 3, 2), n, max(K - 1, 1)).astype(np.int32)  # K-1 empty (K > 1)
    Cg, cg, st, _ = gpu_codebook_grad_step(G, idx, C, lr)
    Cr, cr = oracle.codebook_grad_step(G, idx, C, lr)
    mean = -oracle.codebook_grad_step(G, idx, np.zeros_like(C), 1.0)[0]
    assert st == 0 and np.array_equal(cg, cr)
    _check_step(Cg, C, mean, lr, float(np.abs(G).max()))
    empty = cr == 0
    assert bits_equal(Cg[empty], C[empty])


def test_codebook_grad_step_quadratic_loss_gives_the_centroid():
    # dL/dW'_i = c_{idx_i} - W_i for L = 1/2 sum ||W'_i - W_i||^2; one step with lr = 1
    # reaches the Eq. 1 update
    W = synth.random_kernels(50000, 9, 31, 0.05)
    C = synth.random_kernels(300, 9, 32, 0.05)
    idx, _ = oracle.assign(W, C)
    G = (C[idx] - W).astype(np.float32)
    Cg, cg, st, _ = gpu_codebook_grad_step(G, idx, C, 1.0)
    Cu, cu = oracle.update(W, idx, C)
    assert st == 0 and np.array_equal(cg, cu)
    assert np.abs(Cg - Cu).max() <= 1e-5 * np.abs(Cu).max()


def test_codebook_grad_step_bad_index_and_nonfinite():
    G = synth.random_kernels(1000, 9, 41, 0.1)
    C = synth.random_kernels(10, 9, 42)
    idx = (np.arange(1000) % 10).astype(np.int32)
    idx[5] = 10
    Cg, cg, st, flags = gpu_codebook_grad_step(G, idx, C, 0.5)
    assert st == 5 and flags & kq.FLAG_INDEX_RANGE
    assert np.array_equal(cg, oracle.codebook_grad_step(G, idx, C, 0.5)[1])
    G[3, 3] = np.nan
    _, _, st, flags = gpu_codebook_grad_step(G, (np.arange(1000) % 10).astype(np.int32), C, 0.5)
    assert st == 3 and flags & kq.FLAG_NONFINITE


# --------------------------------------------------------------------------- Sec. 3.2: level step

@pytest.mark.parametrize("n,K,lr", [(1, 1, 1.0), (4096, 16, 0.01), (100003, 1000, 0.1), (4194304, 65536, 0.05)])
def test_levels_grad_step(n, K, lr):
    G = synth.random_kernels(n, 9, n + 5, 0.01)
    C = synth.random_kernels(K, 9, n + 6, 0.05)
    idx = synth.below(synth.stream_key(n + 7, 2), n, K).astype(np.int32)
    levels, codes, _ = oracle.level_fit(C, np.bincount(idx, minlength=K).astype(np.int32), 20)
    ng, cg, st, _ = gpu_levels_grad_step(G, idx, codes, levels, lr)
    nr, cr = oracle.levels_grad_step(G, idx, codes, levels, lr)
    mean = -oracle.levels_grad_step(G, idx, codes, np.zeros(64, np.float32), 1.0)[0]
    assert st == 0 and np.array_equal(cg, cr) and cg.sum() == 9 * n
    _check_step(ng.reshape(1, 64), levels.reshape(1, 64), mean.reshape(1, 64), lr, float(np.abs(G).max()))
    assert bits_equal(ng[cr == 0], levels[cr == 0])


def test_levels_grad_step_bad_index_and_code():
    G = synth.random_kernels(2000, 9, 51, 0.1)
    idx = (np.arange(2000) % 20).astype(np.int32)
    idx[9] = -1
    codes = (np.arange(180) % 64).astype(np.uint8).reshape(20, 9)
    levels = np.linspace(-1, 1, 64).astype(np.float32)
    ng, cg, st, flags = gpu_levels_grad_step(G, idx, codes, levels, 0.25)
    assert st == 5 and flags & kq.FLAG_INDEX_RANGE
    nr, cr = oracle.levels_grad_step(G, idx, codes, levels, 0.25)
    assert np.array_equal(cg, cr)
    codes[4, 2] = 70
    _, _, st, flags = gpu_levels_grad_step(G, (np.arange(2000) % 20).astype(np.int32), codes, levels, 0.25)
    assert st == 5 and flags & kq.FLAG_CODE_RANGE


def test_retraining_steps_deterministic():
    G = synth.random_kernels(300000, 9, 61, 0.02)
    C = synth.random_kernels(4000, 9, 62, 0.05)
    idx = synth.below(synth.stream_key(63, 2), 300000, 4000).astype(np.int32)
    a = gpu_codebook_grad_step(G, idx, C, 0.1)
    b = gpu_codebook_grad_step(G, idx, C, 0.1)
    assert bits_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    levels, codes, _ = oracle.level_fit(C, np.bincount(idx, minlength=4000).astype(np.int32), 20)
    x = gpu_levels_grad_step(G, idx, codes, levels, 0.1)
    y = gpu_levels_grad_step(G, idx, codes, levels, 0.1)
    assert bits_equal(x[0], y[0]) and np.array_equal(x[1], y[1])
