"""GPU parity: every CUDA step through the C ABI against the CPU oracle, one step
at a time from identical inputs (Sec. 3.1 Eq. 1 assign/update, Sec. 3.2 6-bit
codebook quantisation and recovery).

Bars: indices bit-exact (except oracle fp64 near-ties, gpu_util.TIE_RTOL);
distances bit-exact; counts exact; centroids within gpu_util.CENTROID_RTOL
(inf-norm relative per codeword); levels, codes and reconstructed weights
bit-exact given identical fp32 inputs.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import (bits_equal, check_centroids, check_indices, dev, gpu_assign, gpu_assign_cuda_cores, gpu_quantize,
                      gpu_reconstruct,
                      gpu_update, to_dev)
from paper_2003_05148_gb300 import kq

pytestmark = pytest.mark.gpu
THREADS = oracle.default_threads()


def _layer(cfg, li=0):
    lay = synth.workload(cfg).layers[li]
    W, sel = synth.layer_inputs(lay)
    return lay, W, oracle.gather_rows(W, sel)


# --------------------------------------------------------------------------- assign

@pytest.mark.parametrize("cfg,li", [(1, 0), (2, 0), (3, 0), (3, 1), (3, 8), (4, 0), (4, 4), (4, 9)])
def test_assign_workload_layers(cfg, li):
    lay, W, C0 = _layer(cfg, li)
    idx, dist, st, _ = gpu_assign(W, C0)
    assert st == 0
    rows = None
    if lay.n * lay.K > 3e8:  # rows are independent: check a seeded sample on the CPU
        rows = np.sort(synth.below(synth.stream_key(lay.seed, 9), 8192, lay.n))
    Wc = W if rows is None else W[rows]
    idx_ref, dist_ref = oracle.assign(Wc, C0, threads=THREADS)
    ig = idx if rows is None else idx[rows]
    dg = dist if rows is None else dist[rows]
    assert check_indices(W, C0, ig, idx_ref, rows) == 0
    assert bits_equal(dg, dist_ref)


def test_assign_full_size_stress_sampled():
    # 2048x2048 layer, K = 65536: the launch configuration the benchmark times.
    lay, W, C0 = _layer(5)
    idx, dist, st, _ = gpu_assign(W, C0)
    assert st == 0
    rows = np.sort(synth.below(synth.stream_key(lay.seed, 9), 4096, lay.n))
    rows[-1] = lay.n - 1  # include the ragged end of the last CTA
    idx_ref, dist_ref = oracle.assign(W[rows], C0, threads=THREADS)
    assert check_indices(W, C0, idx[rows], idx_ref, rows) == 0
    assert bits_equal(dist[rows], dist_ref)
    # every selected initial kernel is its own nearest codeword at distance 0
    sel = synth.init_selection(lay.n, lay.K, lay.seed + 1)
    assert np.all(dist[sel] == 0)


@pytest.mark.parametrize("n,K", [(1, 1), (3, 2), (1023, 16), (1025, 17), (2047, 300), (6000, 5000),
                                 (300, 300), (5000, 1), (100003, 7)])
def test_assign_ragged_and_split(n, K):
    W = synth.random_kernels(n, 9, n + 17, 0.1)
    C = synth.random_kernels(K, 9, K + 29, 0.1)
    idx, dist, st, _ = gpu_assign(W, C)
    assert st == 0
    idx_ref, dist_ref = oracle.assign(W, C, threads=THREADS)
    assert check_indices(W, C, idx, idx_ref) == 0
    assert bits_equal(dist, dist_ref)


def test_assign_exact_ties_and_duplicates():
    rng = np.random.default_rng(5)
    W = rng.integers(-3, 4, size=(5000, 9)).astype(np.float32)
    C = rng.integers(-3, 4, size=(700, 9)).astype(np.float32)
    C[350:] = C[:350]  # every codeword duplicated: the lower index must win
    idx, dist, st, _ = gpu_assign(W, C)
    idx_ref, dist_ref = oracle.assign(W, C, threads=THREADS)
    assert st == 0 and np.array_equal(idx, idx_ref) and bits_equal(dist, dist_ref)
    assert idx.max() < 350


def _oracle_check(W, C, idx, dist):
    idx_ref, dist_ref = oracle.assign(W, C, threads=THREADS)
    assert check_indices(W, C, idx, idx_ref) == 0
    assert bits_equal(dist, dist_ref)


@pytest.mark.parametrize("case", ["offset", "tiny", "mixed", "subnormal", "large", "near_dup"])
def test_assign_filter_extreme_scales(case):
    # The expanded-form test must stay exact where it is weakest: heavy
    # cancellation (a large common offset), tiny and subnormal values, mixed
    # magnitudes, large values, and codewords a few ulps apart.
    W = synth.random_kernels(20000, 9, 101, 1.0)
    C = synth.random_kernels(3000, 9, 102, 1.0)
    if case == "offset":
        W, C = W * 1e-3 + 1000.0, C * 1e-3 + 1000.0
    elif case == "tiny":
        W, C = W * 1e-30, C * 1e-30
    elif case == "mixed":
        W[::2] *= 1e6
        C[::3] *= 1e-6
    elif case == "subnormal":
        W, C = W * 1e-39, C * 1e-39
    elif case == "large":
        W, C = W * 1e15, C * 1e15
    elif case == "near_dup":
        C[1::2] = np.nextafter(C[0::2], np.float32(np.inf))[: C[1::2].shape[0]]
        W[: C.shape[0]] = C
    W, C = W.astype(np.float32), C.astype(np.float32)
    idx, dist, st, _ = gpu_assign(W, C)
    assert st == 0
    _oracle_check(W, C, idx, dist)
    # the CUDA-core kernel (kq_assign takes the tensor cores at this size) as well
    idx2, dist2 = gpu_assign_cuda_cores(W, C)
    _oracle_check(W, C, idx2, dist2)


TC_MIN_N = 256 * 152  # one row block per SM (from about 256 kernels on the tensor cores run)


@pytest.mark.parametrize("case", ["plain", "offset", "mixed", "large", "near_dup", "ragged", "outlier_codeword",
                                  "outlier_rows"])
def test_assign_tensor_core_path(case):
    # n large enough for the tensor-core path; K = 1000 is not a multiple of the
    # 128-codeword tile, so padding codewords are exercised too. The fp16 operands
    # are scaled by one power of two per call: an outlier codeword sets that scale
    # (every other value then sits low in the fp16 range), and rows far outside the
    # codebook leave the range (they are tested exactly against every codeword).
    n, K = TC_MIN_N + 1000, 1000
    if case == "ragged":
        n = TC_MIN_N + 77
    W = synth.random_kernels(n, 9, 201, 0.05)
    C = synth.random_kernels(K, 9, 202, 0.05)
    if case == "offset":
        W, C = W * 1e-3 + 1000.0, C * 1e-3 + 1000.0
    elif case == "mixed":
        W[::2] *= 1e6
        C[::3] *= 1e-6
    elif case == "large":
        W, C = W * 1e15, C * 1e15
    elif case == "near_dup":
        C[1::2] = np.nextafter(C[0::2], np.float32(np.inf))[: C[1::2].shape[0]]
        W[:K] = C
    elif case == "outlier_codeword":
        C[5] *= 3e4
    elif case == "outlier_rows":
        W[::97] *= 1e4
    W, C = W.astype(np.float32), C.astype(np.float32)
    idx, dist, st, _ = gpu_assign(W, C)
    assert st == 0
    rows = np.sort(synth.below(synth.stream_key(203, 9), 6000, n))
    if case == "outlier_rows":
        rows = np.unique(np.concatenate([rows, np.arange(0, n, 97)[:500]]))
    rows[-1] = n - 1
    idx_ref, dist_ref = oracle.assign(W[rows], C, threads=THREADS)
    assert check_indices(W, C, idx[rows], idx_ref, rows) == 0
    assert bits_equal(dist[rows], dist_ref)


def test_assign_paths_agree():
    # the tensor-core kernel (kq_assign) and the CUDA-core kernel (kq_assign_noalloc)
    # give bit-identical results on the same kernels; n spans several row blocks per
    # SM and a ragged last block, cold and warm-started
    n = 5 * TC_MIN_N + 333
    W = synth.random_kernels(n, 9, 211, 0.05)
    C = synth.random_kernels(2000, 9, 212, 0.05)
    i_tc, d_tc, st1, _ = gpu_assign(W, C)
    assert st1 == 0
    i_cc, d_cc = gpu_assign_cuda_cores(W, C)
    assert np.array_equal(i_tc, i_cc) and bits_equal(d_tc, d_cc)
    for sl in (slice(0, 20000), slice(n - 20000, n)):
        i_s, d_s, st2, _ = gpu_assign(W[sl], C)  # a smaller n: fewer CTAs than SMs
        assert st2 == 0
        assert np.array_equal(i_tc[sl], i_s) and bits_equal(d_tc[sl], d_s)
    hint = synth.below(synth.stream_key(213, 9), n, 2000).astype(np.int32)
    hint[::3] = i_tc[::3]
    i_w, d_w, st3, _ = gpu_assign(W, C, hint=hint)
    assert st3 == 0
    assert np.array_equal(i_w, i_tc) and bits_equal(d_w, d_tc)


@pytest.mark.parametrize("K", [1, 100, 256, 512, 1025, 1536])
def test_assign_small_codebook_many_blocks(K):
    # small codebooks (one to six codeword tiles) over several waves of row blocks
    # and a ragged last block; cold and warm-started, the warm rows grouped by hinted
    # chunk inside each CTA from 256 codewords on. Bit-identical to the CUDA-core
    # kernel, and to the oracle on sampled rows.
    n = 7 * TC_MIN_N + 77
    W = synth.random_kernels(n, 9, 271 + K, 0.05)
    C = W[synth.init_selection(n, K, 272 + K)]
    i_tc, d_tc, st, _ = gpu_assign(W, C)
    assert st == 0
    i_cc, d_cc = gpu_assign_cuda_cores(W, C)
    assert np.array_equal(i_tc, i_cc) and bits_equal(d_tc, d_cc)
    hint = synth.below(synth.stream_key(273 + K, 9), n, K).astype(np.int32)
    hint[::2] = i_tc[::2]
    i_w, d_w, st, _ = gpu_assign(W, C, hint=hint)
    assert st == 0 and np.array_equal(i_w, i_tc) and bits_equal(d_w, d_tc)
    rows = np.sort(synth.below(synth.stream_key(274 + K, 9), 3000, n))
    rows[-1] = n - 1
    idx_ref, dist_ref = oracle.assign(W[rows], C, threads=THREADS)
    assert check_indices(W, C, i_tc[rows], idx_ref, rows) == 0
    assert bits_equal(d_tc[rows], dist_ref)


def test_fit_small_codebook_objective():
    # the fit's objective at a small codebook comes from the assign kernel's per-CTA
    # partial sums (fixed order, rows grouped by hint inside each CTA): the oracle's
    # objective of the same assignment; the final assignment and counts are those of
    # the fit's own codebook
    n, K = 3 * TC_MIN_N + 5, 700
    W = synth.random_kernels(n, 9, 281, 0.05)
    C0 = W[synth.init_selection(n, K, 282)]
    C1, idx1, cnt1, obj = _gpu_fit(W, C0, 1)
    idx_ref, dist_ref = oracle.assign(W, C0, threads=THREADS)
    assert obj[0] == pytest.approx(oracle.objective(dist_ref), rel=1e-12)
    C_ref, _ = oracle.update(W, idx_ref, C0)
    check_centroids(C1, C_ref)
    i2, d2 = oracle.assign(W, C1, threads=THREADS)
    assert check_indices(W, C1, idx1, i2) == 0
    assert np.array_equal(cnt1, np.bincount(idx1, minlength=K))
    assert obj[1] == pytest.approx(oracle.objective(d2), rel=1e-12)


@pytest.mark.parametrize("case", ["kd_leaf_hints", "kd_leaf_hints_duplicates", "pilot", "pilot_above_tree"])
def test_assign_cold_start_paths(case):
    # Without a hint on the tensor-core path, the full pass is seeded with hints: on
    # large problems (n K >= 1e10, up to 65536 codewords) each kernel's nearest codeword
    # in its k-d leaf tile, otherwise (from 16384 codewords) a pilot pass against the
    # first K / 16 codewords.
    # The answer is the plain argmin all the same (the CUDA-core kernel, the oracle on
    # sampled rows, and a run warm-started from the answer); with every codeword
    # present twice, the lower index of each tied pair.
    n, K = {"kd_leaf_hints": (655360 + 123, 16384 + 77), "kd_leaf_hints_duplicates": (655360 + 45, 16384 + 77),
            "pilot": (2 * TC_MIN_N + 123, 16384 + 77), "pilot_above_tree": (2 * TC_MIN_N + 123, 65536 + 1000)}[case]
    W = synth.random_kernels(n, 9, 261, 0.05)
    C = W[synth.init_selection(n, K, 262)]
    if case == "kd_leaf_hints_duplicates":
        C[K // 2:] = C[:K - K // 2]
    i0, d0, st, _ = gpu_assign(W, C)
    assert st == 0
    if K <= 65536:  # the allocation-free CUDA-core variant holds up to 65536 codewords
        i_cc, d_cc = gpu_assign_cuda_cores(W, C)
        assert np.array_equal(i0, i_cc) and bits_equal(d0, d_cc)
    rows = np.sort(synth.below(synth.stream_key(263, 9), 2000, n))
    idx_ref, dist_ref = oracle.assign(W[rows], C, threads=THREADS)
    assert check_indices(W, C, i0[rows], idx_ref, rows) == 0
    assert bits_equal(d0[rows], dist_ref)
    i1, d1, st, _ = gpu_assign(W, C, hint=i0)
    assert st == 0 and np.array_equal(i1, i0) and bits_equal(d1, d0)


def test_assign_hint_order_path():
    # K >= 4096 on the tensor-core path: warm-started rows are processed grouped by
    # hint; the result must be the cold result, whatever the hints (exact, random,
    # out of range), and the cold result matches the oracle on sampled rows
    n, K = 5 * TC_MIN_N + 333, 5000
    W = synth.random_kernels(n, 9, 221, 0.05)
    C = synth.random_kernels(K, 9, 222, 0.05)
    i0, d0, st, _ = gpu_assign(W, C)
    assert st == 0
    rows = np.sort(synth.below(synth.stream_key(223, 9), 3000, n))
    idx_ref, dist_ref = oracle.assign(W[rows], C, threads=THREADS)
    assert check_indices(W, C, i0[rows], idx_ref, rows) == 0
    assert bits_equal(d0[rows], dist_ref)
    rand = synth.below(synth.stream_key(224, 2), n, K).astype(np.int32)
    rand[::7] = -1
    rand[3::11] = K + 5
    for h in (i0, rand, np.where(np.arange(n) % 3 == 0, i0, rand).astype(np.int32)):
        i1, d1, st, _ = gpu_assign(W, C, hint=h)
        assert st == 0 and np.array_equal(i1, i0) and bits_equal(d1, d0)


@pytest.mark.parametrize("K", [2000, 4500])
def test_fit_hint_order_deterministic_and_chained(K):
    # K = 4500: warm starts grouped by hint across the grid; K = 2000: within each CTA
    n = TC_MIN_N + 21000
    W = synth.random_kernels(n, 9, 231, 0.05)
    C0 = W[synth.init_selection(n, K, 232)]
    a = _gpu_fit(W, C0, 3)
    b = _gpu_fit(W, C0, 3)
    for x, y in zip(a, b):
        assert bits_equal(x, y)
    C = C0
    for _ in range(3):
        C = _gpu_fit(W, C, 1)[0]
    assert bits_equal(a[0], C)
    assert np.all(a[3][1:] <= a[3][:-1] * (1 + 1e-6))


def test_fit_second_iteration_against_oracle():
    """The second iteration of a fit with K >= 4096 (a hint-ordered warm start, the
    counts of the first update reused as the grouping's histogram): its centroids are
    the oracle's update of the oracle's assignment against the first iteration's
    centroids, and bit-identical to a one-iteration fit started there. Kernel norms
    spread over a factor of ~100 (log-normal) exercise the fixed-point scale."""
    n, K = TC_MIN_N + 9001, 4200
    rng = np.random.default_rng(244)
    W = (synth.random_kernels(n, 9, 241, 0.05) * np.exp(rng.normal(0.0, 1.0, size=(n, 1)))).astype(np.float32)
    C0 = W[synth.init_selection(n, K, 243)]
    C1 = _gpu_fit(W, C0, 1)[0]
    C2, idx2, cnt2, obj2 = _gpu_fit(W, C0, 2)
    idx1_ref, _ = oracle.assign(W, C1, threads=THREADS)
    C2_ref, _ = oracle.update(W, idx1_ref, C1)
    check_centroids(C2, C2_ref)
    C2b, idx2b, cnt2b, _ = _gpu_fit(W, C1, 1)
    assert bits_equal(C2, C2b) and np.array_equal(idx2, idx2b) and np.array_equal(cnt2, cnt2b)
    assert np.array_equal(cnt2, np.bincount(idx2, minlength=K))


def test_assign_hint_never_changes_result():
    lay, W, C0 = _layer(2)
    idx0, dist0, _, _ = gpu_assign(W, C0)
    n, K = lay.n, lay.K
    hints = [idx0,                                                            # the answer itself
             synth.below(synth.stream_key(5, 2), n, K).astype(np.int32),      # random
             np.full(n, -7, np.int32),                                        # out of range: ignored
             np.where(np.arange(n) % 2 == 0, idx0, K + 3).astype(np.int32)]   # mixed
    for h in hints:
        idx, dist, st, _ = gpu_assign(W, C0, hint=h)
        assert st == 0
        assert np.array_equal(idx, idx0) and bits_equal(dist, dist0)
    # exact ties: the hint points at the higher duplicate, the lower index must still win
    rng = np.random.default_rng(9)
    Wi = rng.integers(-3, 4, size=(4000, 9)).astype(np.float32)
    Ci = rng.integers(-3, 4, size=(600, 9)).astype(np.float32)
    Ci[300:] = Ci[:300]
    ref, dref, _, _ = gpu_assign(Wi, Ci)
    idx, dist, st, _ = gpu_assign(Wi, Ci, hint=(ref + 300).astype(np.int32))
    assert np.array_equal(idx, ref) and bits_equal(dist, dref)
    _oracle_check(Wi, Ci, idx, dist)


def test_assign_nonfinite_flagged():
    W = synth.random_kernels(2000, 9, 3)
    W[1234, 5] = np.nan
    W[77, 0] = np.inf
    C = synth.random_kernels(40, 9, 4)
    idx, dist, st, flags = gpu_assign(W, C)
    assert st == 3 and flags & kq.FLAG_NONFINITE
    idx_ref, dist_ref = oracle.assign(W, C)
    assert np.array_equal(idx, idx_ref) and bits_equal(dist, dist_ref)
    # a non-finite codeword disables the filter for the whole call; still exact
    C[7, 3] = np.nan
    idx, dist, st, flags = gpu_assign(W, C, hint=np.zeros(2000, np.int32))
    assert st == 3
    idx_ref, dist_ref = oracle.assign(W, C)
    assert np.array_equal(idx, idx_ref) and bits_equal(dist, dist_ref)


# --------------------------------------------------------------------------- update

@pytest.mark.parametrize("cfg", [1, 2, 5])
def test_update_from_identical_indices(cfg):
    lay, W, C0 = _layer(cfg)
    if cfg == 5:
        idx = synth.below(synth.stream_key(lay.seed, 8), lay.n, lay.K).astype(np.int32)
    else:
        idx, _ = oracle.assign(W, C0, threads=THREADS)
    C_g, cnt_g, st, _ = gpu_update(W, idx, C0)
    C_r, cnt_r = oracle.update(W, idx, C0)
    assert st == 0
    assert np.array_equal(cnt_g, cnt_r)
    check_centroids(C_g, C_r)
    empty = cnt_r == 0
    assert bits_equal(C_g[empty], C0[empty])


def test_update_empty_clusters_and_bad_index():
    W = synth.random_kernels(3000, 9, 7, 0.2)
    C0 = synth.random_kernels(50, 9, 8)
    idx = synth.below(synth.stream_key(9, 2), 3000, 25).astype(np.int32)  # codewords 25..49 stay empty
    C_g, cnt_g, st, _ = gpu_update(W, idx, C0)
    C_r, cnt_r = oracle.update(W, idx, C0)
    assert st == 0 and np.array_equal(cnt_g, cnt_r)
    check_centroids(C_g, C_r)
    assert bits_equal(C_g[25:], C0[25:])
    idx[17] = 50
    _, cnt_g, st, flags = gpu_update(W, idx, C0)
    assert st == 5 and flags & kq.FLAG_INDEX_RANGE and cnt_g.sum() == 2999


@pytest.mark.parametrize("case", ["zero_prev", "tiny_prev", "outlier", "nonfinite_prev"])
def test_update_scale_fallback(case):
    # kq_update_centroids guesses its fixed-point scale from max|C_prev|; inputs that
    # break the guess take the exact fallback pass and must give the same answer.
    n, K = 50000, 700
    W = synth.random_kernels(n, 9, 5, 0.05)
    C0 = synth.random_kernels(K, 9, 6, 0.05)
    idx = synth.below(synth.stream_key(7, 2), n, K).astype(np.int32)
    if case == "zero_prev":
        C0[:] = 0
    elif case == "tiny_prev":
        C0 *= 1e-6
    elif case == "outlier":
        W[123, 4] = 1e4
    elif case == "nonfinite_prev":
        C0[5, 5] = np.inf
    C_g, cnt_g, st, _ = gpu_update(W, idx, C0)
    C_r, cnt_r = oracle.update(W, idx, C0)
    assert st == 0 and np.array_equal(cnt_g, cnt_r)
    check_centroids(C_g, C_r)
    C_g2, _, _, _ = gpu_update(W, idx, C0)
    assert bits_equal(C_g, C_g2)


def test_update_k1_global_mean():
    W = synth.random_kernels(77777, 9, 11, 0.05)
    C0 = W[:1].copy()
    C_g, cnt_g, st, _ = gpu_update(W, np.zeros(77777, np.int32), C0)
    C_r, _ = oracle.update(W, np.zeros(77777, np.int32), C0)
    assert st == 0 and cnt_g[0] == 77777
    check_centroids(C_g, C_r)


# --------------------------------------------------------------------------- fit

def _gpu_fit(W, C0, iters):
    n, K = W.shape[0], C0.shape[0]
    Wd, Cd = to_dev(W), to_dev(C0)
    C = torch.empty_like(Cd)
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    obj = torch.empty(iters + 1, dtype=torch.float64, device=dev())
    ws = kq.workspace(n, K, dev())
    kq.kq_fit_codebook(Wd, Cd, iters, C, idx, counts, obj, ws)
    st, _ = kq.kq_device_status(ws)
    assert st == 0
    return C.cpu().numpy(), idx.cpu().numpy(), counts.cpu().numpy(), obj.cpu().numpy()


@pytest.mark.parametrize("cfg,li", [(1, 0), (2, 0), (3, 2), (4, 1)])
def test_fit_stepwise(cfg, li):
    lay, W, C0 = _layer(cfg, li)
    T = 3
    C = C0
    objs = []
    for t in range(T):
        C_next, idx_next, cnt_next, obj = _gpu_fit(W, C, 1)
        idx_ref, dist_ref = oracle.assign(W, C, threads=THREADS)
        C_ref, _ = oracle.update(W, idx_ref, C)
        check_centroids(C_next, C_ref)
        objs.append(obj[0])
        assert obj[0] == pytest.approx(oracle.objective(dist_ref), rel=1e-12)
        # the fit's final assignment and counts are those of its own C_next
        i2, d2 = oracle.assign(W, C_next, threads=THREADS)
        assert check_indices(W, C_next, idx_next, i2) == 0
        assert np.array_equal(cnt_next, np.bincount(idx_next, minlength=lay.K))
        assert obj[1] == pytest.approx(oracle.objective(d2), rel=1e-12)
        C = C_next
    # T iterations in one call == T chained single-iteration calls, bit for bit
    C_T, idx_T, cnt_T, obj_T = _gpu_fit(W, C0, T)
    assert bits_equal(C_T, C)
    assert np.all(obj_T[1:] <= obj_T[:-1] * (1 + 1e-6))


def _gpu_fit_run(W, C0, iters, flags, stats=None):
    n, K = W.shape[0], C0.shape[0]
    C = torch.empty(K, 9, dtype=torch.float32, device=dev())
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    obj = torch.empty(iters + 1, dtype=torch.float64, device=dev())
    ws = kq.workspace(n, K, dev())
    run = kq.kq_fit_codebook(to_dev(W), to_dev(C0), iters, C, idx, counts, obj, ws, flags=flags)
    if stats is not None:  # the pruned passes' work, read before any other call on ws
        stats.extend(kq.kq_fit_prune_stats(ws))
    st, _ = kq.kq_device_status(ws)
    assert st == 0
    return (C.cpu().numpy(), idx.cpu().numpy(), counts.cpu().numpy(), obj.cpu().numpy()), run


def _separated(n, P, seed):
    # n kernels around P well-separated prototypes (noise 1e-3 of their spread): no
    # near-ties, and Lloyd reaches a fixed point within a few iterations
    protos = synth.random_kernels(P, 9, seed, 1.0)
    which = synth.below(synth.stream_key(seed, 5), n, P)
    return (protos[which] + synth.random_kernels(n, 9, seed + 1, 1e-3)).astype(np.float32)


@pytest.mark.parametrize("case", ["one_launch", "tensor_cores", "layer"])
def test_fit_stop_on_stable(case):
    if case == "layer":
        lay, W, C0 = _layer(4, 0)  # ResNet-18 conv 64x64, K = 1024: multi-launch path
        iters = 30
    else:
        n, K = (6000, 64) if case == "one_launch" else (40000, 4096)
        W = _separated(n, 2 * K, 31 if case == "one_launch" else 32)
        C0 = W[:K].copy()
        iters = 40
    full, run_full = _gpu_fit_run(W, C0, iters, 0)
    stop, run = _gpu_fit_run(W, C0, iters, kq.STOP_ON_STABLE)
    # a fixed point repeats itself: every output is that of all iterations, bit for bit
    assert run_full == iters and 0 <= run <= iters
    for a, b in zip(full, stop):
        assert bits_equal(a, b)
    if case == "layer":
        return
    # the oracle's own fixed point: the first assignment equal to the previous one
    C, prev, t_ref = C0, None, iters
    for t in range(iters):
        idx, _ = oracle.assign(W, C, threads=THREADS)
        if prev is not None and np.array_equal(idx, prev):
            t_ref = t
            break
        C, _ = oracle.update(W, idx, C)
        prev = idx
    assert run == t_ref < iters


@pytest.mark.parametrize("iters", [0, 1, 2])
@pytest.mark.parametrize("shape", ["one_launch", "multi_launch"])
def test_fit_stop_on_stable_short_fits(shape, iters):
    # no assignment can repeat before the second one: the flag changes nothing
    W = _separated(6000, 128, 33) if shape == "one_launch" else _separated(20000, 1024, 34)
    K = 64 if shape == "one_launch" else 1024
    C0 = W[:K].copy()
    full, run_full = _gpu_fit_run(W, C0, iters, 0)
    stop, run = _gpu_fit_run(W, C0, iters, kq.STOP_ON_STABLE)
    assert run_full == iters and run == iters
    for a, b in zip(full, stop):
        assert bits_equal(a, b)


def test_layers_on_concurrent_streams_match_sequential():
    # A network's layers are independent problems: fitted, quantised and recovered on
    # their own streams with their own workspaces, concurrently, they give the
    # sequential results bit for bit (one-launch fits, tensor-core and CUDA-core
    # assigns, cooperative level fits sharing the GPU).
    picks = [_layer(3, 0), _layer(3, 2), _layer(3, 5), _layer(4, 0)]
    T = 5

    def run(lay, W, C0, stream):
        n, K = W.shape[0], C0.shape[0]
        with torch.cuda.stream(stream):
            Wd, Cd = to_dev(W), to_dev(C0)
            o = {"C": torch.empty(K, 9, device=dev()), "idx": torch.empty(n, dtype=torch.int32, device=dev()),
                 "counts": torch.empty(K, dtype=torch.int32, device=dev()),
                 "obj": torch.empty(T + 1, dtype=torch.float64, device=dev()),
                 "levels": torch.empty(64, device=dev()), "codes": torch.empty(K, 9, dtype=torch.uint8, device=dev()),
                 "Wr": torch.empty(n, 9, device=dev())}
            ws = kq.workspace(n, K, dev())
            kq.kq_fit_codebook(Wd, Cd, T, o["C"], o["idx"], o["counts"], o["obj"], ws)
            kq.kq_quantize_codebook_6bit(o["C"], o["counts"], 100, o["levels"], o["codes"], None, ws)
            kq.kq_reconstruct(o["idx"], None, o["codes"], o["levels"], o["Wr"], ws, K=K)
        return o, ws

    seq = []
    for lay, W, C0 in picks:
        o, ws = run(lay, W, C0, torch.cuda.current_stream())
        assert kq.kq_device_status(ws)[0] == 0
        seq.append({k: v.cpu().numpy() for k, v in o.items()})
    streams = [torch.cuda.Stream(device=dev()) for _ in picks]
    conc = [run(lay, W, C0, s) for (lay, W, C0), s in zip(picks, streams)]
    torch.cuda.synchronize()
    for (o, ws), ref in zip(conc, seq):
        assert kq.kq_device_status(ws)[0] == 0
        for k, v in o.items():
            assert bits_equal(v.cpu().numpy(), ref[k]), k


def test_fit_end_to_end_against_oracle():
    lay, W, C0 = _layer(1)
    C_g, idx_g, cnt_g, obj_g = _gpu_fit(W, C0, 10)
    C_r, idx_r, cnt_r, obj_r = oracle.fit(W, C0, 10, threads=THREADS)
    # GPU means are within ~1.5 ulp of the exact mean, the oracle's within 0.5 ulp,
    # so a few centroid entries differ by an ulp; that could flip an exact near-tie,
    # which this seeded input does not have.
    assert np.array_equal(idx_g, idx_r) and np.array_equal(cnt_g, cnt_r)
    check_centroids(C_g, C_r)
    # An ulp-level centroid difference dc changes a distance d = |x - c|^2 by
    # 2|x - c||dc| <= 2 * 2^-23 |c| |x - c|; with |c| / |x - c| of order 10 on
    # these inputs that is ~3e-6 of d per kernel at worst, far less on average.
    np.testing.assert_allclose(obj_g, obj_r, rtol=3e-6)


def test_fit_zero_iterations_and_identity():
    W = synth.random_kernels(500, 9, 13)
    C_g, idx_g, cnt_g, obj_g = _gpu_fit(W, W, 0)
    assert bits_equal(C_g, W) and np.array_equal(idx_g, np.arange(500)) and np.all(cnt_g == 1)
    assert obj_g[0] == 0.0
    C_g, idx_g, cnt_g, obj_g = _gpu_fit(W, W, 2)  # K = n seeded with all kernels is a fixed point
    assert bits_equal(C_g, W) and np.array_equal(idx_g, np.arange(500)) and np.all(obj_g == 0.0)


@pytest.mark.parametrize("cfg,li,flags", [(2, 0, 0), (3, 8, 0), (4, 9, 0), (4, 9, kq.STOP_ON_STABLE),
                                           (4, 9, kq.FIT_PRUNE)])
def test_fit_objective_optional(cfg, li, flags):
    # The objective's sums ride along with other kernels (the finalise, the delta update)
    # or are skipped when no objective is asked for: codebook, indices and counts are
    # the same either way, and the objective is that of a separate pass over the
    # distances (dist_block_sums + sum_blocks order), i.e. the oracle's within 1e-12.
    lay, W, C0 = _layer(cfg, li)
    n, K, T = W.shape[0], C0.shape[0], 4
    out = []
    for with_obj in (True, False):
        C = torch.empty(K, 9, dtype=torch.float32, device=dev())
        idx = torch.empty(n, dtype=torch.int32, device=dev())
        counts = torch.empty(K, dtype=torch.int32, device=dev())
        obj = torch.full((T + 1,), float("nan"), dtype=torch.float64, device=dev()) if with_obj else None
        ws = kq.workspace(n, K, dev())
        kq.kq_fit_codebook(to_dev(W), to_dev(C0), T, C, idx, counts, obj, ws, flags=flags)
        assert kq.kq_device_status(ws)[0] == 0
        out.append((C.cpu().numpy(), idx.cpu().numpy(), counts.cpu().numpy(), None if obj is None else obj.cpu().numpy()))
    (Ca, ia, ca, oa), (Cb, ib, cb, _) = out
    assert bits_equal(Ca, Cb) and np.array_equal(ia, ib) and np.array_equal(ca, cb)
    assert np.all(np.isfinite(oa))
    # the last objective is the final assignment's: the oracle's distances to C, summed
    idx_ref, dist_ref = oracle.assign(W, Ca, threads=THREADS)
    assert check_indices(W, Ca, ia, idx_ref) == 0
    assert oa[-1] == pytest.approx(oracle.objective(dist_ref), rel=1e-12)


def test_fit_deterministic():
    lay, W, C0 = _layer(2)
    a = _gpu_fit(W, C0, 4)
    b = _gpu_fit(W, C0, 4)
    for x, y in zip(a, b):
        assert bits_equal(x, y)


# --------------------------------------------------------------------------- 6-bit quantisation

@pytest.mark.parametrize("K,seed,high", [(1, 1, 5), (16, 2, 300), (256, 3, 600), (5000, 4, 100), (16384, 6, 64),
                                         (20000, 7, 40), (24000, 8, 40), (65536, 5, 128)])
def test_quantize_random_codebooks(K, seed, high):
    C = synth.random_kernels(K, 9, seed, 0.02)
    counts = synth.random_counts(K, seed + 100, high)
    lv_g, cd_g, it_g, st, _ = gpu_quantize(C, counts)
    lv_r, cd_r, it_r = oracle.level_fit(C, counts)
    assert st == 0
    assert bits_equal(lv_g, lv_r) and np.array_equal(cd_g, cd_r) and it_g == it_r


def test_quantize_fitted_codebook():
    lay, W, C0 = _layer(2)
    C, idx, counts, _ = _gpu_fit(W, C0, 5)
    lv_g, cd_g, it_g, st, _ = gpu_quantize(C, counts)
    lv_r, cd_r, it_r = oracle.level_fit(C, counts)
    assert st == 0 and bits_equal(lv_g, lv_r) and np.array_equal(cd_g, cd_r) and it_g == it_r


@pytest.mark.parametrize("case", ["zero_iters", "no_weights", "constant", "few_values", "max_iters_1"])
def test_quantize_edge_cases(case):
    C = synth.random_kernels(300, 9, 21, 0.05)
    counts = synth.random_counts(300, 22, 40)
    iters = 100
    if case == "zero_iters":
        iters = 0
    elif case == "no_weights":
        counts[:] = 0
    elif case == "constant":
        C[:] = 0.25
    elif case == "few_values":
        C = (np.arange(300 * 9) % 5).astype(np.float32).reshape(300, 9)
    elif case == "max_iters_1":
        iters = 1
    lv_g, cd_g, it_g, st, _ = gpu_quantize(C, counts, iters)
    lv_r, cd_r, it_r = oracle.level_fit(C, counts, iters)
    assert st == 0 and bits_equal(lv_g, lv_r) and np.array_equal(cd_g, cd_r) and it_g == it_r


def test_quantize_negative_count_flagged():
    # a negative count is flagged and treated as 0
    C = synth.random_kernels(1000, 9, 23, 0.05)
    counts = synth.random_counts(1000, 24, 40)
    counts[5] = -3
    lv_g, cd_g, it_g, st, flags = gpu_quantize(C, counts)
    lv_r, cd_r, it_r = oracle.level_fit(C, np.maximum(counts, 0))
    assert st == 5 and flags & kq.FLAG_INDEX_RANGE
    assert bits_equal(lv_g, lv_r) and np.array_equal(cd_g, cd_r) and it_g == it_r


# --------------------------------------------------------------------------- reconstruction

@pytest.mark.parametrize("n,K", [(1, 1), (31, 5), (4096, 16), (100001, 256), (544775, 4096), (1000003, 65536),
                                 (4194304, 65536)])
def test_reconstruct(n, K):
    # ragged ends, and sizes whose last round of chunk pairs leaves warps idle
    C = synth.random_kernels(K, 9, K, 0.05)
    idx = synth.below(synth.stream_key(n, 2), n, K).astype(np.int32)
    counts = np.bincount(idx, minlength=K).astype(np.int32)
    Wk, st, _ = gpu_reconstruct(idx, C)
    assert st == 0 and bits_equal(Wk, oracle.reconstruct(idx, C))
    lv, cd, _ = oracle.level_fit(C, counts, 20)
    Wkc, st, _ = gpu_reconstruct(idx, C, cd, lv)
    assert st == 0 and bits_equal(Wkc, oracle.reconstruct(idx, C, cd, lv))


def gpu_quantize_reconstruct(idx, C, levels, want_codes=True):
    n, K = idx.shape[0], C.shape[0]
    Wr = torch.empty(n, 9, dtype=torch.float32, device=dev())
    codes = torch.empty(K, 9, dtype=torch.uint8, device=dev()) if want_codes else None
    ws = kq.workspace(n, K, dev())
    kq.kq_quantize_reconstruct(to_dev(idx.astype(np.int32)), to_dev(C), to_dev(levels), codes, Wr, ws)
    st, flags = kq.kq_device_status(ws)
    return Wr.cpu().numpy(), (codes.cpu().numpy() if want_codes else None), st, flags


@pytest.mark.parametrize("n,K,case", [(1, 1, "fit"), (31, 5, "fit"), (4096, 16, "fit"), (100001, 256, "fit"),
                                      (4194304, 65536, "fit"), (50000, 3000, "shuffled"), (50000, 3000, "duplicates"),
                                      (50000, 3000, "no_codes")])
def test_quantize_reconstruct_fused(n, K, case):
    # one launch: encode the float codebook against the levels, then gather; equal to
    # encoding with the oracle and reconstructing from those codes
    C = synth.random_kernels(K, 9, K + 7, 0.05)
    idx = synth.below(synth.stream_key(n + 9, 2), n, K).astype(np.int32)
    counts = np.bincount(idx, minlength=K).astype(np.int32)
    levels, _, _ = oracle.level_fit(C, counts, 20)
    if case == "shuffled":  # unsorted levels: the 64-way scan
        levels = levels[synth.below(synth.stream_key(11, 2), 64, 64).argsort(kind="stable")]
    elif case == "duplicates":  # ties between equal levels go to the lower index
        levels = np.repeat(levels[::4], 4).astype(np.float32)
    codes_ref = oracle.encode(C.reshape(-1), levels).reshape(K, 9)
    Wr, codes, st, _ = gpu_quantize_reconstruct(idx, C, levels, want_codes=case != "no_codes")
    assert st == 0
    assert bits_equal(Wr, oracle.reconstruct(idx, C, codes_ref, levels))
    if case != "no_codes":
        assert np.array_equal(codes, codes_ref)


def test_quantize_reconstruct_flags():
    C = synth.random_kernels(10, 9, 3)
    idx = np.arange(100, dtype=np.int32) % 10
    idx[7] = 10
    levels = np.linspace(-1, 1, 64).astype(np.float32)
    Wr, _, st, flags = gpu_quantize_reconstruct(idx, C, levels)
    assert st == 5 and flags & kq.FLAG_INDEX_RANGE and np.all(Wr[7] == 0)
    C[2, 2] = np.nan
    Wr, codes, st, flags = gpu_quantize_reconstruct(np.arange(10, dtype=np.int32), C, levels)
    assert st == 3 and flags & kq.FLAG_NONFINITE and codes[2, 2] == 0


def test_reconstruct_flags_bad_index_and_code():
    C = synth.random_kernels(10, 9, 1)
    idx = np.arange(100, dtype=np.int32) % 10
    idx[7] = 10
    Wr, st, flags = gpu_reconstruct(idx, C)
    assert st == 5 and flags & kq.FLAG_INDEX_RANGE and np.all(Wr[7] == 0)
    codes = np.zeros((10, 9), np.uint8)
    codes[3, 4] = 64
    Wr, st, flags = gpu_reconstruct(np.arange(10, dtype=np.int32), C, codes, np.arange(64, dtype=np.float32))
    assert st == 5 and flags & kq.FLAG_CODE_RANGE and Wr[3, 4] == 0


def test_init_codebook():
    lay = synth.workload(2).layers[0]
    W, sel = synth.layer_inputs(lay)
    C0 = torch.empty(lay.K, 9, dtype=torch.float32, device=dev())
    ws = kq.workspace(lay.n, lay.K, dev())
    kq.kq_init_codebook(to_dev(W), to_dev(sel), C0, ws)
    assert kq.kq_device_status(ws)[0] == 0
    assert bits_equal(C0.cpu().numpy(), oracle.gather_rows(W, sel))


# --------------------------------------------------------------------------- kernel trace

def test_trace_times_every_launch_of_a_fit():
    # a fit on the tensor-core path, traced: one record per launch, in launch order,
    # each with a kernel name and a positive device time (ResNet-18 conv5: n = 8192,
    # K = 2048, multi-launch fit on the tensor-core path, no pilot pass)
    lay, W, C0 = _layer(4, 4)
    n, K = W.shape[0], C0.shape[0]
    Wd, Cd = to_dev(W), to_dev(C0)
    C = torch.empty_like(Cd)
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    ws = kq.workspace(n, K, dev())
    kq.kq_fit_codebook(Wd, Cd, 2, C, idx, counts, None, ws)  # warm-up
    torch.cuda.synchronize()
    kq.kq_trace_start(256)
    l0 = kq.kq_kernel_launches()
    kq.kq_fit_codebook(Wd, Cd, 2, C, idx, counts, None, ws)
    launched = kq.kq_kernel_launches() - l0
    kq.kq_trace_stop()
    kq.kq_fit_codebook(Wd, Cd, 1, C, idx, counts, None, ws)  # not recorded
    trace = kq.kq_trace_read()
    assert kq.kq_device_status(ws)[0] == 0
    assert len(trace) == launched > 0
    names = [name for name, _ in trace]
    assert names.count("assign_tc_kernel") == 3  # two updates, then the final assignment
    assert all(ms > 0 for _, ms in trace)
    assert names[-1] == "histogram_kernel"  # the final assignment's cluster sizes
    with pytest.raises(kq.KQError):
        kq.kq_trace_start(0)


# --------------------------------------------------------------------------- pruned fit

def _fit_both(W, C0, iters):
    # both fits, and the pruned one's work: every assignment of the fit runs pruned, so
    # its passes hold (iters + 1) x blocks x tiles (256-kernel block, 256-codeword tile)
    # pairs, of which the first pass (no bounds yet) processes all
    n, K = W.shape[0], C0.shape[0]
    per_pass = -(-n // 256) * -(-K // 256)
    work, none = [], []
    pruned, run_p = _gpu_fit_run(W, C0, iters, kq.FIT_PRUNE, work)
    plain, run_q = _gpu_fit_run(W, C0, iters, 0, none)
    tiles_run, tiles_all = work
    assert tiles_all == (iters + 1) * per_pass
    assert per_pass <= tiles_run <= tiles_all
    assert none == [0, 0]  # a fresh workspace, a fit without pruning
    return pruned, plain, tiles_run / tiles_all


@pytest.mark.parametrize("case", ["k4096", "k4097_ragged_tile", "k12345", "dup_codewords", "resnet_k16384",
                                  "iters0", "iters1"])
def test_fit_pruned_matches_plain(case):
    # Tile pruning (k-d codebook order, per-tile bound records, skipped tiles) only
    # changes speed: every output equals the plain fit's, bit for bit.
    iters = 4
    if case == "resnet_k16384":
        lay, W, C0 = _layer(4, 9)  # 256 -> 256, n = 65536, K = 16384
    else:
        n = {"k4096": 40000, "k4097_ragged_tile": 41000, "k12345": 60000, "dup_codewords": 40000,
             "iters0": 40000, "iters1": 40000}[case]
        K = {"k4097_ragged_tile": 4097, "k12345": 12345}.get(case, 4096)
        lay = synth.Layer("t", 64, n // 64, K, 4 * K, 70 + len(case))
        W = synth.conv_weights(lay)  # 64 (n // 64) kernels
        C0 = oracle.gather_rows(W, synth.init_selection(W.shape[0], K, 71 + len(case)))
        if case == "dup_codewords":
            # exact ties between codewords far apart in the original numbering
            C0[[5, 700, 2900, 4000]] = C0[[3000, 4095, 12, 64]]
        iters = {"iters0": 0, "iters1": 1}.get(case, iters)
    pruned, plain, _ = _fit_both(W, C0, iters)
    for a, b in zip(pruned, plain):
        assert bits_equal(a, b)


def test_fit_pruned_stepwise_against_oracle():
    # ResNet-18 128 -> 256 layer (n = 32768, K = 8192): the pruned fit's every step
    # against the oracle from the same codebook, and a 3-iteration fit equal to the
    # chained one-iteration fits
    lay, W, C0 = _layer(4, 8)
    C = C0
    for t in range(3):
        (C_next, idx_next, cnt_next, obj), _ = _gpu_fit_run(W, C, 1, kq.FIT_PRUNE)
        idx_ref, dist_ref = oracle.assign(W, C, threads=THREADS)
        C_ref, _ = oracle.update(W, idx_ref, C)
        check_centroids(C_next, C_ref)
        assert obj[0] == pytest.approx(oracle.objective(dist_ref), rel=1e-12)
        i2, d2 = oracle.assign(W, C_next, threads=THREADS)
        assert check_indices(W, C_next, idx_next, i2) == 0
        assert np.array_equal(cnt_next, np.bincount(idx_next, minlength=lay.K))
        C = C_next
    (C_T, idx_T, _, obj_T), _ = _gpu_fit_run(W, C0, 3, kq.FIT_PRUNE)
    assert bits_equal(C_T, C)
    i3, _ = oracle.assign(W, C_T, threads=THREADS)
    assert check_indices(W, C_T, idx_T, i3) == 0
    assert np.all(obj_T[1:] <= obj_T[:-1] * (1 + 1e-6))


def test_fit_pruned_full_size_stress():
    # the stress layer (n = 4,194,304, K = 65,536: 256 tiles, the largest pruned
    # codebook), 3 iterations, pruned and plain bit for bit; sampled rows of the
    # final assignment against the oracle
    lay, W, C0 = _layer(5)
    pruned, plain, frac = _fit_both(W, C0, 3)
    for a, b in zip(pruned, plain):
        assert bits_equal(a, b)
    assert frac < 1.0  # the later passes skip tiles
    C_T, idx_T = pruned[0], pruned[1]
    rows = np.sort(synth.below(synth.stream_key(lay.seed, 11), 2048, lay.n))
    idx_ref, _ = oracle.assign(W[rows], C_T, threads=THREADS)
    assert check_indices(W, C_T, idx_T[rows], idx_ref, rows) == 0
