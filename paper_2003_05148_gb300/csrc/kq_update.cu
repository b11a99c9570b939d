// kq_update.cu -- update step of KQ's k-means (Sec. 3.1, Eq. 1): c_k = mean of S_k.
//
// Deterministic without floating-point atomics: every coordinate of every kernel
// is converted to an int64 fixed-point number q = rint(v * 2^S) (integer
// operations only, see fixed_rn) and added with integer atomics
// (red.global.add.u64), which are associative, so the sums do not depend on the
// order the hardware applies them in. With a bound B >= |v| for every value and
// n * B = f * 2^e (f in [0.5, 1)), S = 62 - e keeps every sum below 2^63.
//
// Where B comes from:
//  - exact: B = max|W| from a pass over W (kq_fit_codebook does this once per fit);
//  - guess (kq_update_centroids): B = 256 * max|C_prev|, read from the small
//    codebook instead of W. Every value is checked against B while it is added; if
//    any finite |w| > B, a cooperative fallback pass clears the sums, takes max|W|
//    and accumulates again with that exact bound. Either way the sums are exact
//    fixed-point sums at the scale recorded in the workspace header.
//
// The accumulator of codeword k is one 128-byte line: 9 coordinate sums and the
// member count (layout of the adds: see accumulate_rows). The throughput limit is
// the atomic path, not HBM: about 1.4 64-bit RED lanes per clock per SM get
// through L1TEX (86% busy in ncu), 10 lanes per kernel.
#include "kq_internal.cuh"

namespace kq {

constexpr int U_THREADS = 256;
constexpr int SCALE_INVALID = -100000;
constexpr float GUESS_FACTOR = 256.f;
constexpr float F32_MAX = 3.402823466e38f;

// Scale exponent for n values bounded by B; SCALE_INVALID when B is zero,
// negative, infinite or NaN.
__device__ __forceinline__ int update_scale(float B, int64_t n) {
    if (!(B > 0.f) || !(B <= F32_MAX)) return SCALE_INVALID;
    int e;
    frexp((double)n * (double)B, &e);
    return 62 - e;
}

// Adds the kernels of 32-kernel chunks it0, it0 + step, ... into the accumulators
// at scale S. In pass i a lane handles float lane + 32 i of the chunk (coalesced
// loads straight from global memory): kernel rr[i] of the chunk, coordinate jj[i];
// that kernel's codeword comes from lane rr[i] by shuffle. All 32 lanes add in
// every pass; each lane also adds one count.
// With `check`, a finite value above B sets the violation flag (the exact fallback
// pass then redoes the sums).
__device__ __forceinline__ void accumulate_rows(const float *__restrict__ W, int64_t n, const int32_t *__restrict__ idx,
                                                int32_t K, int S, float B, bool check, unsigned long long *acc,
                                                Header *hdr, int64_t it0, int64_t step, bool do_tail) {
    const int lane = threadIdx.x & 31;
    int rr[D], jj[D];
#pragma unroll
    for (int i = 0; i < D; ++i) {
        rr[i] = (lane + 32 * i) / D;
        jj[i] = (lane + 32 * i) - D * rr[i];
    }
    bool bad_idx = false, too_big = false, nonfinite = false;
    const int64_t nchunks = n / 32;
    // Chunks are visited last-to-first: a max|W| pass that just streamed W front to
    // back leaves the tail of W in L2.
    for (int64_t it = it0; it < nchunks; it += step) {
        const int64_t r0 = (nchunks - 1 - it) * 32;
        const float *src = W + r0 * D;
        float v[D];
#pragma unroll
        for (int i = 0; i < D; ++i) v[i] = __ldg(src + lane + 32 * i);
        const int32_t myk = __ldcs(idx + r0 + lane);
        const bool okk = (uint32_t)myk < (uint32_t)K;
        bad_idx |= !okk;
#pragma unroll
        for (int i = 0; i < D; ++i) {
            const float a = fabsf(v[i]);
            nonfinite |= !(a <= F32_MAX);
            too_big |= check && a > B && a <= F32_MAX;
            const int32_t k = __shfl_sync(0xffffffffu, myk, rr[i]);
            if ((uint32_t)k < (uint32_t)K)
                atomicAdd(acc + (int64_t)k * ACC_WORDS + jj[i], (unsigned long long)fixed_rn(v[i], S));
        }
        if (okk) atomicAdd(acc + (int64_t)myk * ACC_WORDS + D, 1ull);
    }
    // ragged end (< 32 kernels): one thread per kernel
    if (do_tail) {
        const int64_t i = nchunks * 32 + threadIdx.x;
        if (threadIdx.x < 32 && i < n) {
            const int32_t k = idx[i];
            if ((uint32_t)k < (uint32_t)K) {
#pragma unroll
                for (int j = 0; j < D; ++j) {
                    const float x = W[i * D + j];
                    const float a = fabsf(x);
                    nonfinite |= !(a <= F32_MAX);
                    too_big |= check && a > B && a <= F32_MAX;
                    atomicAdd(acc + (int64_t)k * ACC_WORDS + j, (unsigned long long)fixed_rn(x, S));
                }
                atomicAdd(acc + (int64_t)k * ACC_WORDS + D, 1ull);
            } else {
                bad_idx = true;
            }
        }
    }
    if (bad_idx) set_flag(&hdr->status, KQ_FLAG_INDEX_RANGE);
    if (nonfinite) set_flag(&hdr->status, KQ_FLAG_NONFINITE);
    if (too_big) atomicExch(&hdr->upd_violation, 1u);
}

__global__ void __launch_bounds__(256) maxabs_kernel(const float *__restrict__ W, int64_t count,
                                                     uint32_t *maxabs_bits, uint32_t *status) {
    float m = 0.f;
    bool ok = true;
    const int64_t n4 = count / 4;
    const float4 *W4 = reinterpret_cast<const float4 *>(W);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (; v + 3 * stride < n4; v += 4 * stride) {  // four independent loads in flight per thread
        float4 t[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) t[u] = __ldg(W4 + v + u * stride);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            ok &= isfinite(t[u].x) & isfinite(t[u].y) & isfinite(t[u].z) & isfinite(t[u].w);
            m = fmaxf(m, fmaxf(fmaxf(fabsf(t[u].x), fabsf(t[u].y)), fmaxf(fabsf(t[u].z), fabsf(t[u].w))));
        }
    }
    for (; v < n4; v += stride) {
        const float4 t = __ldg(W4 + v);
        ok &= isfinite(t.x) & isfinite(t.y) & isfinite(t.z) & isfinite(t.w);
        m = fmaxf(m, fmaxf(fmaxf(fabsf(t.x), fabsf(t.y)), fmaxf(fabsf(t.z), fabsf(t.w))));
    }
    for (int64_t u = n4 * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < count; u += stride) {
        const float t = W[u];
        ok &= isfinite(t);
        m = fmaxf(m, fabsf(t));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if (!__all_sync(0xffffffffu, ok) && (threadIdx.x & 31) == 0) set_flag(status, KQ_FLAG_NONFINITE);
    if ((threadIdx.x & 31) == 0) atomicMax(maxabs_bits, __float_as_uint(m));  // m >= +0: bits order as values
}

// Clears the accumulators; in guess mode also reduces max|C_prev| into upd_bound.
__global__ void __launch_bounds__(256) update_prepare_kernel(const float *__restrict__ C_prev, int32_t K,
                                                             unsigned long long *__restrict__ acc, Header *hdr,
                                                             bool guess) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    ulonglong2 *a2 = reinterpret_cast<ulonglong2 *>(acc);
    for (int64_t w = t0; w < (int64_t)K * ACC_WORDS / 2; w += stride) a2[w] = make_ulonglong2(0ull, 0ull);
    if (!guess) return;
    float m = 0.f;
    for (int64_t e = t0; e < (int64_t)K * D; e += stride) {
        const float a = fabsf(C_prev[e]);
        m = a <= F32_MAX ? fmaxf(m, a) : __int_as_float(0x7f800000);  // non-finite: no usable guess
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((threadIdx.x & 31) == 0) atomicMax(&hdr->upd_bound, __float_as_uint(m));
}

__global__ void __launch_bounds__(U_THREADS)
accumulate_kernel(const float *__restrict__ W, int64_t n, const int32_t *__restrict__ idx, int32_t K, Header *hdr,
                  unsigned long long *__restrict__ acc, bool guess) {
    const float B = guess ? __uint_as_float(__ldcg(&hdr->upd_bound)) * GUESS_FACTOR  // power-of-two scaling
                          : __uint_as_float(__ldcg(&hdr->maxabs_bits));
    int S = update_scale(B, n);
    if (S == SCALE_INVALID) {
        if (guess) {  // no usable guess: leave everything to the exact pass
            if (blockIdx.x == 0 && threadIdx.x == 0) atomicExch(&hdr->upd_violation, 1u);
            return;
        }
        S = 0;  // all-zero W (nothing to scale) or non-finite W (flagged)
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) hdr->upd_scale = S;
    accumulate_rows(W, n, idx, K, S, B, guess, acc, hdr, (int64_t)blockIdx.x * (U_THREADS / 32) + (threadIdx.x >> 5),
                    (int64_t)gridDim.x * (U_THREADS / 32), blockIdx.x == 0);
}

// Runs only when the guessed bound was violated (the flag is final: the accumulate
// kernel has completed). Cooperative launch: all CTAs are resident, so they can
// meet at the bounded grid barrier between clearing/measuring and re-adding.
__global__ void __launch_bounds__(U_THREADS)
update_fallback_kernel(const float *__restrict__ W, int64_t n, const int32_t *__restrict__ idx, int32_t K,
                       Header *hdr, unsigned long long *__restrict__ acc) {
    if (__ldcg(&hdr->upd_violation) == 0u) return;  // the common case: nothing to do
    unsigned epoch = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    ulonglong2 *a2 = reinterpret_cast<ulonglong2 *>(acc);
    for (int64_t w = t0; w < (int64_t)K * ACC_WORDS / 2; w += stride) a2[w] = make_ulonglong2(0ull, 0ull);
    float m = 0.f;
    for (int64_t e = t0; e < n * D; e += stride) {
        const float a = fabsf(W[e]);
        m = a <= F32_MAX ? fmaxf(m, a) : m;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((threadIdx.x & 31) == 0) atomicMax(&hdr->maxabs_bits, __float_as_uint(m));
    if (!grid_barrier(hdr, gridDim.x, epoch)) return;
    const float B = __uint_as_float(__ldcg(&hdr->maxabs_bits));
    int S = update_scale(B, n);
    if (S == SCALE_INVALID) S = 0;
    if (blockIdx.x == 0 && threadIdx.x == 0) hdr->upd_scale = S;
    accumulate_rows(W, n, idx, K, S, B, false, acc, hdr, (int64_t)blockIdx.x * (U_THREADS / 32) + (threadIdx.x >> 5),
                    (int64_t)gridDim.x * (U_THREADS / 32), blockIdx.x == 0);
}

// c_k = (sum * 2^-S) / z_k in fp32 (keep C_prev when z_k = 0); clears the
// accumulator row for the next call unless the sums are kept (the fit's next update
// only moves the rows whose codeword changed). fp32 arithmetic (GB300's fp64 rate is
// low): sum -> fp32, exact power-of-two scaling, one IEEE division; within ~1.5 ulp
// of the exact mean.
// obj (nullable): CTA 0 also writes the objective of the assignment the update came
// from, the sum of its nblocks block sums in the order of sum_blocks_kernel (256
// strided partial sums, xor butterflies within the warps, the eight warp sums in order).
__global__ void __launch_bounds__(256)
finalize_kernel(unsigned long long *__restrict__ acc, int32_t K, const Header *hdr, const float *C_prev,
                float *C_next, int32_t *__restrict__ counts, bool keep, const double *__restrict__ blocksum,
                int nblocks, double *obj) {
    if (obj && blockIdx.x == 0) {
        __shared__ double wsum[8];
        objective_sum_256(blocksum, nblocks, obj, wsum);
    }
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    finalize_codeword(acc, k, __ldcg(&hdr->upd_scale), C_prev, C_next, counts, keep);
}

// The sums of idx_old (in acc, at the scale in hdr->upd_scale) become those of
// idx_new: a row whose codeword changed is subtracted from the old codeword's sums
// and added to the new one's (the same fixed-point values the full accumulation
// adds, so the result is the full accumulation's, bit for bit; integer arithmetic
// is exact whatever the order). Rows that kept their codeword cost two index loads.
// dist (nullable): the assignment's distances, whose per-256-row sums go to
// blocksum[b] exactly as dist_block_sums_kernel computes them (the CTA works on whole
// 256-row blocks, one thread per row).
__global__ void __launch_bounds__(256)
accumulate_delta_kernel(const float *__restrict__ W, int64_t n, const int32_t *__restrict__ idx_old,
                        const int32_t *__restrict__ idx_new, int32_t K, Header *hdr,
                        unsigned long long *__restrict__ acc, uint32_t *moved, const float *__restrict__ dist,
                        double *__restrict__ blocksum) {
    __shared__ F2 ws[8];
    const int S = __ldcg(&hdr->upd_scale);
    bool bad = false, any = false;
    const int64_t nblk = (n + 255) / 256;
    for (int64_t blk = blockIdx.x; blk < nblk; blk += gridDim.x) {  // block-uniform trip count
        const int64_t i = blk * 256 + threadIdx.x;
        if (dist) {
            const F2 v = f2_warp_sum(i < n ? __ldcs(dist + i) : 0.f);
            if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = v;
            __syncthreads();
            if (threadIdx.x == 0) {
                F2 t{0.f, 0.f};
                for (int w = 0; w < 8; ++w) t = f2_add(t, ws[w]);
                blocksum[blk] = f2_to_double(t);
            }
            __syncthreads();  // ws is the next block's
        }
        if (i >= n) continue;
        const int32_t a = __ldcs(idx_old + i), b = __ldcs(idx_new + i);
        if (a == b) continue;
        any = true;
        if ((uint32_t)a >= (uint32_t)K || (uint32_t)b >= (uint32_t)K) {
            bad = true;
            continue;
        }
        unsigned long long *ra = acc + (int64_t)a * ACC_WORDS, *rb = acc + (int64_t)b * ACC_WORDS;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            const unsigned long long q = (unsigned long long)fixed_rn(W[i * D + j], S);
            atomicAdd(rb + j, q);
            atomicAdd(ra + j, 0ull - q);
        }
        atomicAdd(rb + D, 1ull);
        atomicAdd(ra + D, ~0ull);  // - 1
    }
    if (bad) set_flag(&hdr->status, KQ_FLAG_INDEX_RANGE);
    if (moved && __any_sync(0xffffffffu, any) && (threadIdx.x & 31) == 0) atomicOr(moved, 1u);
}

cudaError_t launch_accumulate_delta(const float *W, int64_t n, const int32_t *idx_old, const int32_t *idx_new,
                                    int32_t K, Header *hdr, unsigned long long *acc, int num_sms, cudaStream_t s,
                                    uint32_t *moved, const float *dist, double *blocksum, int *nblocksum) {
    int64_t blocks = (n + 255) / 256;
    if (dist) *nblocksum = (int)blocks;
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    accumulate_delta_kernel<<<(unsigned)blocks, 256, 0, s>>>(W, n, idx_old, idx_new, K, hdr, acc, moved, dist,
                                                             blocksum);
    launch_end(s, "accumulate_delta_kernel");
    return cudaGetLastError();
}

__global__ void __launch_bounds__(256) fill_objective_kernel(double *obj, int32_t from, int32_t to) {
    const double v = obj[from];
    for (int64_t j = (int64_t)from + 1 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j <= to;
         j += (int64_t)gridDim.x * blockDim.x)
        obj[j] = v;
}

cudaError_t launch_fill_objective(double *obj, int32_t from, int32_t to, cudaStream_t s) {
    if (to <= from) return cudaSuccess;
    int64_t blocks = ((int64_t)to - from + 255) / 256;
    if (blocks > 1024) blocks = 1024;
    launch_begin(s);
    fill_objective_kernel<<<(unsigned)blocks, 256, 0, s>>>(obj, from, to);
    launch_end(s, "fill_objective_kernel");
    return cudaGetLastError();
}

// counts[k] = #{i : idx[i] == k} with integer atomics (order-independent).
__global__ void __launch_bounds__(256) histogram_kernel(const int32_t *__restrict__ idx, int64_t n, int32_t K,
                                                        int32_t *counts, uint32_t *status) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int32_t k = __ldcs(idx + i);
        if ((uint32_t)k < (uint32_t)K)
            atomicAdd(counts + k, 1);
        else
            set_flag(status, KQ_FLAG_INDEX_RANGE);
    }
}

cudaError_t launch_histogram(const int32_t *idx, int64_t n, int32_t K, int32_t *counts, uint32_t *status,
                             int num_sms, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(counts, 0, (size_t)K * sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    histogram_kernel<<<(unsigned)blocks, 256, 0, s>>>(idx, n, K, counts, status);
    launch_end(s, "histogram_kernel");
    return cudaGetLastError();
}

cudaError_t launch_maxabs(const float *W, int64_t count, uint32_t *maxabs_bits, uint32_t *status, int num_sms,
                          cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(maxabs_bits, 0, sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    int64_t blocks = (count / 4 + 255) / 256;
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    maxabs_kernel<<<(unsigned)blocks, 256, 0, s>>>(W, count, maxabs_bits, status);
    launch_end(s, "maxabs_kernel");
    return cudaGetLastError();
}

cudaError_t launch_update_prepare(const float *C_prev, int32_t K, unsigned long long *acc, Header *hdr,
                                  bool guess_from_codebook, cudaStream_t s) {
    // scale state (bound, violation flag, scale) and the fallback's barrier words
    cudaError_t e = cudaMemsetAsync(&hdr->upd_bound, 0, 3 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(&hdr->barrier, 0, 2 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    if (guess_from_codebook) {
        e = cudaMemsetAsync(&hdr->maxabs_bits, 0, sizeof(uint32_t), s);
        if (e != cudaSuccess) return e;
    }
    int64_t blocks = ((int64_t)K * ACC_WORDS / 2 + 255) / 256;
    if (blocks > 4 * 152) blocks = 4 * 152;
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    update_prepare_kernel<<<(unsigned)blocks, 256, 0, s>>>(C_prev, K, acc, hdr, guess_from_codebook);
    launch_end(s, "update_prepare_kernel");
    return cudaGetLastError();
}

cudaError_t launch_accumulate(const float *W, int64_t n, const int32_t *idx, int32_t K, Header *hdr,
                              unsigned long long *acc, bool guess, int num_sms, cudaStream_t s) {
    const int64_t chunks = n / 32 + 1;
    int64_t blocks = (chunks + U_THREADS / 32 - 1) / (U_THREADS / 32);
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    accumulate_kernel<<<(unsigned)blocks, U_THREADS, 0, s>>>(W, n, idx, K, hdr, acc, guess);
    launch_end(s, "accumulate_kernel");
    return cudaGetLastError();
}

cudaError_t launch_update_fallback(const float *W, int64_t n, const int32_t *idx, int32_t K, Header *hdr,
                                   unsigned long long *acc, int num_sms, cudaStream_t s) {
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, update_fallback_kernel, U_THREADS, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const unsigned blocks = (unsigned)num_sms;  // one CTA per SM: co-resident by construction
    void *params[] = {(void *)&W, (void *)&n, (void *)&idx, (void *)&K, (void *)&hdr, (void *)&acc};
    launch_begin(s);
    e = cudaLaunchCooperativeKernel((const void *)update_fallback_kernel, dim3(blocks), dim3(U_THREADS), params, 0, s);
    if (e != cudaSuccess) return e;
    launch_end(s, "update_fallback_kernel");
    return cudaGetLastError();
}

cudaError_t launch_finalize(unsigned long long *acc, int32_t K, const Header *hdr, const float *C_prev,
                            float *C_next, int32_t *counts, cudaStream_t s, bool keep_sums, const double *blocksum,
                            int nblocks, double *obj) {
    launch_begin(s);
    finalize_kernel<<<(K + 255) / 256, 256, 0, s>>>(acc, K, hdr, C_prev, C_next, counts, keep_sums, blocksum,
                                                     nblocks, obj);
    launch_end(s, "finalize_kernel");
    return cudaGetLastError();
}

}  // namespace kq
