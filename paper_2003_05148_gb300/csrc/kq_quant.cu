// kq_quant.cu -- 6-bit quantisation by 64-level 1-D k-means (Sec. 3.2) on sm_103a:
// of the kernel codebook (the K*9 codebook scalars, weight of a scalar = appearance
// count z_k of its codeword) and of fully-connected layers (any m scalars, weight 1).
//
// One cooperative launch runs the whole iteration: each CTA assigns a grid-stride
// slice of scalars to the nearest level (levels held in shared memory),
// accumulates per-level (weight, weight * fixed-point value) sums in per-warp
// shared int64 atomics, flushes them with global int64 atomics, and meets the
// other CTAs at a bounded grid barrier; after it every CTA computes the same new
// levels from the same integer sums. Integer sums make the result independent of
// the order of the atomics, so the levels and codes are bit-identical from run to
// run and to an exact-arithmetic CPU reference.
//
// Per-iteration global state is triple buffered (iteration it accumulates into
// slot it%3 while CTA 0 clears slot (it+1)%3, last read two barriers earlier),
// so one grid barrier per iteration suffices.
#include "kq_internal.cuh"

namespace kq {

constexpr int Q_THREADS = 512;
constexpr int Q_WARPS = Q_THREADS / 32;
struct LevelArgs {
    const float *C;  // the N scalars
    int64_t N;
    const int32_t *counts;  // weight of scalar m: counts[m / 9], or 1 for every scalar when null
    int32_t max_iters;
    float *levels;
    uint8_t *codes;
    int32_t *iters_run;
    Header *hdr;
};

// Nearest of the 64 levels by fp32 |v - level|, lower index on ties (Sec. 3.2 encode).
__device__ __forceinline__ int nearest_level(float v, const float *L) {
    float best = __int_as_float(0x7f800000);
    int bl = 0;
#pragma unroll 16
    for (int l = 0; l < LEVELS; ++l) {
        const float d = fabsf(v - L[l]);
        if (d < best) {
            best = d;
            bl = l;
        }
    }
    return bl;
}

// nearest_level for levels in non-decreasing order, by binary search; the same
// code. With p the last level <= v, d_l = |fl(v - L_l)| is non-increasing on
// [0, p] and non-decreasing on [p, 63] (rounding is monotone), so the minimum is
// d_p or d_{p+1}; the first index holding it (the scan's tie rule) is p + 1 when
// d_{p+1} < d_p, else the start of the run of levels <= p whose distance equals
// d_p, which is a suffix of [0, p]. A minimum of +inf gives 0, as in the scan.
__device__ __forceinline__ int nearest_level_sorted(float v, const float *L) {
    if (v != v) return 0;  // NaN: no distance is below +inf
    int cnt = 0;           // number of levels <= v
#pragma unroll
    for (int step = 32; step > 0; step >>= 1)
        if (L[cnt + step - 1] <= v) cnt += step;
    cnt += L[cnt] <= v;  // cnt could only reach 63 above
    const int p = cnt - 1;
    if (p < 0) return 0;  // every level is above v: distances grow with l
    const float dp = fabsf(v - L[p]);
    if (p < LEVELS - 1 && fabsf(v - L[p + 1]) < dp) return p + 1;
    if (!(dp < __int_as_float(0x7f800000))) return 0;  // the minimum distance is +inf
    if (p == 0 || fabsf(v - L[p - 1]) > dp) return p;
    int f = 0;  // number of levels l < p with d_l > d_p (a prefix)
#pragma unroll
    for (int step = 32; step > 0; step >>= 1)
        if (f + step - 1 < p && fabsf(v - L[f + step - 1]) > dp) f += step;
    return f;
}

// Levels in non-decreasing order (and no NaN), so that nearest_level_sorted applies.
__device__ __forceinline__ bool levels_sorted(const float *L) {
    bool ok = true;
#pragma unroll 8
    for (int l = 0; l < LEVELS - 1; ++l) ok &= L[l] <= L[l + 1];
    return ok;
}

__global__ void __launch_bounds__(Q_THREADS) level_fit_kernel(LevelArgs a) {
    __shared__ float L[LEVELS];
    __shared__ unsigned long long bw[Q_WARPS][LEVELS], bq[Q_WARPS][LEVELS];
    __shared__ int s_changed;
    __shared__ int s_stop;
    __shared__ int s_sorted;
    Header *h = a.hdr;
    const int64_t N = a.N;
    const int warp = threadIdx.x >> 5;
    const int64_t tid0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    unsigned epoch = 0;

    // Phase 0: value ranges, max |v| and total weight.
    {
        float lo_w = __int_as_float(0x7f800000), hi_w = -lo_w, lo_a = lo_w, hi_a = -lo_w, mv = 0.f;
        unsigned long long wt = 0;
        bool ok = true, badc = false;
        for (int64_t m = tid0; m < N; m += stride) {
            const float v = a.C[m];
            int32_t z = a.counts ? a.counts[m / D] : 1;
            if (z < 0) {
                badc = true;
                z = 0;
            }
            if (!isfinite(v)) {
                ok = false;
                continue;
            }
            lo_a = fminf(lo_a, v);
            hi_a = fmaxf(hi_a, v);
            if (z > 0) {
                lo_w = fminf(lo_w, v);
                hi_w = fmaxf(hi_w, v);
                mv = fmaxf(mv, fabsf(v));
                wt += (unsigned long long)z;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            lo_w = fminf(lo_w, __shfl_xor_sync(0xffffffffu, lo_w, o));
            hi_w = fmaxf(hi_w, __shfl_xor_sync(0xffffffffu, hi_w, o));
            lo_a = fminf(lo_a, __shfl_xor_sync(0xffffffffu, lo_a, o));
            hi_a = fmaxf(hi_a, __shfl_xor_sync(0xffffffffu, hi_a, o));
            mv = fmaxf(mv, __shfl_xor_sync(0xffffffffu, mv, o));
            wt += __shfl_xor_sync(0xffffffffu, wt, o);
        }
        const bool all_ok = __all_sync(0xffffffffu, ok), any_bad = __any_sync(0xffffffffu, badc);
        if ((threadIdx.x & 31) == 0) {
            atomicMin(&h->lo_w, f2ord(lo_w));
            atomicMax(&h->hi_w, f2ord(hi_w));
            atomicMin(&h->lo_a, f2ord(lo_a));
            atomicMax(&h->hi_a, f2ord(hi_a));
            atomicMax(&h->maxv_w, __float_as_uint(mv));
            if (wt) atomicAdd(&h->wtotal, wt);
            if (!all_ok) set_flag(&h->status, KQ_FLAG_NONFINITE);
            if (any_bad) set_flag(&h->status, KQ_FLAG_INDEX_RANGE);
        }
    }
    if (!grid_barrier(h, gridDim.x, epoch)) return;

    // Phase 1: initial levels linspace(lo, hi, 64) in fp64, and the fixed-point scale.
    const unsigned long long A = __ldcg(&h->wtotal);
    const bool any = A > 0;
    const float lo = ord2f(__ldcg(any ? &h->lo_w : &h->lo_a));
    const float hi = ord2f(__ldcg(any ? &h->hi_w : &h->hi_a));
    const float M = __uint_as_float(__ldcg(&h->maxv_w));
    int S = 0;
    if (any && M > 0.f) {
        int e;
        frexp(__dmul_rn(__ull2double_rn(A), (double)M), &e);
        S = 62 - e;
    }
    const double down = ldexp(1.0, -S);
    if (threadIdx.x < LEVELS) {
        const double t = __ddiv_rn(__dmul_rn(__dsub_rn((double)hi, (double)lo), (double)threadIdx.x), 63.0);
        L[threadIdx.x] = __double2float_rn(__dadd_rn((double)lo, t));
    }
    __syncthreads();
    if (threadIdx.x == 0) s_sorted = levels_sorted(L);

    int32_t updates = 0;
    for (int32_t it = 0; it < a.max_iters; ++it) {
        const int buf = it % 3, nxt = (it + 1) % 3;
        for (int t = threadIdx.x; t < Q_WARPS * LEVELS; t += Q_THREADS) {
            (&bw[0][0])[t] = 0ull;
            (&bq[0][0])[t] = 0ull;
        }
        if (threadIdx.x == 0) s_changed = 0;
        if (blockIdx.x == 0) {
            if (threadIdx.x < 2 * LEVELS) (&h->lacc[nxt][0][0])[threadIdx.x] = 0ull;
            if (threadIdx.x == 0) h->changed[nxt] = 0u;
        }
        __syncthreads();
        bool changed = false;
        const bool sorted = s_sorted;
        for (int64_t m = tid0; m < N; m += stride) {
            const float v = a.C[m];
            const int code = sorted ? nearest_level_sorted(v, L) : nearest_level(v, L);
            if (it > 0 && a.codes[m] != (uint8_t)code) changed = true;
            a.codes[m] = (uint8_t)code;
            const int32_t z = a.counts ? a.counts[m / D] : 1;
            if (z > 0) {
                const long long q = fixed_rn(v, S);
                atomicAdd(&bw[warp][code], (unsigned long long)z);
                atomicAdd(&bq[warp][code], (unsigned long long)((long long)z * q));
            }
        }
        if (__any_sync(0xffffffffu, changed) && (threadIdx.x & 31) == 0) s_changed = 1;
        __syncthreads();
        if (threadIdx.x < LEVELS) {
            unsigned long long sw = 0ull, sq = 0ull;
#pragma unroll 4
            for (int w = 0; w < Q_WARPS; ++w) {
                sw += bw[w][threadIdx.x];
                sq += bq[w][threadIdx.x];
            }
            if (sw) {
                atomicAdd(&h->lacc[buf][threadIdx.x][0], sw);
                atomicAdd(&h->lacc[buf][threadIdx.x][1], sq);
            }
        }
        if (threadIdx.x == 0 && s_changed) atomicOr(&h->changed[buf], 1u);
        if (!grid_barrier(h, gridDim.x, epoch)) return;
        if (threadIdx.x == 0) s_stop = (it > 0) && (__ldcg(&h->changed[buf]) == 0u);
        __syncthreads();
        if (s_stop) break;
        if (threadIdx.x < LEVELS) {
            const unsigned long long Wl = __ldcg(&h->lacc[buf][threadIdx.x][0]);
            const long long Ql = (long long)__ldcg(&h->lacc[buf][threadIdx.x][1]);
            if (Wl > 0)
                L[threadIdx.x] =
                    __double2float_rn(__ddiv_rn(__dmul_rn(__ll2double_rn(Ql), down), __ull2double_rn(Wl)));
        }
        __syncthreads();
        if (threadIdx.x == 0) s_sorted = levels_sorted(L);
        ++updates;
    }

    // Codes of the final levels.
    __syncthreads();
    const bool sorted = s_sorted;
    for (int64_t m = tid0; m < N; m += stride)
        a.codes[m] = (uint8_t)(sorted ? nearest_level_sorted(a.C[m], L) : nearest_level(a.C[m], L));
    if (blockIdx.x == 0) {
        if (threadIdx.x < LEVELS) a.levels[threadIdx.x] = L[threadIdx.x];
        if (threadIdx.x == 0 && a.iters_run) *a.iters_run = updates;
    }
}

cudaError_t launch_level_fit(const float *C, int64_t N, const int32_t *counts, int32_t max_iters, float *levels,
                             uint8_t *codes, int32_t *iters_run, Header *hdr, int num_sms, cudaStream_t s) {
    // Clear everything but the sticky status word; minima start at the top of the order.
    cudaError_t e = cudaMemsetAsync(&hdr->maxabs_bits, 0, sizeof(Header) - offsetof(Header, maxabs_bits), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(&hdr->lo_w, 0xff, 2 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, level_fit_kernel, Q_THREADS, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    int64_t blocks = (N + Q_THREADS - 1) / Q_THREADS;
    if (blocks > (int64_t)num_sms) blocks = num_sms;  // one CTA per SM is plenty, and co-resident
    if (blocks < 1) blocks = 1;
    LevelArgs args{C, N, counts, max_iters, levels, codes, iters_run, hdr};
    void *params[] = {&args};
    e = cudaLaunchCooperativeKernel((const void *)level_fit_kernel, dim3((unsigned)blocks), dim3(Q_THREADS), params,
                                    0, s);
    if (e != cudaSuccess) return e;
    count_launch();
    return cudaGetLastError();
}

}  // namespace kq
