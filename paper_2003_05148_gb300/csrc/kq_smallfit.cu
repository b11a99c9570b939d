// kq_smallfit.cu -- the k-means fit of Eq. 1 (Sec. 3.1) for small codebooks in one
// cooperative launch.
//
// For K <= 512 a Lloyd iteration is a few microseconds of GPU work spread over
// 6-11 kernel launches, so the launches, not the kernels, set the time. Here every
// CTA stays resident for the whole fit and the CTAs meet at bounded grid barriers:
//   phase 0      max|W| (the fixed-point scale of the sums, once per fit);
//   iteration t  assign every kernel against C_t (exact fp32 direct-form argmin,
//                lowest index on ties) and add it to the int64 fixed-point sums of
//                its codeword; barrier; C_{t+1} = sums / counts (empty keeps C_t),
//                objective J_t = sum of the distances; barrier;
//   final        assign against C_T, cluster sizes of that assignment, J_T.
// With stop_on_stable an assignment equal to the previous one ends the fit early: it
// is a fixed point (C_{t+1} would be C_t bit for bit), so it is the final assignment,
// C_t the final codebook and J_t every later objective entry.
// The distances are the definition's (t_j = fl(x_j - c_j), acc = fma(t_j, t_j, acc),
// j = 0..8), two codewords at a time with packed fp32x2 arithmetic (each half is the
// scalar sequence); the sums use the integer conversion and scale of the update
// kernels, so centroids, indices and counts are bit-identical to the multi-launch fit.
#include "kq_internal.cuh"

namespace kq {

constexpr int SF_THREADS = 256;
constexpr int SF_ROWS = 4;             // kernels per group (codebook loads shared)
constexpr int SF_SPLIT = 8;            // lanes that share a group's codebook scan
constexpr int32_t SF_MAX_K = 512;      // codebook pairs in shared memory: 9 x 256 x 8 B = 18 KB

struct SmallFitArgs {
    const float *W;
    int64_t n;
    const float *C0;
    int32_t K;
    int32_t iters;
    float *C_out;
    int32_t *idx;
    int32_t *counts;
    double *objective;
    unsigned long long *acc;  // K x ACC_WORDS, zero on entry, zero again on exit
    float *cbuf0, *cbuf1;     // C_t alternates between the two
    double *blocksum;         // one partial objective per CTA
    Header *hdr;
    int stop_on_stable;
};

// One pass of the assignment against the codebook pairs in shared memory; adds the
// kernels to the sums (accumulate) or only to the counts (final pass), and returns
// this thread's share of the objective. A group of SF_ROWS kernels is searched by
// SF_SPLIT consecutive lanes: lane s of the group takes the codeword pairs p with
// p % SF_SPLIT == s (consecutive lanes read consecutive pairs: no bank conflicts), and
// the lanes' (distance, index) minima merge lexicographically, so the lowest index
// wins ties as in one sequential scan. Lane s < SF_ROWS then records kernel s.
__device__ __forceinline__ F2 small_fit_assign(const SmallFitArgs &a, const unsigned long long (*cp)[SF_MAX_K / 2],
                                                   int32_t npairs, int S, bool accumulate, bool &nonfinite,
                                                   bool compare, bool &moved) {
    const int lane = threadIdx.x & 31, slice = lane % SF_SPLIT;
    const unsigned gmask = 0xffu << (lane & ~(SF_SPLIT - 1));  // the group's lanes
    const int64_t gstride = (int64_t)gridDim.x * (SF_THREADS / SF_SPLIT);
    F2 part{0.f, 0.f};
    // groups of SF_ROWS kernels dealt round-robin over the CTAs, so every CTA has work
    for (int64_t g = (int64_t)(threadIdx.x / SF_SPLIT) * gridDim.x + blockIdx.x; g * SF_ROWS < a.n; g += gstride) {
        const int64_t r0 = g * SF_ROWS;
        unsigned long long x2[SF_ROWS][D];
#pragma unroll
        for (int r = 0; r < SF_ROWS; ++r)
#pragma unroll
            for (int j = 0; j < D; ++j) {
                const float v = r0 + r < a.n ? a.W[(r0 + r) * D + j] : 0.f;
                x2[r][j] = pack2(v, v);
            }
        float best[SF_ROWS];
        int32_t bi[SF_ROWS];
#pragma unroll
        for (int r = 0; r < SF_ROWS; ++r) {
            best[r] = __int_as_float(0x7f800000);
            bi[r] = 0;
        }
        for (int32_t p = slice; p < npairs; p += SF_SPLIT) {
            unsigned long long c2[D];
#pragma unroll
            for (int j = 0; j < D; ++j) c2[j] = cp[j][p];
#pragma unroll
            for (int r = 0; r < SF_ROWS; ++r) {
                unsigned long long t = sub2(x2[r][0], c2[0]);
                unsigned long long acc2 = mul2(t, t);  // fma(t, t, 0) = the rounded square
#pragma unroll
                for (int j = 1; j < D; ++j) {
                    t = sub2(x2[r][j], c2[j]);
                    acc2 = fma2(t, t, acc2);
                }
                float d0, d1;
                unpack2(acc2, d0, d1);
                if (d0 < best[r]) {
                    best[r] = d0;
                    bi[r] = 2 * p;
                }
                if (d1 < best[r]) {
                    best[r] = d1;
                    bi[r] = 2 * p + 1;
                }
            }
        }
#pragma unroll
        for (int r = 0; r < SF_ROWS; ++r)
#pragma unroll
            for (int o = SF_SPLIT / 2; o > 0; o >>= 1) {
                const float od = __shfl_xor_sync(gmask, best[r], o);
                const int32_t oi = __shfl_xor_sync(gmask, bi[r], o);
                if (od < best[r] || (od == best[r] && oi < bi[r])) {
                    best[r] = od;
                    bi[r] = oi;
                }
            }
        // lane s < SF_ROWS of the group records kernel r0 + s (static indexing: a select chain)
        float mb = best[0];
        int32_t mi = bi[0];
#pragma unroll
        for (int r = 1; r < SF_ROWS; ++r)
            if (slice == r) {
                mb = best[r];
                mi = bi[r];
            }
        const int64_t row = r0 + slice;
        if (slice < SF_ROWS && row < a.n) {
            if (compare) moved |= a.idx[row] != mi;  // the previous assignment, written by this lane
            a.idx[row] = mi;
            part = f2_add(part, F2{mb, 0.f});
            unsigned long long *acc = a.acc + (int64_t)mi * ACC_WORDS;
            if (accumulate) {
#pragma unroll
                for (int j = 0; j < D; ++j) {
                    const float v = a.W[row * D + j];  // the row again (L1)
                    nonfinite |= !isfinite(v);
                    atomicAdd(acc + j, (unsigned long long)fixed_rn(v, S));
                }
            }
            atomicAdd(acc + D, 1ull);
        }
    }
    return part;
}

__global__ void __launch_bounds__(SF_THREADS) small_fit_kernel(SmallFitArgs a) {
    __shared__ unsigned long long cp[D][SF_MAX_K / 2];  // codewords 2p, 2p + 1 packed per coordinate
    __shared__ F2 wsum[SF_THREADS / 32];
    Header *h = a.hdr;
    unsigned epoch = 0;
    const int64_t gtid = (int64_t)blockIdx.x * SF_THREADS + threadIdx.x;
    const int64_t nthr = (int64_t)gridDim.x * SF_THREADS;
    const int32_t npairs = (a.K + 1) / 2;
    bool nonfinite = false;

    // phase 0: max|W| for the scale; C_0 into the first buffer
    {
        float m = 0.f;
        for (int64_t e = gtid; e < a.n * D; e += nthr) m = fmaxf(m, fabsf(a.W[e]));  // inf kept, NaN skipped
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if ((threadIdx.x & 31) == 0) atomicMax(&h->maxabs_bits, __float_as_uint(m));
        for (int64_t e = gtid; e < (int64_t)a.K * D; e += nthr) a.cbuf0[e] = a.C0[e];
        if (gtid == 0) h->fit_moved = h->fit_moved1 = 0u;  // first set after the barrier below
    }
    if (!grid_barrier(h, gridDim.x, epoch)) return;
    const int S = fit_sum_scale(__uint_as_float(__ldcg(&h->maxabs_bits)), a.n);

    for (int32_t t = 0; t <= a.iters; ++t) {
        const bool last = t == a.iters;
        const float *Ct = (t & 1) ? a.cbuf1 : a.cbuf0;
        // codebook C_t into shared memory, two codewords per packed word (an odd K
        // is padded with a +inf codeword: distance +inf, never chosen)
        for (int e = threadIdx.x; e < D * npairs; e += SF_THREADS) {
            const int j = e / npairs, p = e - j * npairs;
            const int32_t k0 = 2 * p, k1 = 2 * p + 1;
            const float c0 = __ldcg(Ct + (int64_t)k0 * D + j);
            const float c1 = k1 < a.K ? __ldcg(Ct + (int64_t)k1 * D + j) : __int_as_float(0x7f800000);
            nonfinite |= !isfinite(c0) || (k1 < a.K && !isfinite(c1));
            cp[j][p] = pack2(c0, c1);
        }
        __syncthreads();
        bool moved = false;
        F2 part = small_fit_assign(a, cp, npairs, S, !last, nonfinite, a.stop_on_stable && t > 0, moved);
        uint32_t *moved_word = (t & 1) ? &h->fit_moved1 : &h->fit_moved;
        if (__any_sync(0xffffffffu, moved) && (threadIdx.x & 31) == 0) atomicOr(moved_word, 1u);
        // per-CTA partial of the objective, fixed order
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
            part = f2_add(part, F2{__shfl_xor_sync(0xffffffffu, part.hi, o), __shfl_xor_sync(0xffffffffu, part.lo, o)});
        if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = part;
        __syncthreads();
        if (threadIdx.x == 0) {  // the CTA's pair, in the 8 bytes of its block-sum slot
            F2 s{0.f, 0.f};
            for (int w = 0; w < SF_THREADS / 32; ++w) s = f2_add(s, wsum[w]);
            reinterpret_cast<F2 *>(a.blocksum)[blockIdx.x] = s;
        }
        if (!grid_barrier(h, gridDim.x, epoch)) return;
        // a fixed point: this assignment is the final one (the same word in every CTA;
        // the other parity's word was last read before the previous barrier)
        const bool stable = a.stop_on_stable && t > 0 && !last && __ldcg(moved_word) == 0u;
        if (gtid == 0) *((t & 1) ? &h->fit_moved : &h->fit_moved1) = 0u;
        const bool fin = last || stable;
        // C_{t+1} = mean of each set (the update's arithmetic), or the cluster sizes of
        // the final assignment; the accumulators are cleared for the next pass
        float *Cn = (t & 1) ? a.cbuf0 : a.cbuf1;
        for (int64_t k = gtid; k < a.K; k += nthr) {
            unsigned long long *row = a.acc + k * ACC_WORDS;
            const long long z = (long long)__ldcg(row + D);
            if (!fin) {
                const float zf = (float)z;
#pragma unroll
                for (int j = 0; j < D; ++j) {
                    const float sum = scalbnf(__ll2float_rn((long long)__ldcg(row + j)), -S);
                    Cn[k * D + j] = z > 0 ? __fdiv_rn(sum, zf) : __ldcg(Ct + k * D + j);
                }
            } else {
#pragma unroll
                for (int j = 0; j < D; ++j) a.C_out[k * D + j] = __ldcg(Ct + k * D + j);
            }
            a.counts[k] = (int32_t)z;
#pragma unroll
            for (int j = 0; j <= D; ++j) row[j] = 0ull;
        }
        if (a.objective && gtid < 32) {  // warp 0 of CTA 0: lane l takes CTAs l, l + 32, ..., then a butterfly
            const F2 *bs = reinterpret_cast<const F2 *>(a.blocksum);
            F2 s{0.f, 0.f};
            for (unsigned b = (unsigned)gtid; b < gridDim.x; b += 32) {
                const float2 v = __ldcg(reinterpret_cast<const float2 *>(bs + b));
                s = f2_add(s, F2{v.x, v.y});
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1)
                s = f2_add(s, F2{__shfl_xor_sync(0xffffffffu, s.hi, o), __shfl_xor_sync(0xffffffffu, s.lo, o)});
            if (gtid == 0)
                for (int32_t u = t; u <= (stable ? a.iters : t); ++u) a.objective[u] = f2_to_double(s);
        }
        if (gtid == 0 && fin) h->fit_iters = t;
        if (fin) break;
        if (!grid_barrier(h, gridDim.x, epoch)) return;
    }
    if (__any_sync(0xffffffffu, nonfinite) && (threadIdx.x & 31) == 0) set_flag(&h->status, KQ_FLAG_NONFINITE);
}

// Up to 2^22 kernel x codeword pairs per iteration: beyond that the multi-launch
// kernels (tensor cores, split-K CUDA-core assign) are faster (VGG-16 conv3_2, 16.8M
// pairs: 1.57 vs 1.10 ms per 20-iteration fit; conv 64x64, 65,536 pairs: 0.27 vs 0.50 ms).
bool small_fit_eligible(int64_t n, int32_t K) { return K <= SF_MAX_K && (int64_t)n * K <= (1LL << 22); }

cudaError_t launch_small_fit(const float *W, int64_t n, const float *C0, int32_t K, int32_t iters, float *C_out,
                             int32_t *idx, int32_t *counts, double *objective, unsigned long long *acc, float *cbuf0,
                             float *cbuf1, double *blocksum, int max_blocksum, Header *hdr, int num_sms,
                             cudaStream_t s, bool stop_on_stable) {
    cudaError_t e = cudaMemsetAsync(acc, 0, (size_t)K * ACC_WORDS * sizeof(unsigned long long), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(&hdr->maxabs_bits, 0, 3 * sizeof(uint32_t), s);  // max|W|, barrier counter, abort word
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, small_fit_kernel, SF_THREADS, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const int64_t groups = (n + SF_ROWS - 1) / SF_ROWS;
    int64_t blocks = (groups + 31) / 32;  // about 32 groups per CTA
    if (blocks > (int64_t)per_sm * num_sms) blocks = (int64_t)per_sm * num_sms;  // co-resident by construction
    if (blocks > max_blocksum) blocks = max_blocksum;
    if (blocks < 1) blocks = 1;
    SmallFitArgs a{W, n, C0, K, iters, C_out, idx, counts, objective, acc, cbuf0, cbuf1, blocksum, hdr,
                   stop_on_stable ? 1 : 0};
    void *params[] = {&a};
    launch_begin(s);
    e = cudaLaunchCooperativeKernel((const void *)small_fit_kernel, dim3((unsigned)blocks), dim3(SF_THREADS), params, 0,
                                    s);
    if (e != cudaSuccess) return e;
    launch_end(s, "small_fit_kernel");
    return cudaGetLastError();
}

}  // namespace kq
