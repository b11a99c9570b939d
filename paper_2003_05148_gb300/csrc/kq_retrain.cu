// kq_retrain.cu -- retraining with averaged gradients on sm_103a.
//
// Sec. 3.1, Eq. 2: during retraining every kernel m_i mapped to codebook entry
// c_k contributes its loss gradient g_i = dL/dm_i, and the entry moves against
// the element-wise average of those gradients:
//     c_k <- c_k - lr * (1 / z_k) * sum_{i in S_k} g_i.
// Sec. 3.2 retrains the 6-bit codebook the same way: a weight of the network is
// levels[codes[idx_i][j]], so level l moves against the average gradient of all
// the weights whose value it is.
//
// Both averages are exact, order-independent int64 fixed-point sums (the
// conversion of kq_update.cu, scale chosen from max|G| so that no sum can
// overflow), so the results are bitwise reproducible. The codebook step reuses
// the update's accumulators (kq_update.cu) and only adds its own finalise; the
// level step is a 64-key segment sum: every lane keeps private per-level sums in
// shared memory (its own column: no atomics, no bank conflicts), and each CTA
// adds its 64 totals to the workspace header with integer atomics.
#include "kq_internal.cuh"

namespace kq {

constexpr int LG_THREADS = 128;  // 4 warps: 96 KB of private bins, two CTAs per SM
constexpr int LG_WARPS = LG_THREADS / 32;
constexpr int LG_UNROLL = 4;     // 32-kernel chunks whose loads a warp has in flight together
constexpr uint32_t NO_KERNEL = 0x100u;  // "code" of a padding lane or an out-of-range index

// c_k <- c_k - lr * mean, mean = (sum * 2^-S) / z_k in fp32 (the update's mean:
// sum -> fp32, exact power-of-two scaling, one IEEE division), step = fl(lr * mean),
// result = fl(c_k - step); z_k = 0 keeps c_k. Clears the accumulator row.
__global__ void __launch_bounds__(256)
grad_finalize_kernel(unsigned long long *__restrict__ acc, int32_t K, const Header *hdr, float lr, const float *C,
                     float *C_next, int32_t *__restrict__ counts) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    const int S = __ldcg(&hdr->upd_scale);
    unsigned long long *a = acc + (int64_t)k * ACC_WORDS;
    const long long z = (long long)a[D];
    const float zf = (float)z;
    float c[D];
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const float cj = C[(int64_t)k * D + j];
        const float mean = __fdiv_rn(scalbnf(__ll2float_rn((long long)a[j]), -S), zf);
        c[j] = z > 0 ? __fsub_rn(cj, __fmul_rn(lr, mean)) : cj;
    }
#pragma unroll
    for (int j = 0; j < D; ++j) C_next[(int64_t)k * D + j] = c[j];
    counts[k] = (int32_t)z;
    ulonglong2 *a2 = reinterpret_cast<ulonglong2 *>(a);
#pragma unroll
    for (int w = 0; w < ACC_WORDS / 2; ++w) a2[w] = make_ulonglong2(0ull, 0ull);
}

struct LevelBins {
    unsigned long long sum[LG_WARPS][LEVELS][32];  // [warp][level][lane]
    uint32_t cnt[LG_WARPS][LEVELS][32];
};

// Per-level sums of G over all weights (i, j) with code l = codes[idx_i * 9 + j].
// A warp takes LG_UNROLL chunks of 32 kernels at a time; in pass p a lane loads
// float lane + 32 p of a chunk (coalesced): kernel rr[p], coordinate jj[p], whose
// codeword comes from lane rr[p] by shuffle.
__global__ void __launch_bounds__(LG_THREADS)
level_grad_kernel(const float *__restrict__ G, int64_t n, const int32_t *__restrict__ idx, int32_t K,
                  const uint8_t *__restrict__ codes, Header *hdr) {
    extern __shared__ __align__(16) unsigned char lg_smem[];
    LevelBins &B = *reinterpret_cast<LevelBins *>(lg_smem);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int l = 0; l < LEVELS; ++l) {
        B.sum[warp][l][lane] = 0ull;
        B.cnt[warp][l][lane] = 0u;
    }
    // scale: N = 9n values bounded by max|G|
    const float gmax = __uint_as_float(__ldcg(&hdr->maxabs_bits));
    int S = 0;
    if (gmax > 0.f && gmax <= 3.402823466e38f) {
        int e;
        frexp((double)(n * D) * (double)gmax, &e);
        S = 62 - e;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) hdr->upd_scale = S;
    int rr[D], jj[D];
#pragma unroll
    for (int p = 0; p < D; ++p) {
        rr[p] = (lane + 32 * p) / D;
        jj[p] = (lane + 32 * p) - D * rr[p];
    }
    bool bad_idx = false, bad_code = false;
    const int64_t nchunks = (n + 31) / 32;
    const int64_t step = (int64_t)gridDim.x * LG_WARPS;
    for (int64_t c0 = (int64_t)blockIdx.x * LG_WARPS + warp; c0 < nchunks; c0 += step * LG_UNROLL) {
        float v[LG_UNROLL][D];
        int32_t myk[LG_UNROLL];
#pragma unroll
        for (int u = 0; u < LG_UNROLL; ++u) {
            const int64_t c = c0 + u * step;
            const int64_t r0 = c * 32;
            const bool full = c < nchunks && r0 + 32 <= n;
#pragma unroll
            for (int p = 0; p < D; ++p) {
                const int64_t e = r0 * D + lane + 32 * p;
                v[u][p] = full || (c < nchunks && e < n * D) ? __ldcs(G + e) : 0.f;
            }
            myk[u] = (c < nchunks && r0 + lane < n) ? __ldcs(idx + r0 + lane) : -1;
            bad_idx |= (c < nchunks && r0 + lane < n) && (uint32_t)myk[u] >= (uint32_t)K;
        }
        uint32_t code[LG_UNROLL][D];
#pragma unroll
        for (int u = 0; u < LG_UNROLL; ++u)
#pragma unroll
            for (int p = 0; p < D; ++p) {
                const int32_t k = __shfl_sync(0xffffffffu, myk[u], rr[p]);
                code[u][p] = (uint32_t)k < (uint32_t)K ? (uint32_t)__ldg(codes + (int64_t)k * D + jj[p]) : NO_KERNEL;
            }
#pragma unroll
        for (int u = 0; u < LG_UNROLL; ++u)
#pragma unroll
            for (int p = 0; p < D; ++p) {
                const uint32_t l = code[u][p];
                if (l < (uint32_t)LEVELS) {
                    B.sum[warp][l][lane] += (unsigned long long)fixed_rn(v[u][p], S);
                    B.cnt[warp][l][lane] += 1u;
                } else if (l != NO_KERNEL) {
                    bad_code = true;
                }
            }
    }
    if (bad_idx) set_flag(&hdr->status, KQ_FLAG_INDEX_RANGE);
    if (bad_code) set_flag(&hdr->status, KQ_FLAG_CODE_RANGE);
    __syncthreads();
    // CTA totals: thread t sums level t & 63 over half of the (warp, lane) columns
    __shared__ unsigned long long part_s[LEVELS];
    __shared__ unsigned long long part_c[LEVELS];
    const int l = threadIdx.x & (LEVELS - 1), half = threadIdx.x >> 6;
    unsigned long long ss = 0ull, cc = 0ull;
    for (int w = half * (LG_WARPS / 2); w < (half + 1) * (LG_WARPS / 2); ++w)
#pragma unroll 8
        for (int ln = 0; ln < 32; ++ln) {
            ss += B.sum[w][l][ln];
            cc += B.cnt[w][l][ln];
        }
    if (half == 1) {
        part_s[l] = ss;
        part_c[l] = cc;
    }
    __syncthreads();
    if (half == 0) {
        ss += part_s[l];
        cc += part_c[l];
        if (cc) {
            atomicAdd(&hdr->lacc[0][l][0], cc);
            atomicAdd(&hdr->lacc[0][l][1], ss);
        }
    }
}

// levels_next[l] = levels[l] - fl(lr * mean_l) (mean as in grad_finalize_kernel),
// or levels[l] when no weight has code l; counts[l] = that number of weights.
__global__ void level_grad_finalize_kernel(const Header *hdr, float lr, const float *levels, float *levels_next,
                                           int64_t *counts) {
    const int l = threadIdx.x;
    if (l >= LEVELS) return;
    const int S = __ldcg(&hdr->upd_scale);
    const unsigned long long z = __ldcg(&hdr->lacc[0][l][0]);
    const long long q = (long long)__ldcg(&hdr->lacc[0][l][1]);
    const float L = levels[l];
    const float mean = __fdiv_rn(scalbnf(__ll2float_rn(q), -S), __ull2float_rn(z));
    levels_next[l] = z > 0 ? __fsub_rn(L, __fmul_rn(lr, mean)) : L;
    if (counts) counts[l] = (int64_t)z;
}

cudaError_t launch_grad_finalize(unsigned long long *acc, int32_t K, const Header *hdr, float lr, const float *C,
                                 float *C_next, int32_t *counts, cudaStream_t s) {
    launch_begin(s);
    grad_finalize_kernel<<<(K + 255) / 256, 256, 0, s>>>(acc, K, hdr, lr, C, C_next, counts);
    launch_end(s, "grad_finalize_kernel");
    return cudaGetLastError();
}

cudaError_t launch_level_grad(const float *G, int64_t n, const int32_t *idx, int32_t K, const uint8_t *codes,
                              float lr, const float *levels, float *levels_next, int64_t *counts, Header *hdr,
                              int num_sms, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(&hdr->lacc[0][0][0], 0, sizeof(hdr->lacc[0]), s);
    if (e != cudaSuccess) return e;
    const int smem = (int)sizeof(LevelBins);
    e = cudaFuncSetAttribute(level_grad_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int64_t chunks = (n + 31) / 32;
    int64_t blocks = (chunks + LG_WARPS * LG_UNROLL - 1) / (LG_WARPS * LG_UNROLL);
    if (blocks > 2LL * num_sms) blocks = 2LL * num_sms;  // two CTAs per SM fit in shared memory
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    level_grad_kernel<<<(unsigned)blocks, LG_THREADS, smem, s>>>(G, n, idx, K, codes, hdr);
    launch_end(s, "level_grad_kernel");
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    launch_begin(s);
    level_grad_finalize_kernel<<<1, LEVELS, 0, s>>>(hdr, lr, levels, levels_next, counts);
    launch_end(s, "level_grad_finalize_kernel");
    return cudaGetLastError();
}

}  // namespace kq
