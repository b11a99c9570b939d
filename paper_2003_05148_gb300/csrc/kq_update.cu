// kq_update.cu -- update step of KQ's k-means (Sec. 3.1, Eq. 1): c_k = mean of S_k.
//
// Deterministic without floating-point atomics: every coordinate of every kernel
// is converted to an int64 fixed-point number q = rint(v * 2^S) and added with
// integer atomics (red.global.add.u64), which are associative, so the sums do not
// depend on the order the hardware applies them in. S is chosen from max |W| and
// n so that no sum can overflow: with n*max|W| = f * 2^e (f in [0.5, 1)),
// S = 62 - e gives sum |q| <= 2^62 + n/2 < 2^63.
//
// The accumulator of codeword k is one 128-byte line: 9 coordinate sums and the
// member count. A warp takes 32 kernels (1152 contiguous bytes) per step with
// coalesced loads; every lane converts and adds 9 coordinates and one count.
#include "kq_internal.cuh"

namespace kq {

constexpr int U_THREADS = 256;

__device__ __forceinline__ int update_scale(uint32_t maxabs_bits, int64_t n) {
    const float M = __uint_as_float(maxabs_bits);
    if (!(M > 0.f) || isinf(M)) return 0;
    int e;
    frexp((double)n * (double)M, &e);
    return 62 - e;
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
    for (int64_t v = n4 * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < count; v += stride) {
        const float t = W[v];
        ok &= isfinite(t);
        m = fmaxf(m, fabsf(t));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if (!__all_sync(0xffffffffu, ok) && (threadIdx.x & 31) == 0) set_flag(status, KQ_FLAG_NONFINITE);
    if ((threadIdx.x & 31) == 0) atomicMax(maxabs_bits, __float_as_uint(m));  // m >= +0: bits order as values
}

__global__ void __launch_bounds__(U_THREADS)
accumulate_kernel(const float *__restrict__ W, int64_t n, const int32_t *__restrict__ idx, int32_t K,
                  const uint32_t *__restrict__ maxabs_bits, unsigned long long *__restrict__ acc,
                  uint32_t *status) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = update_scale(*maxabs_bits, n);
    // A chunk is 32 kernels = 288 consecutive floats. In pass i a lane handles float
    // lane + 32 i of the chunk (coalesced loads straight from global memory): kernel
    // rr[i] of the chunk, coordinate jj[i]; the kernel's codeword comes from lane rr[i].
    int rr[D], jj[D];
#pragma unroll
    for (int i = 0; i < D; ++i) {
        rr[i] = (lane + 32 * i) / D;
        jj[i] = (lane + 32 * i) - D * rr[i];
    }
    bool bad = false;
    const int64_t nchunks = n / 32;
    // Chunks are visited last-to-first: a max|W| pass that just streamed W front to
    // back leaves the tail of W in L2.
    for (int64_t it = (int64_t)blockIdx.x * (U_THREADS / 32) + warp; it < nchunks;
         it += (int64_t)gridDim.x * (U_THREADS / 32)) {
        const int64_t r0 = (nchunks - 1 - it) * 32;
        const float *src = W + r0 * D;
        float v[D];
#pragma unroll
        for (int i = 0; i < D; ++i) v[i] = __ldg(src + lane + 32 * i);
        const int32_t myk = __ldcs(idx + r0 + lane);
        const bool okk = (uint32_t)myk < (uint32_t)K;
        bad |= !okk;
#pragma unroll
        for (int i = 0; i < D; ++i) {
            const int32_t k = __shfl_sync(0xffffffffu, myk, rr[i]);
            if ((uint32_t)k < (uint32_t)K)
                atomicAdd(acc + (int64_t)k * ACC_WORDS + jj[i], (unsigned long long)fixed_rn(v[i], S));
        }
        if (okk) atomicAdd(acc + (int64_t)myk * ACC_WORDS + D, 1ull);
    }
    // ragged end (< 32 kernels): one thread per kernel in CTA 0
    if (blockIdx.x == 0) {
        const int64_t i = nchunks * 32 + threadIdx.x;
        if (threadIdx.x < 32 && i < n) {
            const int32_t k = idx[i];
            if ((uint32_t)k < (uint32_t)K) {
#pragma unroll
                for (int j = 0; j < D; ++j)
                    atomicAdd(acc + (int64_t)k * ACC_WORDS + j, (unsigned long long)fixed_rn(W[i * D + j], S));
                atomicAdd(acc + (int64_t)k * ACC_WORDS + D, 1ull);
            } else {
                bad = true;
            }
        }
    }
    if (bad) set_flag(status, KQ_FLAG_INDEX_RANGE);
}

// c_k = (sum * 2^-S) / z_k in fp32 (keep C_prev when z_k = 0); clears the
// accumulator row for the next call. fp32
// arithmetic (GB300's fp64 rate is low): sum -> fp32, exact power-of-two scaling,
// one IEEE division; within ~1.5 ulp of the exact mean.
__global__ void __launch_bounds__(256)
finalize_kernel(unsigned long long *__restrict__ acc, int32_t K, int64_t n, const uint32_t *__restrict__ maxabs_bits,
                const float *C_prev, float *C_next, int32_t *__restrict__ counts) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    const int S = update_scale(*maxabs_bits, n);
    unsigned long long *a = acc + (int64_t)k * ACC_WORDS;
    const long long z = (long long)a[D];
    const float zf = (float)z;  // exact below 2^24, within half an ulp above
    float c[D];
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const float sum = scalbnf(__ll2float_rn((long long)a[j]), -S);
        c[j] = z > 0 ? __fdiv_rn(sum, zf) : C_prev[(int64_t)k * D + j];
    }
#pragma unroll
    for (int j = 0; j < D; ++j) C_next[(int64_t)k * D + j] = c[j];
    counts[k] = (int32_t)z;
    ulonglong2 *a2 = reinterpret_cast<ulonglong2 *>(a);
#pragma unroll
    for (int w = 0; w < ACC_WORDS / 2; ++w) a2[w] = make_ulonglong2(0ull, 0ull);
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
    histogram_kernel<<<(unsigned)blocks, 256, 0, s>>>(idx, n, K, counts, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_maxabs(const float *W, int64_t count, uint32_t *maxabs_bits, uint32_t *status, int num_sms,
                          cudaStream_t s) {
    int64_t blocks = (count / 4 + 255) / 256;
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    maxabs_kernel<<<(unsigned)blocks, 256, 0, s>>>(W, count, maxabs_bits, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_accumulate(const float *W, int64_t n, const int32_t *idx, int32_t K,
                              const uint32_t *maxabs_bits, unsigned long long *acc, uint32_t *status,
                              int num_sms, cudaStream_t s) {
    const int64_t chunks = n / 32 + 1;
    int64_t blocks = (chunks + U_THREADS / 32 - 1) / (U_THREADS / 32);
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    accumulate_kernel<<<(unsigned)blocks, U_THREADS, 0, s>>>(W, n, idx, K, maxabs_bits, acc, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_finalize(unsigned long long *acc, int32_t K, int64_t n, const uint32_t *maxabs_bits,
                            const float *C_prev, float *C_next, int32_t *counts, cudaStream_t s) {
    finalize_kernel<<<(K + 255) / 256, 256, 0, s>>>(acc, K, n, maxabs_bits, C_prev, C_next, counts);
    count_launch();
    return cudaGetLastError();
}

}  // namespace kq
