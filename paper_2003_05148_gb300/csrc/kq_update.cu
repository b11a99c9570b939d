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
// member count. A warp stages 32 kernels (1152 contiguous bytes) in shared memory
// with float4 loads; each half-warp then adds one kernel: lanes 0..8 a coordinate,
// lane 9 the count, so one warp-wide RED touches two lines.
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
    for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < n4; v += stride) {
        const float4 t = __ldcs(W4 + v);
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
    __shared__ __align__(16) float sw[U_THREADS / 32][32 * D];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const double up = ldexp(1.0, update_scale(*maxabs_bits, n));
    float *buf = sw[warp];
    const int64_t nchunks = (n + 31) / 32;
    for (int64_t ch = (int64_t)blockIdx.x * (U_THREADS / 32) + warp; ch < nchunks;
         ch += (int64_t)gridDim.x * (U_THREADS / 32)) {
        const int64_t r0 = ch * 32;
        const int rows = (int)min((int64_t)32, n - r0);
        const float *src = W + r0 * D;
        if (rows == 32) {
            const float4 *s4 = reinterpret_cast<const float4 *>(src);
            float4 *b4 = reinterpret_cast<float4 *>(buf);
            for (int v = lane; v < 32 * D / 4; v += 32) b4[v] = __ldcs(s4 + v);
        } else {
            for (int v = lane; v < rows * D; v += 32) buf[v] = src[v];
        }
        const int32_t myk = lane < rows ? __ldcs(idx + r0 + lane) : 0;
        __syncwarp();
#pragma unroll 4
        for (int rr = 0; rr < 16; ++rr) {
            const int r = 2 * rr + (lane >> 4);
            const int j = lane & 15;
            const int32_t k = __shfl_sync(0xffffffffu, myk, r);
            if (r < rows && j <= D) {
                if ((uint32_t)k < (uint32_t)K) {
                    const unsigned long long add =
                        j < D ? (unsigned long long)__double2ll_rn((double)buf[r * D + j] * up) : 1ull;
                    atomicAdd(acc + (int64_t)k * ACC_WORDS + j, add);
                } else if (j == 0) {
                    set_flag(status, KQ_FLAG_INDEX_RANGE);
                }
            }
        }
        __syncwarp();
    }
}

// c_k = (sum * 2^-S) / z_k rounded to fp32 (keep C_prev when z_k = 0); also writes
// the packed copy used by the next assignment and clears the accumulator row.
__global__ void __launch_bounds__(256)
finalize_kernel(unsigned long long *__restrict__ acc, int32_t K, int64_t n, const uint32_t *__restrict__ maxabs_bits,
                const float *C_prev, float *C_next, int32_t *__restrict__ counts, float *__restrict__ Cd_next) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    const double down = ldexp(1.0, -update_scale(*maxabs_bits, n));
    unsigned long long *a = acc + (int64_t)k * ACC_WORDS;
    const long long z = (long long)a[D];
    float c[D];
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const double sum = __ll2double_rn((long long)a[j]) * down;
        c[j] = z > 0 ? __double2float_rn(__ddiv_rn(sum, (double)z)) : C_prev[(int64_t)k * D + j];
    }
#pragma unroll
    for (int j = 0; j < D; ++j) C_next[(int64_t)k * D + j] = c[j];
    counts[k] = (int32_t)z;
    if (Cd_next) {
        float4 *dst = reinterpret_cast<float4 *>(Cd_next + (int64_t)k * CD_FLOATS);
        dst[0] = make_float4(c[0], c[0], c[1], c[1]);
        dst[1] = make_float4(c[2], c[2], c[3], c[3]);
        dst[2] = make_float4(c[4], c[4], c[5], c[5]);
        dst[3] = make_float4(c[6], c[6], c[7], c[7]);
        dst[4] = make_float4(c[8], c[8], 0.f, 0.f);
    }
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
    const int64_t chunks = (n + 31) / 32;
    int64_t blocks = (chunks + U_THREADS / 32 - 1) / (U_THREADS / 32);
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    accumulate_kernel<<<(unsigned)blocks, U_THREADS, 0, s>>>(W, n, idx, K, maxabs_bits, acc, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_finalize(unsigned long long *acc, int32_t K, int64_t n, const uint32_t *maxabs_bits,
                            const float *C_prev, float *C_next, int32_t *counts, float *Cd_next,
                            cudaStream_t s) {
    finalize_kernel<<<(K + 255) / 256, 256, 0, s>>>(acc, K, n, maxabs_bits, C_prev, C_next, counts, Cd_next);
    count_launch();
    return cudaGetLastError();
}

}  // namespace kq
