// kq_reconstruct.cu -- test-time recovery (Sec. 3.2, last paragraph) and the
// codeword initialisation gather, on sm_103a.
//
// Recovery runs in the paper's order: first the kernel codebook is decoded once
// per codeword (C_hat[k][j] = levels[codes[k][j]], or C itself without codes) into
// 48-byte rows that are 16-byte aligned, then the weight tensor is gathered,
// W'[i] = C_hat[idx[i]]. The gather is HBM-bound (4 B of index read and 36 B of
// weights written per kernel); the decoded codebook (<= a few MB) stays in L2.
// A warp handles 32 consecutive kernels: each lane fetches its codeword row with
// three 16-byte loads and drops it into a per-warp shared tile, and the warp then
// writes the 1152 contiguous output bytes with coalesced streaming float4 stores.
#include "kq_internal.cuh"

namespace kq {

constexpr int R_THREADS = 256;

__global__ void __launch_bounds__(256)
decode_codebook_kernel(const float *__restrict__ C, int32_t K, const uint8_t *__restrict__ codes,
                       const float *__restrict__ levels, float *__restrict__ Cp, uint32_t *status) {
    __shared__ float sl[LEVELS];
    if (codes && threadIdx.x < LEVELS) sl[threadIdx.x] = levels[threadIdx.x];
    __syncthreads();
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    float c[CP_FLOATS];
    bool bad = false;
#pragma unroll
    for (int j = 0; j < D; ++j) {
        if (codes) {
            const uint8_t q = codes[(int64_t)k * D + j];
            bad |= q >= LEVELS;
            c[j] = q < LEVELS ? sl[q] : 0.f;
        } else {
            c[j] = C[(int64_t)k * D + j];
        }
    }
#pragma unroll
    for (int j = D; j < CP_FLOATS; ++j) c[j] = 0.f;
    if (bad) set_flag(status, KQ_FLAG_CODE_RANGE);
    float4 *dst = reinterpret_cast<float4 *>(Cp + (int64_t)k * CP_FLOATS);
    dst[0] = make_float4(c[0], c[1], c[2], c[3]);
    dst[1] = make_float4(c[4], c[5], c[6], c[7]);
    dst[2] = make_float4(c[8], c[9], c[10], c[11]);
}

__global__ void __launch_bounds__(R_THREADS)
gather_rows_kernel(const int32_t *__restrict__ idx, int64_t n, const float *__restrict__ Cp, int32_t K,
                   float *__restrict__ W_out, uint32_t *status) {
    __shared__ __align__(16) float tile[R_THREADS / 32][32 * D];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *t = tile[warp];
    const int64_t nchunks = (n + 31) / 32;
    for (int64_t ch = (int64_t)blockIdx.x * (R_THREADS / 32) + warp; ch < nchunks;
         ch += (int64_t)gridDim.x * (R_THREADS / 32)) {
        const int64_t r0 = ch * 32;
        const int rows = (int)min((int64_t)32, n - r0);
        if (lane < rows) {
            const int32_t k = __ldcs(idx + r0 + lane);
            float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a, c = a;
            if ((uint32_t)k < (uint32_t)K) {
                const float4 *src = reinterpret_cast<const float4 *>(Cp + (int64_t)k * CP_FLOATS);
                a = __ldg(src);
                b = __ldg(src + 1);
                c = __ldg(src + 2);
            } else {
                set_flag(status, KQ_FLAG_INDEX_RANGE);
            }
            float *row = t + lane * D;
            row[0] = a.x; row[1] = a.y; row[2] = a.z; row[3] = a.w;
            row[4] = b.x; row[5] = b.y; row[6] = b.z; row[7] = b.w;
            row[8] = c.x;
        }
        __syncwarp();
        float *dst = W_out + r0 * D;
        if (rows == 32) {
            const float4 *t4 = reinterpret_cast<const float4 *>(t);
            float4 *d4 = reinterpret_cast<float4 *>(dst);
            for (int v = lane; v < 32 * D / 4; v += 32) __stcs(d4 + v, t4[v]);
        } else {
            for (int v = lane; v < rows * D; v += 32) dst[v] = t[v];
        }
        __syncwarp();
    }
}

__global__ void __launch_bounds__(256)
init_codebook_kernel(const float *__restrict__ W, int64_t n, const int64_t *__restrict__ sel, int32_t K,
                     float *__restrict__ C0, uint32_t *status) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)K * D) return;
    const int64_t j = e / D, c = e - j * D;
    const int64_t r = sel[j];
    if (r >= 0 && r < n) {
        C0[e] = W[r * D + c];
    } else {
        C0[e] = 0.f;
        if (c == 0) set_flag(status, KQ_FLAG_INDEX_RANGE);
    }
}

cudaError_t launch_decode_codebook(const float *C, int32_t K, const uint8_t *codes, const float *levels,
                                   float *Cp, uint32_t *status, cudaStream_t s) {
    decode_codebook_kernel<<<(K + 255) / 256, 256, 0, s>>>(C, K, codes, levels, Cp, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const int32_t *idx, int64_t n, const float *Cp, int32_t K, float *W_out,
                               uint32_t *status, int num_sms, cudaStream_t s) {
    const int64_t chunks = (n + 31) / 32;
    int64_t blocks = (chunks + R_THREADS / 32 - 1) / (R_THREADS / 32);
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    gather_rows_kernel<<<(unsigned)blocks, R_THREADS, 0, s>>>(idx, n, Cp, K, W_out, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_init_codebook(const float *W, int64_t n, const int64_t *sel, int32_t K, float *C0,
                                 uint32_t *status, cudaStream_t s) {
    const int64_t total = (int64_t)K * D;
    init_codebook_kernel<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(W, n, sel, K, C0, status);
    count_launch();
    return cudaGetLastError();
}

}  // namespace kq
