// kq_assign.cu -- assignment step of KQ's k-means (Sec. 3.1, Eq. 1) on sm_103a.
//
// Design (FP32-pipe bound: 9 FSUB + 9 FFMA lane-ops per kernel x codeword pair):
//  * A CTA owns ROW_BLOCK = 1024 kernels: 256 threads x 4 rows. Each thread keeps
//    its 4 rows in registers as two fp32x2 row pairs, so one packed instruction
//    evaluates the same codeword against two kernels (sub.rn.f32x2 / fma.rn.f32x2
//    halve the issue slots; every lane is still an IEEE fp32 op, so the distance
//    is bit-identical to the scalar fp32 direct form).
//  * Codewords are pre-packed once per call (pack_codebook) into 80-byte rows of
//    duplicated pairs (c_j, c_j), j = 0..9 (c_9 = 0), and staged tile by tile in
//    shared memory; every warp reads the same codeword, so the LDS.128 reads are
//    broadcasts.
//  * Argmin: strict '<' in ascending k per thread, so ties go to the lowest k.
//  * Small n: the codebook is split across gridDim.y CTAs (split-K); the per-split
//    winners are merged lexicographically on (distance bits, k), which is exact.
//  * The Eq. 1 objective is reduced per CTA in a fixed order (bitwise
//    reproducible) and summed over CTAs by sum_blocks in block order.
#include "kq_internal.cuh"

namespace kq {

constexpr int A_THREADS = 256;
constexpr int A_ROWS = 4;   // rows per thread (two fp32x2 pairs)
constexpr int A_TILE = 256; // codewords per shared-memory tile (20 KiB)
static_assert(A_THREADS * A_ROWS == ROW_BLOCK, "row block mismatch");

__global__ void pack_codebook_kernel(const float *__restrict__ C, int32_t K, float *__restrict__ Cd,
                                     uint32_t *status) {
    int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    float c[D];
    bool ok = true;
#pragma unroll
    for (int j = 0; j < D; ++j) {
        c[j] = C[(int64_t)k * D + j];
        ok &= isfinite(c[j]);
    }
    if (!ok) set_flag(status, KQ_FLAG_NONFINITE);
    float4 *dst = reinterpret_cast<float4 *>(Cd + (int64_t)k * CD_FLOATS);
    dst[0] = make_float4(c[0], c[0], c[1], c[1]);
    dst[1] = make_float4(c[2], c[2], c[3], c[3]);
    dst[2] = make_float4(c[4], c[4], c[5], c[5]);
    dst[3] = make_float4(c[6], c[6], c[7], c[7]);
    dst[4] = make_float4(c[8], c[8], 0.f, 0.f);
}

// Deterministic fp64 sum over a CTA: fixed xor-shuffle tree, then warps in order.
template <int THREADS>
__device__ __forceinline__ double block_sum_fixed(double v) {
    __shared__ double wsum[THREADS / 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = v;
    __syncthreads();
    double s = 0.0;
    if (threadIdx.x == 0)
        for (int w = 0; w < THREADS / 32; ++w) s += wsum[w];
    return s;
}

__device__ __forceinline__ unsigned long long pack_key(float d, int k) {
    return ((unsigned long long)__float_as_uint(d) << 32) | (unsigned int)k;
}

__global__ void __launch_bounds__(A_THREADS, 2)
assign_kernel(const float *__restrict__ W, int64_t n, const float *__restrict__ Cd, int32_t K, int32_t kps,
              int32_t *__restrict__ idx, float *__restrict__ dist, double *__restrict__ blocksum,
              unsigned long long *__restrict__ part, int64_t part_stride, uint32_t *status) {
    constexpr int P = A_ROWS / 2;
    __shared__ __align__(16) float4 sm[A_TILE * (CD_FLOATS / 4)];

    const int64_t row0 = ((int64_t)blockIdx.x * A_THREADS + threadIdx.x) * A_ROWS;
    float w[A_ROWS * D];
    if (row0 + A_ROWS <= n) {
        const float4 *src = reinterpret_cast<const float4 *>(W + row0 * D);
#pragma unroll
        for (int v = 0; v < A_ROWS * D / 4; ++v) {
            float4 t = __ldg(src + v);
            w[4 * v + 0] = t.x;
            w[4 * v + 1] = t.y;
            w[4 * v + 2] = t.z;
            w[4 * v + 3] = t.w;
        }
    } else {
#pragma unroll
        for (int r = 0; r < A_ROWS; ++r)
#pragma unroll
            for (int j = 0; j < D; ++j) w[r * D + j] = (row0 + r < n) ? W[(row0 + r) * D + j] : 0.f;
    }
    if (blockIdx.y == 0) {
        bool ok = true;
#pragma unroll
        for (int e = 0; e < A_ROWS * D; ++e) ok &= isfinite(w[e]);
        if (!ok) set_flag(status, KQ_FLAG_NONFINITE);
    }

    unsigned long long X[P][D];
#pragma unroll
    for (int p = 0; p < P; ++p)
#pragma unroll
        for (int j = 0; j < D; ++j) X[p][j] = pack2(w[(2 * p) * D + j], w[(2 * p + 1) * D + j]);

    const int32_t kb = blockIdx.y * kps;
    const int32_t ke = min(K, kb + kps);
    float best[A_ROWS];
    int32_t bi[A_ROWS];
#pragma unroll
    for (int r = 0; r < A_ROWS; ++r) {
        best[r] = __int_as_float(0x7f800000);  // +inf
        bi[r] = kb;
    }

    for (int32_t kt = kb; kt < ke; kt += A_TILE) {
        const int cnt = min(A_TILE, ke - kt);
        __syncthreads();
        const float4 *gsrc = reinterpret_cast<const float4 *>(Cd + (int64_t)kt * CD_FLOATS);
        for (int v = threadIdx.x; v < cnt * (CD_FLOATS / 4); v += A_THREADS) sm[v] = __ldg(gsrc + v);
        __syncthreads();
#pragma unroll 2
        for (int c = 0; c < cnt; ++c) {
            const ulonglong2 *cw = reinterpret_cast<const ulonglong2 *>(&sm[c * (CD_FLOATS / 4)]);
            const ulonglong2 c01 = cw[0], c23 = cw[1], c45 = cw[2], c67 = cw[3], c8p = cw[4];
            const unsigned long long Cj[D] = {c01.x, c01.y, c23.x, c23.y, c45.x, c45.y, c67.x, c67.y, c8p.x};
            const int32_t k = kt + c;
#pragma unroll
            for (int p = 0; p < P; ++p) {
                unsigned long long t = sub2(X[p][0], Cj[0]);
                unsigned long long acc = mul2(t, t);  // == fma(t, t, +0) bit for bit
#pragma unroll
                for (int j = 1; j < D; ++j) {
                    t = sub2(X[p][j], Cj[j]);
                    acc = fma2(t, t, acc);
                }
                float d0, d1;
                unpack2(acc, d0, d1);
                if (d0 < best[2 * p]) {
                    best[2 * p] = d0;
                    bi[2 * p] = k;
                }
                if (d1 < best[2 * p + 1]) {
                    best[2 * p + 1] = d1;
                    bi[2 * p + 1] = k;
                }
            }
        }
    }

    if (gridDim.y == 1) {
        double s = 0.0;
#pragma unroll
        for (int r = 0; r < A_ROWS; ++r) {
            if (row0 + r < n) {
                idx[row0 + r] = bi[r];
                if (dist) dist[row0 + r] = best[r];
                s += (double)best[r];
            }
        }
        s = block_sum_fixed<A_THREADS>(s);
        if (threadIdx.x == 0) blocksum[blockIdx.x] = s;
    } else {
#pragma unroll
        for (int r = 0; r < A_ROWS; ++r)
            if (row0 + r < n) part[(int64_t)blockIdx.y * part_stride + row0 + r] = pack_key(best[r], bi[r]);
    }
}

// Merge split-K winners: lexicographic min on (distance bits, k). Distances are
// >= +0 or +inf, so their fp32 bit patterns order like the values.
__global__ void __launch_bounds__(256)
combine_kernel(const unsigned long long *__restrict__ part, int64_t part_stride, int G, int64_t n,
               int32_t *__restrict__ idx, float *__restrict__ dist, double *__restrict__ blocksum) {
    const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
    double s = 0.0;
    if (i < n) {
        unsigned long long key = part[i];
        for (int g = 1; g < G; ++g) {
            unsigned long long o = part[(int64_t)g * part_stride + i];
            key = o < key ? o : key;
        }
        const float d = __uint_as_float((uint32_t)(key >> 32));
        idx[i] = (int32_t)(key & 0xffffffffu);
        if (dist) dist[i] = d;
        s = (double)d;
    }
    s = block_sum_fixed<256>(s);
    if (threadIdx.x == 0) blocksum[blockIdx.x] = s;
}

__global__ void __launch_bounds__(256) sum_blocks_kernel(const double *__restrict__ bs, int nb, double *out) {
    double s = 0.0;
    for (int b = threadIdx.x; b < nb; b += 256) s += bs[b];
    s = block_sum_fixed<256>(s);
    if (threadIdx.x == 0) *out = s;
}

cudaError_t launch_pack_codebook(const float *C, int32_t K, float *Cd, uint32_t *status, cudaStream_t s) {
    pack_codebook_kernel<<<(K + 255) / 256, 256, 0, s>>>(C, K, Cd, status);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_assign(const float *W, int64_t n, const float *Cd, int32_t K, int32_t *idx, float *dist,
                          double *blocksum, int *nblocksum, unsigned long long *part, uint32_t *status,
                          int num_sms, cudaStream_t s) {
    const int64_t row_blocks = (n + ROW_BLOCK - 1) / ROW_BLOCK;
    const int64_t target = 2LL * num_sms;  // two resident CTAs per SM
    int64_t G = 1;
    if (row_blocks < target) {
        G = (target + row_blocks - 1) / row_blocks;
        const int64_t by_tiles = (K + A_TILE - 1) / A_TILE;
        const int64_t by_room = MAX_PART_BLOCKS / row_blocks;
        if (G > by_tiles) G = by_tiles;
        if (G > by_room) G = by_room;
        if (G < 1) G = 1;
    }
    int32_t kps = (int32_t)((K + G - 1) / G);
    G = (K + kps - 1) / kps;
    const int64_t part_stride = row_blocks * ROW_BLOCK;
    dim3 grid((unsigned)row_blocks, (unsigned)G);
    assign_kernel<<<grid, A_THREADS, 0, s>>>(W, n, Cd, K, kps, idx, dist, blocksum, part, part_stride, status);
    count_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (G > 1) {
        const int64_t cb = (n + 255) / 256;
        combine_kernel<<<(unsigned)cb, 256, 0, s>>>(part, part_stride, (int)G, n, idx, dist, blocksum);
        count_launch();
        *nblocksum = (int)cb;
    } else {
        *nblocksum = (int)row_blocks;
    }
    return cudaGetLastError();
}

cudaError_t launch_sum_blocks(const double *blocksum, int nblocks, double *out, cudaStream_t s) {
    sum_blocks_kernel<<<1, 256, 0, s>>>(blocksum, nblocks, out);
    count_launch();
    return cudaGetLastError();
}

}  // namespace kq
