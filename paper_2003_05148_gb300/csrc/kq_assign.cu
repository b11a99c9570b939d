// kq_assign.cu -- assignment step of KQ's k-means (Sec. 3.1, Eq. 1) on sm_103a.
//
// The result is exactly the fp32 direct-form argmin (9 FSUB + 9 FFMA per kernel x
// codeword pair, lowest index on ties). Most pairs are settled by a cheaper,
// certified test instead of the direct form:
//
//   expanded form   e = sum_j x_j c_j - h   (9 FFMA from -h, h ~ |c|^2 / 2), so
//                   D = |x - c|^2 = |x|^2 + (|c|^2 - 2h) - 2 sum_j x_j c_j exactly.
//   error bounds    fl(e) is within g9 (|h| + |x||c|) of e (recursive FMA sum of 10
//                   terms, g9 >= 9u/(1-9u), u = 2^-24), and the fp32 direct form
//                   D_dir >= D (1 - g11) (nine non-negative terms, g11 >= 11u/(1-11u)).
//   (plus an absolute 2^-126 for underflowing intermediate results),
//   so with Cmax >= |c|, Hmax >= |h|, Qmax >= ||c|^2 - 2h| over the codebook and
//   X2lo <= |x|^2, fl(e) < thr := (X2lo - Qmax - 2 g9 (Hmax + |x| Cmax) - best/(1-g11)) / 2
//   implies D_dir > best: the codeword cannot improve (or tie) the running best and
//   is skipped. thr is evaluated with directed rounding so that the rounded value
//   never exceeds the exact one; NaN thresholds become -inf (skip nothing).
//
// Only codewords that pass the test (the running records and near-ties) get the
// exact direct form, so the steady state costs 9 FP32-pipe lane ops per pair.
//
// Layout: a CTA owns ROW_BLOCK = 1024 kernels: 128 threads x 8 rows, held in
// registers as four fp32x2 row pairs (fma.rn.f32x2 / sub.rn.f32x2: one packed
// instruction evaluates a codeword against two kernels, each lane an IEEE fp32 op,
// bit-identical to the scalar form). Codewords are packed once per call into
// 80-byte rows of duplicated pairs (c_j, c_j), j = 0..8, plus (-h, -h), staged 256
// at a time in shared memory and read with broadcast LDS.128. Small n: the codebook
// is split over gridDim.y CTAs and the per-split winners are merged
// lexicographically on (distance bits, k), which is exact. An optional warm start
// (a previous assignment) seeds each row's running best, which removes most
// record updates in later Lloyd iterations; the tie rule keeps the lowest index.
// The Eq. 1 objective is reduced per CTA in a fixed order (bitwise reproducible).
#include "kq_internal.cuh"

namespace kq {

constexpr int A_THREADS = 128;
constexpr int A_ROWS = 8;    // rows per thread (four fp32x2 pairs)
constexpr int A_TILE = 256;  // codewords per shared-memory tile (20 KiB)
static_assert(A_THREADS * A_ROWS == ROW_BLOCK, "row block mismatch");
constexpr float G9 = 6.0e-7f;           // >= gamma_9 = 9u / (1 - 9u) = 5.364e-7
constexpr float ONE_M_G11 = 0.9999993f;  // <= 1 - gamma_11 = 1 - 6.557e-7

__global__ void pack_codebook_kernel(const float *__restrict__ C, int32_t K, float *__restrict__ Cd, Header *hdr) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    float cmax = 0.f, hmax = 0.f, qmax = 0.f;
    if (k < K) {
        float c[D];
        bool ok = true;
        float s = 0.f, c2lo = 0.f, c2hi = 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            c[j] = C[(int64_t)k * D + j];
            ok &= isfinite(c[j]);
            s = fmaf(c[j], c[j], s);
            c2lo = __fadd_rd(c2lo, __fmul_rd(c[j], c[j]));
            c2hi = __fadd_ru(c2hi, __fmul_ru(c[j], c[j]));
        }
        if (!ok) set_flag(&hdr->status, KQ_FLAG_NONFINITE);
        const float h = 0.5f * s;
        const float h2 = h + h;  // exact
        cmax = __fsqrt_ru(c2hi);
        hmax = fabsf(h);
        qmax = fmaxf(fabsf(__fsub_ru(c2hi, h2)), fabsf(__fsub_rd(c2lo, h2)));
        if (!ok) cmax = hmax = qmax = __int_as_float(0x7fc00000);  // NaN: disables the filter
        float4 *dst = reinterpret_cast<float4 *>(Cd + (int64_t)k * CD_FLOATS);
        dst[0] = make_float4(c[0], c[0], c[1], c[1]);
        dst[1] = make_float4(c[2], c[2], c[3], c[3]);
        dst[2] = make_float4(c[4], c[4], c[5], c[5]);
        dst[3] = make_float4(c[6], c[6], c[7], c[7]);
        dst[4] = make_float4(c[8], c[8], -h, -h);
    }
    // non-negative floats (and NaN, which must win) order like their bit patterns
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        cmax = __uint_as_float(max(__float_as_uint(cmax), __shfl_xor_sync(0xffffffffu, __float_as_uint(cmax), o)));
        hmax = __uint_as_float(max(__float_as_uint(hmax), __shfl_xor_sync(0xffffffffu, __float_as_uint(hmax), o)));
        qmax = __uint_as_float(max(__float_as_uint(qmax), __shfl_xor_sync(0xffffffffu, __float_as_uint(qmax), o)));
    }
    if ((threadIdx.x & 31) == 0) {
        atomicMax(&hdr->cb_cmax, __float_as_uint(cmax));
        atomicMax(&hdr->cb_hmax, __float_as_uint(hmax));
        atomicMax(&hdr->cb_qmax, __float_as_uint(qmax));
    }
}

// Threshold of the certified test for a row with running best `b` (see top of file).
__device__ __forceinline__ float filter_threshold(float x2lo, float slack, float b) {
    const float t = __fmul_rd(__fsub_rd(__fsub_rd(x2lo, slack), __fdiv_ru(b, ONE_M_G11)), 0.5f);
    return t == t ? t : __int_as_float(0xff800000);
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

__global__ void __launch_bounds__(A_THREADS, 3)
assign_kernel(const float *__restrict__ W, int64_t n, const float *__restrict__ Cd, const float *__restrict__ C,
              int32_t K, int32_t kps, const int32_t *hint, int32_t *idx, float *__restrict__ dist,
              double *__restrict__ blocksum, unsigned long long *__restrict__ part, int64_t part_stride,
              Header *hdr) {
    constexpr int P = A_ROWS / 2;
    __shared__ __align__(16) float4 sm[A_TILE * (CD_FLOATS / 4)];

    const int64_t row0 = ((int64_t)blockIdx.x * A_THREADS + threadIdx.x) * A_ROWS;
    float w[A_ROWS * D];
    if (row0 + A_ROWS <= n) {
        const float4 *src = reinterpret_cast<const float4 *>(W + row0 * D);
#pragma unroll
        for (int v = 0; v < A_ROWS * D / 4; ++v) {
            const float4 t = __ldg(src + v);
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
        if (!ok) set_flag(&hdr->status, KQ_FLAG_NONFINITE);
    }
    const float cmax = __uint_as_float(__ldcg(&hdr->cb_cmax));
    const float hmax = __uint_as_float(__ldcg(&hdr->cb_hmax));
    const float qmax = __uint_as_float(__ldcg(&hdr->cb_qmax));

    const int32_t kb = blockIdx.y * kps;
    const int32_t ke = min(K, kb + kps);
    float x2lo[A_ROWS], slack[A_ROWS], best[A_ROWS], thr[A_ROWS];
    int32_t bi[A_ROWS];
#pragma unroll
    for (int r = 0; r < A_ROWS; ++r) {
        float lo = 0.f, hi = 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            lo = __fadd_rd(lo, __fmul_rd(w[r * D + j], w[r * D + j]));
            hi = __fadd_ru(hi, __fmul_ru(w[r * D + j], w[r * D + j]));
        }
        x2lo[r] = lo;
        slack[r] = __fadd_ru(qmax, __fmul_ru(2.f * G9, __fadd_ru(hmax, __fmul_ru(__fsqrt_ru(hi), cmax))));
        slack[r] = __fadd_ru(slack[r], 1.1754944e-38f);  // absolute part: underflow of the 9 FMAs, < 20 * 2^-150
        best[r] = __int_as_float(0x7f800000);  // +inf
        bi[r] = kb;
        thr[r] = __int_as_float(0xff800000);   // -inf: nothing is skipped
        if (hint != nullptr && row0 + r < n) {
            const int32_t h = hint[row0 + r];
            if ((uint32_t)h < (uint32_t)K) {
                float acc = 0.f;
#pragma unroll
                for (int j = 0; j < D; ++j) {
                    const float t = w[r * D + j] - C[(int64_t)h * D + j];
                    acc = fmaf(t, t, acc);
                }
                if (acc < best[r]) {  // a NaN or +inf warm start is no start
                    best[r] = acc;
                    bi[r] = h;
                    thr[r] = filter_threshold(x2lo[r], slack[r], acc);
                }
            }
        }
    }

    unsigned long long X[P][D];
#pragma unroll
    for (int p = 0; p < P; ++p)
#pragma unroll
        for (int j = 0; j < D; ++j) X[p][j] = pack2(w[(2 * p) * D + j], w[(2 * p + 1) * D + j]);

    for (int32_t kt = kb; kt < ke; kt += A_TILE) {
        const int cnt = min(A_TILE, ke - kt);
        __syncthreads();
        const float4 *gsrc = reinterpret_cast<const float4 *>(Cd + (int64_t)kt * CD_FLOATS);
        for (int v = threadIdx.x; v < cnt * (CD_FLOATS / 4); v += A_THREADS) sm[v] = __ldg(gsrc + v);
        __syncthreads();
#pragma unroll 1
        for (int c = 0; c < cnt; ++c) {
            const ulonglong2 *cw = reinterpret_cast<const ulonglong2 *>(&sm[c * (CD_FLOATS / 4)]);
            const ulonglong2 c01 = cw[0], c23 = cw[1], c45 = cw[2], c67 = cw[3], c8h = cw[4];
            const unsigned long long Cj[D] = {c01.x, c01.y, c23.x, c23.y, c45.x, c45.y, c67.x, c67.y, c8h.x};
            bool pass[P];
            bool any = false;
#pragma unroll
            for (int p = 0; p < P; ++p) {
                unsigned long long e = c8h.y;  // (-h, -h)
#pragma unroll
                for (int j = 0; j < D; ++j) e = fma2(X[p][j], Cj[j], e);
                float e0, e1;
                unpack2(e, e0, e1);
                pass[p] = !(e0 < thr[2 * p]) || !(e1 < thr[2 * p + 1]);
                any |= pass[p];
            }
            if (any) {
                const int32_t k = kt + c;
#pragma unroll
                for (int p = 0; p < P; ++p) {
                    if (!pass[p]) continue;
                    unsigned long long t = sub2(X[p][0], Cj[0]);
                    unsigned long long acc = mul2(t, t);  // == fma(t, t, +0) bit for bit
#pragma unroll
                    for (int j = 1; j < D; ++j) {
                        t = sub2(X[p][j], Cj[j]);
                        acc = fma2(t, t, acc);
                    }
                    float d[2];
                    unpack2(acc, d[0], d[1]);
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        const int r = 2 * p + q;
                        if (d[q] < best[r] || (d[q] == best[r] && k < bi[r])) {
                            best[r] = d[q];
                            bi[r] = k;
                            thr[r] = filter_threshold(x2lo[r], slack[r], d[q]);
                        }
                    }
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

cudaError_t launch_pack_codebook(const float *C, int32_t K, float *Cd, Header *hdr, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(&hdr->cb_cmax, 0, 3 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    launch_begin(s);
    pack_codebook_kernel<<<(K + 255) / 256, 256, 0, s>>>(C, K, Cd, hdr);
    launch_end(s, "pack_codebook_kernel");
    return cudaGetLastError();
}

cudaError_t launch_assign(const float *W, int64_t n, const float *Cd, const float *C, int32_t K, const int32_t *hint,
                          int32_t *idx, float *dist, double *blocksum, int *nblocksum, unsigned long long *part,
                          Header *hdr, int num_sms, cudaStream_t s) {
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, assign_kernel, A_THREADS, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int64_t row_blocks = (n + ROW_BLOCK - 1) / ROW_BLOCK;
    const int64_t target = (int64_t)per_sm * num_sms;  // one full wave of resident CTAs
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
    launch_begin(s);
    assign_kernel<<<grid, A_THREADS, 0, s>>>(W, n, Cd, C, K, kps, hint, idx, dist, blocksum, part, part_stride, hdr);
    launch_end(s, "assign_kernel");
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (G > 1) {
        const int64_t cb = (n + 255) / 256;
        launch_begin(s);
        combine_kernel<<<(unsigned)cb, 256, 0, s>>>(part, part_stride, (int)G, n, idx, dist, blocksum);
        launch_end(s, "combine_kernel");
        *nblocksum = (int)cb;
    } else {
        *nblocksum = (int)row_blocks;
    }
    return cudaGetLastError();
}

cudaError_t launch_sum_blocks(const double *blocksum, int nblocks, double *out, cudaStream_t s) {
    launch_begin(s);
    sum_blocks_kernel<<<1, 256, 0, s>>>(blocksum, nblocks, out);
    launch_end(s, "sum_blocks_kernel");
    return cudaGetLastError();
}

}  // namespace kq
