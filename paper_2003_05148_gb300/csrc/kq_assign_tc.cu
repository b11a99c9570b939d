// kq_assign_tc.cu -- assignment step (Sec. 3.1, Eq. 1) with the certified test on
// the 5th-generation tensor cores (tcgen05, sm_103a).
//
// Same answer as kq_assign.cu (the fp32 direct-form argmin, lowest index on ties);
// only the cheap test that rules codewords out moves to the tensor cores:
//
//   e = x . c - h for a 128-row x 128-codeword tile is one GEMM, kind::tf32. The
//   tensor core truncates fp32 operands to tf32 (relative error < 2^-10 each;
//   measured: products match truncated inputs to fp32 accumulation error). To keep
//   fp32-like accuracy every value is split exactly into v = v_hi + v_lo with v_hi
//   = v truncated to tf32, and the three significant cross terms go side by side
//   along the GEMM's K dimension (K = 32, two MMAs per 16-column half):
//     A[i] = ( x_hi,  1,     x_hi,  1,     x_lo, 0, 0, 0 )
//     B[k] = ( c_hi, -h_hi,  c_lo, -h_lo,  c_hi, 0, 0, 0 )     (9 + 1 + 9 + 1 + 9 + 3)
//   so e_tc = x.c - h - x_lo.c_lo + (truncation of the lo parts) + (fp32 accumulation):
//   |e_tc - e| <= (3 * 2^-20 + 29 * 2^-23) (sum |x_j c_j| + |h|) < 2^-16 (|x| Cmax + Hmax),
//   plus an absolute 2^-120 (Cmax + |x| + 1) for subnormal inputs flushed to zero.
//   With that bound in place of the fp32 one, the threshold test of kq_assign.cu
//   is unchanged: e_tc < thr proves D_dir > best. Codewords that pass get the exact
//   fp32 direct form on the CUDA cores, reading c = c_hi + c_lo (exact) from the
//   shared tile.
//
// Warp roles in a CTA of 320 threads that owns 256 kernels (two 128-row MMA tiles):
//   warp 0      producer: streams packed codeword tiles (128 codewords x 128 B,
//               already in the tensor-core layout) into a 4-stage shared ring with
//               one bulk asynchronous copy per tile (TMA engine), mbarrier tx counts;
//   warp 1      owns TMEM (all 512 columns: two buffers x two row tiles x 128
//               columns) and issues the MMAs from one thread; tcgen05.commit
//               publishes the TMEM buffer;
//   warps 2-9   epilogue: one kernel (row) per thread; per tile, tcgen05.ld 32
//               columns at a time, max, compare with the row's threshold, exact
//               pass for the rare candidates from the shared tile, then release
//               the TMEM buffer and the shared stage.
// Every wait is bounded; a wait that runs out sets KQ_FLAG_TIMEOUT and an abort
// word, every role then drains out, and warp 1 frees TMEM before the CTA exits.
#include "kq_internal.cuh"

namespace kq {

constexpr int TC_M = 128;                  // rows per MMA tile
constexpr int TC_RT = 2;                   // row tiles per CTA
constexpr int TC_ROWS = TC_M * TC_RT;      // kernels per CTA
constexpr int TC_N = 128;                  // codewords per tile
constexpr int TC_KD = 32;                  // K of the GEMM (hi/lo split, see top of file)
constexpr int TC_STAGES = 4;
constexpr int TC_TILE_BYTES = TC_N * TC_KD * 4;  // 16 KiB per codeword tile
constexpr int TC_A_BYTES = TC_M * TC_KD * 4;     // 16 KiB per row tile
constexpr int TC_THREADS = 320;
constexpr int TC_EPI_WARPS = 8;
constexpr uint32_t TC_COLS = 512;          // TMEM columns allocated (2 buffers x 2 row tiles x 128)
constexpr uint32_t TC_LBO = 128;           // K-adjacent core matrices (8 rows x 16 B each)
constexpr uint32_t TC_SBO = TC_KD / 4 * 128; // next 8-row group (8 core matrices along K)
constexpr long long TC_WAIT_LIMIT = 4000000;
constexpr float G_TC = 1.52587890625e-5f;  // 2^-16 (see top of file)
constexpr float ONE_M_G11_TC = 0.9999993f; // <= 1 - gamma_11 (direct-form bound)

// Byte offset of element (row, k) in a K-major, no-swizzle core-matrix tile.
__host__ __device__ __forceinline__ uint32_t tc_offset(int row, int k) {
    return (uint32_t)(row / 8) * TC_SBO + (uint32_t)(k / 4) * TC_LBO + (uint32_t)(row % 8) * 16 + (uint32_t)(k % 4) * 4;
}

__device__ __forceinline__ uint64_t tc_smem_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFF);
    d |= (uint64_t)((TC_LBO >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((TC_SBO >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version for sm_100-class tcgen05; no swizzle, base offset 0
    return d;
}

// kind::tf32 instruction descriptor: D f32, A and B tf32, both K-major, M x N.
__host__ __device__ constexpr uint32_t tc_idesc(int m, int n) {
    return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}

// Bounded wait for the phase with the given parity; false if it ran out or the CTA aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, volatile uint32_t *abort_flag,
                                          uint32_t *status) {
    for (long long it = 0; it < TC_WAIT_LIMIT; ++it) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(done)
            : "r"(a), "r"(parity)
            : "memory");
        if (done) return true;
        if ((it & 255) == 255 && *abort_flag) return false;
    }
    *abort_flag = 1u;
    set_flag(status, KQ_FLAG_TIMEOUT);
    return false;
}

// 32 consecutive TMEM columns of this warp's 32 lanes (one row per thread).
__device__ __forceinline__ void tc_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

// v = hi + lo exactly, hi = v truncated to tf32 (10 explicit mantissa bits).
__device__ __forceinline__ float tf32_hi(float v) { return __uint_as_float(__float_as_uint(v) & 0xFFFFE000u); }

// Slot s of the K = 32 row layout for one operand (see top of file). `a_side`
// selects the A pattern (x_hi, 1, x_hi, 1, x_lo) or the B pattern (c_hi, -h_hi,
// c_lo, -h_lo, c_hi); v holds the 9 values, extra the 10th (1 for A, -h for B).
__device__ __forceinline__ void tc_row(const float (&v)[D], float extra, bool a_side, float (&out)[TC_KD]) {
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const float hi = tf32_hi(v[j]), lo = v[j] - hi;
        out[j] = hi;
        out[10 + j] = a_side ? hi : lo;
        out[20 + j] = a_side ? lo : hi;
    }
    const float ehi = tf32_hi(extra);
    out[D] = a_side ? 1.f : ehi;
    out[19] = a_side ? 1.f : extra - ehi;
    out[29] = out[30] = out[31] = 0.f;
}

// Packs C into tensor-core tiles (Kpad codewords, Kpad a multiple of TC_N) and
// reduces the same codebook bounds as pack_codebook_kernel into hdr->cb_*.
// Padding codewords get c = 0 and -h = -inf, so their e is -inf.
__global__ void __launch_bounds__(256) pack_codebook_tc_kernel(const float *__restrict__ C, int32_t K, int32_t Kpad,
                                                               float *__restrict__ Cpk, Header *hdr) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    float cmax = 0.f, hmax = 0.f, qmax = 0.f;
    if (k < Kpad) {
        float c[D];
        float mh = __int_as_float(0xff800000);  // -h; -inf for padding codewords
#pragma unroll
        for (int j = 0; j < D; ++j) c[j] = 0.f;
        if (k < K) {
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
            const float h = 0.5f * s;
            const float h2 = h + h;
            mh = -h;
            cmax = __fsqrt_ru(c2hi);
            hmax = fabsf(h);
            qmax = fmaxf(fabsf(__fsub_ru(c2hi, h2)), fabsf(__fsub_rd(c2lo, h2)));
            if (!ok) {
                set_flag(&hdr->status, KQ_FLAG_NONFINITE);
                cmax = hmax = qmax = __int_as_float(0x7fc00000);  // NaN: disables the test
            }
        }
        float v[TC_KD];
        tc_row(c, mh, false, v);
        if (!(mh >= -3.402823466e38f)) v[19] = 0.f;  // padding: -inf already sits in the hi slot
        unsigned char *tile = reinterpret_cast<unsigned char *>(Cpk) + (int64_t)(k / TC_N) * TC_TILE_BYTES;
        const int kl = k % TC_N;
#pragma unroll
        for (int q = 0; q < TC_KD / 4; ++q)
            *reinterpret_cast<float4 *>(tile + tc_offset(kl, 4 * q)) =
                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    }
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

__device__ __forceinline__ float tc_threshold(float x2lo, float slack, float b) {
    const float t = __fmul_rd(__fsub_rd(__fsub_rd(x2lo, slack), __fdiv_ru(b, ONE_M_G11_TC)), 0.5f);
    return t == t ? t : __int_as_float(0xff800000);
}

__device__ __forceinline__ float direct_distance(const float (&x)[D], const float *__restrict__ c) {
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const float t = x[j] - c[j];
        acc = fmaf(t, t, acc);
    }
    return acc;
}

struct TcShared {
    unsigned char a[TC_RT][TC_A_BYTES];             // row tiles (tensor-core layout)
    unsigned char b[TC_STAGES][TC_TILE_BYTES];      // codeword tiles
    unsigned long long full[TC_STAGES], empty[TC_STAGES], tfull[2], tempty[2], done;
    uint32_t tmem_base;
    uint32_t abort_flag;
    double wsum[TC_EPI_WARPS];
};

__global__ void __launch_bounds__(TC_THREADS, 1)
assign_tc_kernel(const float *__restrict__ W, int64_t n, const float *__restrict__ C, const float *__restrict__ Cpk,
                 int32_t K, int32_t ntiles, const int32_t *hint, int32_t *idx, float *__restrict__ dist,
                 double *__restrict__ blocksum, Header *hdr) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    TcShared &S = *reinterpret_cast<TcShared *>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile uint32_t *abort_flag = &S.abort_flag;
    uint32_t *status = &hdr->status;

    // ---- epilogue threads: own one kernel each; load it, bounds, warm start, A tile row
    const bool epi = warp >= 2;
    const int q = warp & 3;                           // TMEM lane quarter this warp may access
    const int half = epi ? (warp - 2) / 4 : 0;        // row tile
    const int rloc = half * TC_M + q * 32 + lane;     // row within the CTA
    const int64_t row = (int64_t)blockIdx.x * TC_ROWS + rloc;
    float x[D];
    float x2lo = 0.f, slack = 0.f, best = __int_as_float(0x7f800000), thr = __int_as_float(0xff800000);
    int32_t bi = 0;
    if (epi) {
#pragma unroll
        for (int j = 0; j < D; ++j) x[j] = row < n ? W[row * D + j] : 0.f;
        bool ok = true;
#pragma unroll
        for (int j = 0; j < D; ++j) ok &= isfinite(x[j]);
        if (row < n && !ok) set_flag(status, KQ_FLAG_NONFINITE);
        const float cmax = __uint_as_float(__ldcg(&hdr->cb_cmax));
        const float hmax = __uint_as_float(__ldcg(&hdr->cb_hmax));
        const float qmax = __uint_as_float(__ldcg(&hdr->cb_qmax));
        float hi = 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            x2lo = __fadd_rd(x2lo, __fmul_rd(x[j], x[j]));
            hi = __fadd_ru(hi, __fmul_ru(x[j], x[j]));
        }
        const float xn = __fsqrt_ru(hi);
        slack = __fadd_ru(qmax, __fmul_ru(2.f * G_TC, __fadd_ru(hmax, __fmul_ru(xn, cmax))));
        // absolute part: tf32 inputs below 2^-126 may be flushed to zero; each such
        // term is below 2^-126 times the other factor
        slack = __fadd_ru(slack, __fmul_ru(7.52316384526264e-37f /* 2^-120 */, __fadd_ru(__fadd_ru(cmax, xn), 1.f)));
        if (hint != nullptr && row < n) {
            const int32_t h = hint[row];
            if ((uint32_t)h < (uint32_t)K) {
                const float d = direct_distance(x, C + (int64_t)h * D);
                if (d < best) {
                    best = d;
                    bi = h;
                    thr = tc_threshold(x2lo, slack, d);
                }
            }
        }
        float a[TC_KD];
        tc_row(x, 1.f, true, a);
        const int r = q * 32 + lane;
#pragma unroll
        for (int u = 0; u < TC_KD / 4; ++u)
            *reinterpret_cast<float4 *>(&S.a[half][tc_offset(r, 4 * u)]) = make_float4(a[4 * u], a[4 * u + 1], a[4 * u + 2], a[4 * u + 3]);
    }

    // ---- barriers and TMEM
    if (tid == 0) {
        for (int s = 0; s < TC_STAGES; ++s) {
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.full[s]), 1);
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.empty[s]), TC_EPI_WARPS);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.tfull[b]), 1);
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.tempty[b]), TC_EPI_WARPS);
        }
        mbar_init((uint32_t)__cvta_generic_to_shared(&S.done), 1);
        S.abort_flag = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         (uint32_t)__cvta_generic_to_shared(&S.tmem_base)),
                     "r"(TC_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // A tiles -> tensor core
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = S.tmem_base;

    if (warp == 0) {
        // ---- producer
        if (lane == 0) {
            for (int i = 0; i < ntiles; ++i) {
                const int s = i % TC_STAGES;
                if (i >= TC_STAGES &&
                    !mbar_wait((uint32_t)__cvta_generic_to_shared(&S.empty[s]), ((i / TC_STAGES) - 1) & 1, abort_flag,
                               status))
                    break;
                const uint32_t fb = (uint32_t)__cvta_generic_to_shared(&S.full[s]);
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb), "r"(TC_TILE_BYTES)
                             : "memory");
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                        (uint32_t)__cvta_generic_to_shared(S.b[s])),
                    "l"(reinterpret_cast<const unsigned char *>(Cpk) + (int64_t)i * TC_TILE_BYTES), "r"(TC_TILE_BYTES),
                    "r"(fb)
                    : "memory");
            }
        }
    } else if (warp == 1) {
        // ---- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = tc_idesc(TC_M, TC_N);
            const uint32_t a0 = (uint32_t)__cvta_generic_to_shared(S.a[0]);
            for (int i = 0; i < ntiles; ++i) {
                const int s = i % TC_STAGES, b = i & 1;
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.full[s]), (i / TC_STAGES) & 1, abort_flag, status))
                    break;
                if (i >= 2 && !mbar_wait((uint32_t)__cvta_generic_to_shared(&S.tempty[b]), ((i / 2) - 1) & 1,
                                         abort_flag, status))
                    break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t b0 = (uint32_t)__cvta_generic_to_shared(S.b[s]);
#pragma unroll
                for (int r = 0; r < TC_RT; ++r) {
                    const uint32_t dcol = tmem + (uint32_t)(b * TC_RT * TC_N + r * TC_N);
#pragma unroll
                    for (int kb = 0; kb < TC_KD / 8; ++kb) {
                        const uint64_t ad = tc_smem_desc(a0 + r * TC_A_BYTES + kb * 2 * TC_LBO);
                        const uint64_t bd = tc_smem_desc(b0 + kb * 2 * TC_LBO);  // 8 tf32 of K per MMA
                        asm volatile(
                            "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                            " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}" ::"r"(dcol),
                            "l"(ad), "l"(bd), "r"(idesc), "r"((uint32_t)kb)
                            : "memory");
                    }
                }
                asm volatile(
                    "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                        (uint32_t)__cvta_generic_to_shared(&S.tfull[b]))
                    : "memory");
            }
            // every MMA this thread issued has finished before TMEM can be freed
            const uint32_t db = (uint32_t)__cvta_generic_to_shared(&S.done);
            asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(db)
                         : "memory");
            for (long long it = 0; it < TC_WAIT_LIMIT; ++it) {
                uint32_t ok;
                asm volatile(
                    "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
                    : "=r"(ok)
                    : "r"(db)
                    : "memory");
                if (ok) break;
                if (it + 1 == TC_WAIT_LIMIT) set_flag(status, KQ_FLAG_TIMEOUT);
            }
        }
    } else {
        // ---- epilogue: one row per thread
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        for (int i = 0; i < ntiles; ++i) {
            const int b = i & 1, st = i % TC_STAGES;
            if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.tfull[b]), (i / 2) & 1, abort_flag, status)) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t col0 = (uint32_t)(b * TC_RT * TC_N + half * TC_N);
            const unsigned char *tile = S.b[st];
#pragma unroll 1
            for (int c = 0; c < TC_N; c += 32) {
                float v[32];
                tc_ld32(tmem + lane_base + col0 + (uint32_t)c, v);
                float m0 = fmaxf(fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3])), fmaxf(fmaxf(v[4], v[5]), fmaxf(v[6], v[7])));
                float m1 = fmaxf(fmaxf(fmaxf(v[8], v[9]), fmaxf(v[10], v[11])), fmaxf(fmaxf(v[12], v[13]), fmaxf(v[14], v[15])));
                float m2 = fmaxf(fmaxf(fmaxf(v[16], v[17]), fmaxf(v[18], v[19])), fmaxf(fmaxf(v[20], v[21]), fmaxf(v[22], v[23])));
                float m3 = fmaxf(fmaxf(fmaxf(v[24], v[25]), fmaxf(v[26], v[27])), fmaxf(fmaxf(v[28], v[29]), fmaxf(v[30], v[31])));
                const float m = fmaxf(fmaxf(m0, m1), fmaxf(m2, m3));
                // A NaN test value only arises when the row's threshold is already -inf
                // (non-finite or overflowing inputs), where every chunk takes this path.
                if (!(m < thr)) {  // rare: some codeword of these 32 may improve or tie
                    // candidate mask with static indexing, so v stays in registers
                    uint32_t mask = 0u;
#pragma unroll
                    for (int j = 0; j < 32; ++j) mask |= (v[j] < thr) ? 0u : (1u << j);
                    while (mask) {
                        const int j = __ffs(mask) - 1;
                        mask &= mask - 1u;
                        const int kl = c + j;
                        const int32_t k = i * TC_N + kl;
                        if (k >= K) break;
                        float cw[D];
#pragma unroll
                        for (int u = 0; u < D; ++u)
                            cw[u] = *reinterpret_cast<const float *>(tile + tc_offset(kl, u)) +
                                    *reinterpret_cast<const float *>(tile + tc_offset(kl, 10 + u));  // c_hi + c_lo = c
                        const float d = direct_distance(x, cw);
                        if (d < best || (d == best && k < bi)) {
                            best = d;
                            bi = k;
                            thr = tc_threshold(x2lo, slack, d);
                        }
                    }
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) {
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"((uint32_t)__cvta_generic_to_shared(&S.tempty[b]))
                             : "memory");
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"((uint32_t)__cvta_generic_to_shared(&S.empty[st]))
                             : "memory");
            }
        }
        if (row < n) {
            idx[row] = bi;
            if (dist) dist[row] = best;
        }
    }

    // ---- objective partial sum (fixed order) and teardown
    double sum = (epi && row < n) ? (double)best : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (epi && lane == 0) S.wsum[warp - 2] = sum;
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (tid == 0) {
        double s = 0.0;
        for (int w = 0; w < TC_EPI_WARPS; ++w) s += S.wsum[w];
        blocksum[blockIdx.x] = s;
    }
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TC_COLS) : "memory");
    }
}

int32_t tc_kpad(int32_t K) { return (K + TC_N - 1) / TC_N * TC_N; }

bool tc_eligible(int64_t n, int num_sms) { return n >= (int64_t)TC_ROWS * num_sms; }

cudaError_t launch_pack_codebook_tc(const float *C, int32_t K, float *Cpk, Header *hdr, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(&hdr->cb_cmax, 0, 3 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    const int32_t Kpad = tc_kpad(K);
    pack_codebook_tc_kernel<<<(Kpad + 255) / 256, 256, 0, s>>>(C, K, Kpad, Cpk, hdr);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_assign_tc(const float *W, int64_t n, const float *C, const float *Cpk, int32_t K,
                             const int32_t *hint, int32_t *idx, float *dist, double *blocksum, int *nblocksum,
                             Header *hdr, cudaStream_t s) {
    // More shared memory than two CTAs can share, so one CTA per SM owns all of TMEM.
    const int smem = 120 * 1024;
    static_assert(sizeof(TcShared) + 1024 <= 120 * 1024, "shared layout too large");
    cudaError_t e = cudaFuncSetAttribute(assign_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int64_t blocks = (n + TC_ROWS - 1) / TC_ROWS;
    const int32_t ntiles = tc_kpad(K) / TC_N;
    assign_tc_kernel<<<(unsigned)blocks, TC_THREADS, smem, s>>>(W, n, C, Cpk, K, ntiles, hint, idx, dist, blocksum, hdr);
    count_launch();
    *nblocksum = (int)blocks;
    return cudaGetLastError();
}

}  // namespace kq
