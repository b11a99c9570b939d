// kq_assign_tc.cu -- assignment step (Sec. 3.1, Eq. 1) with the certified test on
// the 5th-generation tensor cores (tcgen05, sm_103a).
//
// Same answer as kq_assign.cu (the fp32 direct-form argmin, lowest index on ties);
// only the cheap test that rules codewords out moves to the tensor cores, and the
// row's threshold moves into the GEMM so that the test is one sign bit:
//
//   g = x . c - h - R - T' for a 128-row x 256-codeword tile is one GEMM,
//   kind::f16 (fp16 operands, fp32 accumulation; twice the tf32 rate). All values
//   are first scaled by one power of two beta per call (the codebook's largest
//   norm lands in [32, 64), so every operand sits well inside the fp16 range);
//   that scales g by beta^2 and leaves its sign alone, and every quantity below is
//   in scaled units. To keep fp32-like accuracy each value is split into
//   v = v_hi + v_lo + d, v_hi = v truncated to fp16, v_lo = (v - v_hi) truncated
//   to fp16, and the three significant cross terms go side by side along the
//   GEMM's K dimension (K = 32):
//     A[i] = ( x_hi,  1,     x_hi,  1,     x_lo,  -T'0, -R, -T'1 )
//     B[k] = ( c_hi, -h_hi,  c_lo, -h_lo,  c_hi,  s0,    1,  s1  )   (9 + 1 + 9 + 1 + 9 + 3)
//   where (s0, s1) = (1, 0) for the first 128 codewords of a tile and (0, 1) for
//   the other 128, so each half of a tile row sees its own T' (each half is tested
//   by its own thread, with its own running best). R (fixed per row, about
//   |x|^2 / 2) and T' are normal fp16 values or 0, so they are exact operands
//   even for a tensor core that flushes fp16 subnormals; the other half's T'
//   meets an exact 0. |d| <= 2^-20 |v| + 2^-13 (relative while v_lo is a normal
//   fp16 value, absolute below that, flushed subnormals included); products of
//   fp16 values are exact in fp32, so dropping x_lo.c_lo and accumulating 31
//   products in fp32 give
//     |g - (e - R - T')| <= E = 2^-16 (|x| Cmax + Hmax + |R| + |T'|) + 2^-11 (|x| + Cmax + 1)
//   (3 * 2^-20 + 31 * 2^-23 (1 + 2^-8) < 2^-16 on the first group, 31 * 2^-23 on R
//   and T'; 3 * 2^-13 (|x| + Cmax) + 2^-13 from the absolute parts of d, with
//   sum_j |v_j| <= 3 |v|, on the second). A row whose scaled norm exceeds 256 (R and
//   the products would leave the fp16 / exact-product range) enters the GEMM with
//   x = 0 and is tested exactly against every codeword.
//   The kernel keeps R + T' + E < thr0, where e < thr0 proves D_dir > best (the
//   test of kq_assign.cu without its arithmetic slack), so a negative g (sign bit
//   set, -0 included since E > 0) rules the codeword out. The TMEM load reduces as
//   it reads (tcgen05.ld.red.max, sm_103a): a 32-codeword chunk whose maximum g has
//   its sign bit set is ruled out with no further work (NaN test values, which the
//   maximum skips, only arise in rows whose thread tests every codeword anyway: see
//   -T' = 2^15 below). Only a chunk with a non-negative maximum sends the row to
//   the exact fp32 direct form on the CUDA cores, which reads c in fp32 from the
//   same shared stage (every streamed tile carries its codewords in fp32 after the
//   fp16 operands). When a row's best improves, its thread rewrites its T' (one
//   2-byte shared store). MMAs already issued, or issued before the
//   store is seen, use the older T', which satisfied the inequality for the older,
//   larger best, and so for the current one: the test stays sound at every moment.
//   A half row without a usable T' (no running best yet, non-finite or out-of-range
//   inputs) holds -T' = 2^15, finite so that the other half's 0 meets no
//   infinity, and its thread tests every codeword exactly.
//
// Warm starts (a hint per kernel): a row's own hinted codeword always passes the
// test (its distance is the best, which the test cannot rule out), so every row
// takes the exact path once per pass. With K >= 4096 the caller hands the kernel a
// permutation that groups rows by hint (hint_histogram / scan_counts /
// hint_scatter below); a warp's rows then share that tile and the warp takes the
// exact path once instead of once per distinct hint. The kernel's slot s works on
// row perm[s]; results do not depend on the order.
//
// Warp roles in a CTA of 352 threads that owns 256 kernels (two 128-row tiles):
//   warp 0      producer: streams packed codeword tiles (256 codewords x 100 B:
//               64 B of fp16 operands in the tensor-core layout, then 36 B of fp32
//               codeword) into a 6-stage shared ring with one bulk asynchronous
//               copy per tile (TMA engine), mbarrier tx counts;
//   warps 1-2   MMA issuers, one per row tile (warp 1 also owns TMEM: 512 columns,
//               one 256-column accumulator per row tile): from one thread, the 2
//               MMAs (M = 128, N = 256, K = 16 each) of its row tile for a codeword
//               tile, then tcgen05.commit. The epilogue drains one accumulator
//               while the tensor core fills the other. Two issuers, because the
//               first shared-memory access (a barrier wait) of a thread after its
//               MMAs waits until they have executed: with one issuer the tensor
//               core would idle at every such wait, with two the other's MMAs run;
//   warps 3-10  epilogue: a thread owns one kernel in each row tile and one
//               128-codeword half of every tile: four reducing tcgen05.ld of 32
//               columns and one wait, the accumulator goes back at once, then the
//               sign test of the chunk maxima and the exact pass for the rare
//               candidates; the shared stage goes back when both row tiles are done.
//               The halves merge at the end.
// The producer and MMA loops run in lane 0 of their warps while lanes 1-31 wait at
// the CTA barrier that opens the teardown: a lone lane waits on a completed
// mbarrier phase in ~20 cycles, a whole warp (or a lane whose partners wait at a
// warp-level sync) in ~100-300, all of it idle time for the tensor core when it is
// the MMA issuer's. (Back to back, one thread's MMAs run at the full rate with N = 256
// or 128; here N = 128 jobs on two accumulators per row tile were slower. What
// bounds the kernel is the per-job hand-back: issue, execution, commit, TMEM loads,
// arrive and the next issue take ~880 cycles per row tile, of which only the other
// row tile's 256 cycles of MMA overlap.)
// Every wait is bounded; a wait that runs out sets KQ_FLAG_TIMEOUT and an abort
// word, every role then drains out, and warp 1 frees TMEM before the CTA exits.
#include <cuda_fp16.h>

#include "kq_internal.cuh"

namespace kq {

constexpr int TC_M = 128;                  // rows per MMA (row tile)
constexpr int TC_RT = 2;                   // row tiles per CTA
constexpr int TC_ROWS = TC_M * TC_RT;      // kernels per CTA
// Warm starts with 256 to 4096 codewords (no global hint order) group a CTA's rows by
// the 32-codeword chunk of their hint: at most 128 chunks, plus rows without a hint.
// In a fit's later passes (few rows change codeword) this keeps a warp's exact-path
// entries to its hints' few chunks: at n = 262,144, K = 512, 56 instead of 63 us per
// pass (VGG-16's 13 layers 19.6 instead of 20.3 ms per fit); the first warm pass after
// an update, where many rows move, gains nothing (85 us either way).
constexpr int32_t TC_LGROUP_MINK = 256;
constexpr int32_t TC_LGROUP_MAXK = 4096;
constexpr int TC_LBINS = TC_LGROUP_MAXK / 32 + 1;
// TC_N codewords per tile (N of every MMA), TC_KD = K of the GEMM in fp16 elements
// (hi/lo split, see top of file); a tile is TC_TILE_H bytes of fp16 operands and
// the tile's codewords in fp32, TC_TILE_BYTES = 25 KiB streamed (kq_internal.cuh).
constexpr int TC_HALF = TC_N / 2;          // codewords of a tile one epilogue thread tests
constexpr int TC_STAGES = 6;               // tile ring of the plain kernel
constexpr int TC_STAGES_YY = 4;            // and of the pruned one (its records take the rest; as fast)
constexpr int TC_A_BYTES = TC_M * TC_KD * 2;     // 8 KiB per row tile
constexpr int TC_THREADS = 352;
constexpr int TC_EPI_WARP0 = 3;            // first epilogue warp (0: producer, 1-2: MMA issuers)
constexpr int TC_EPI_WARPS = 8;
constexpr uint32_t TC_COLS = 512;          // TMEM columns allocated (2 row tiles x 256)
constexpr uint32_t TC_LBO = 128;           // K-adjacent core matrices (8 rows x 16 B each)
constexpr uint32_t TC_SBO = TC_KD / 8 * 128; // next 8-row group (4 core matrices along K)
constexpr long long TC_WAIT_LIMIT = 4000000;
constexpr float TWO_G_TC = 3.0517578125e-5f;  // 2 x 2^-16 (see top of file)
constexpr float TWO_ABS_TC = 9.765625e-4f;     // 2 x 2^-11: twice the absolute part of E, per unit of |x| + Cmax + 1
constexpr float INV_ONE_M_G11_TC = 1.0000008344650269f;  // 1 + 7 * 2^-23 >= 1 / (1 - gamma_11) (direct-form bound)
constexpr int TC_SLOT_T0 = 29, TC_SLOT_R = 30, TC_SLOT_T1 = 31;  // K slots of -T'0, -R, -T'1
constexpr float TC_T_EVERY = 32768.f;      // -T' of a half row tested exactly (finite in fp16)
constexpr float TC_T_LIMIT = 16384.f;      // |T'| bound that keeps -T' an fp16 operand
constexpr float TC_X_LIMIT = 256.f;        // scaled |x| above which a row is tested exactly
constexpr float F16_MIN_NORMAL = 6.103515625e-05f;  // 2^-14

// Byte offset of fp16 element (row, k) in a K-major, no-swizzle core-matrix tile.
__host__ __device__ __forceinline__ uint32_t tc_offset(int row, int k) {
    return (uint32_t)(row / 8) * TC_SBO + (uint32_t)(k / 8) * TC_LBO + (uint32_t)(row % 8) * 16 + (uint32_t)(k % 8) * 2;
}

__device__ __forceinline__ uint64_t tc_smem_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFF);
    d |= (uint64_t)((TC_LBO >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((TC_SBO >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version for sm_100-class tcgen05; no swizzle, base offset 0
    return d;
}

// kind::f16 instruction descriptor: D f32, A and B f16, both K-major, M x N.
__host__ __device__ constexpr uint32_t tc_idesc(int m, int n) {
    return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}

// Bounded wait for the phase with the given parity; false if it ran out (after
// `limit` polls) or the CTA aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, volatile uint32_t *abort_flag,
                                          uint32_t *status, long long limit) {
    for (long long it = 0; it < limit; ++it) {
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

// Starts loading 32 consecutive TMEM columns of this warp's 32 lanes (one row per
// thread) into r, and their maximum (NaN skipped, as fmaxf) into m; both are valid
// only after tcgen05.wait::ld.
__device__ __forceinline__ void tc_ld32_max(uint32_t taddr, uint32_t (&r)[32], float &m) {
    asm volatile(
        "tcgen05.ld.red.sync.aligned.32x32b.x32.max.f32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, %32, [%33];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
          "=f"(m)
        : "r"(taddr));
}

// Orders every later use of r and m after the tcgen05.wait::ld that precedes it
// (volatile asm statements keep their order; the "+" operands make the uses depend
// on this one).
__device__ __forceinline__ void tc_regs_ready(uint32_t (&r)[32], float &m) {
    asm volatile(""
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                   "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                   "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                   "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                   "+r"(r[29]), "+r"(r[30]), "+r"(r[31]), "+f"(m));
}

// Bit j = sign bit of r[j]: 32 shifts, then a 5-level tree of multiply-adds (FMA
// pipe) instead of a chain of 32 dependent ORs.
__device__ __forceinline__ uint32_t sign_mask32(const uint32_t (&r)[32]) {
    uint32_t s[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) s[j] = r[j] >> 31;
#pragma unroll
    for (int w = 1; w < 32; w *= 2)
#pragma unroll
        for (int j = 0; j < 32; j += 2 * w) s[j] = s[j + w] * (1u << w) + s[j];
    return s[0];
}

// v truncated to fp16 (toward zero), back in fp32.
__device__ __forceinline__ float f16_rz(float v) { return __half2float(__float2half_rz(v)); }

// fp16 bits of a value that fp16 represents exactly.
__device__ __forceinline__ uint32_t f16_bits(float v) { return (uint32_t)__half_as_ushort(__float2half_rn(v)); }

// v (finite, |v| < 2^14) rounded toward -inf to a normal fp16 value or 0: a
// subnormal result becomes 0 (v > 0) or -2^-14 (v < 0), still <= v, so a tensor
// core that flushes subnormal inputs sees the same operand.
__device__ __forceinline__ float f16_rd_normal(float v) {
    float r = __half2float(__float2half_rd(v));
    if (r != 0.f && fabsf(r) < F16_MIN_NORMAL) r = r > 0.f ? 0.f : -F16_MIN_NORMAL;
    return r;
}

// The scale beta = 2^(6 - e) of the fp16 operands for a codebook whose largest
// norm is f 2^e (f in [0.5, 1)): the scaled norm lands in [32, 64). 1 when that
// norm is zero or not finite; the exponent stays within +-60 so that beta^2 is a
// normal fp32 number.
__device__ __forceinline__ float tc_scale(float craw) {
    if (!(craw > 0.f) || !(craw <= 3.402823466e38f)) return 1.f;
    int e;
    frexpf(craw, &e);
    return ldexpf(1.f, min(60, max(-60, 6 - e)));
}

// The first 29 slots of the K = 32 row layout for one operand (see top of file), as
// fp16-representable values. `a_side` selects the A pattern (x_hi, 1, x_hi, 1,
// x_lo) or the B pattern (c_hi, -h_hi, c_lo, -h_lo, c_hi); v holds the 9 scaled
// values, extra the 10th (1 for A, -h for B). The caller fills slots 29-31.
__device__ __forceinline__ void tc_row(const float (&v)[D], float extra, bool a_side, float (&out)[TC_KD]) {
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const float hi = f16_rz(v[j]), lo = f16_rz(v[j] - hi);
        out[j] = hi;
        out[10 + j] = a_side ? hi : lo;
        out[20 + j] = a_side ? lo : hi;
    }
    const float ehi = f16_rz(extra);
    out[D] = a_side ? 1.f : ehi;
    out[19] = a_side ? 1.f : f16_rz(extra - ehi);
}

// Row `row` of an fp16 operand tile: the 32 slot values, four 16-byte stores.
__device__ __forceinline__ void tc_store_row(unsigned char *tile, int row, const float (&v)[TC_KD]) {
#pragma unroll
    for (int q = 0; q < TC_KD / 8; ++q) {
        uint32_t w[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) w[p] = f16_bits(v[8 * q + 2 * p]) | (f16_bits(v[8 * q + 2 * p + 1]) << 16);
        *reinterpret_cast<uint4 *>(tile + tc_offset(row, 8 * q)) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// Norm of codeword k rounded up, NaN when a value is not finite.
__device__ __forceinline__ float codeword_norm_ru(const float *__restrict__ C, int64_t k) {
    bool ok = true;
    float c2hi = 0.f;
#pragma unroll
    for (int j = 0; j < D; ++j) {
        const float c = C[k * D + j];
        ok &= isfinite(c);
        c2hi = __fadd_ru(c2hi, __fmul_ru(c, c));
    }
    return ok ? __fsqrt_ru(c2hi) : __int_as_float(0x7fc00000);
}

// Maximum of non-negative floats and NaN through their bits (NaN orders above all).
__device__ __forceinline__ float max_bits(float a, float b) {
    return __uint_as_float(max(__float_as_uint(a), __float_as_uint(b)));
}
__device__ __forceinline__ float warp_max_bits(float m) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = __uint_as_float(max(__float_as_uint(m), __shfl_xor_sync(0xffffffffu, __float_as_uint(m), o)));
    return m;
}

// Codeword k into position p of the padded codebook (p < Kpad; p >= K: padding):
// the fp16 operands of beta c, then c in fp32 for the exact path; returns the
// scaled bounds of pack_codebook_kernel (cmax, hmax, qmax; NaN for a non-finite
// codeword, 0 for padding). Padding codewords get c = 0 and -h = -inf, so their g
// is -inf.
__device__ __forceinline__ void pack_codeword_tc(const float *__restrict__ C, int32_t K, int32_t k, int32_t p,
                                                 float beta, float *__restrict__ Cpk, Header *hdr, float &cmax,
                                                 float &hmax, float &qmax) {
    float c[D], c32[D];
    float mh = __int_as_float(0xff800000);  // -h; -inf for padding codewords
#pragma unroll
    for (int j = 0; j < D; ++j) c[j] = c32[j] = 0.f;
    cmax = hmax = qmax = 0.f;
    if (p < K) {
        bool ok = true;
        float s = 0.f, c2lo = 0.f, c2hi = 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            c32[j] = C[(int64_t)k * D + j];
            c[j] = beta * c32[j];  // exact: a power of two, inside the normal range
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
    const int kl = p % TC_N;
    float v[TC_KD];
    tc_row(c, mh, false, v);
    if (!(mh >= -3.402823466e38f)) v[19] = 0.f;  // padding: -inf already sits in the hi slot
    v[TC_SLOT_T0] = kl < TC_HALF ? 1.f : 0.f;
    v[TC_SLOT_R] = 1.f;
    v[TC_SLOT_T1] = kl < TC_HALF ? 0.f : 1.f;
    unsigned char *tile = reinterpret_cast<unsigned char *>(Cpk) + (int64_t)(p / TC_N) * TC_TILE_BYTES;
    tc_store_row(tile, kl, v);
    float *cw = reinterpret_cast<float *>(tile + TC_TILE_H) + kl * D;
#pragma unroll
    for (int j = 0; j < D; ++j) cw[j] = c32[j];
}

__device__ __forceinline__ void publish_bounds_tc(float cmax, float hmax, float qmax, Header *hdr) {
    cmax = warp_max_bits(cmax);
    hmax = warp_max_bits(hmax);
    qmax = warp_max_bits(qmax);
    if ((threadIdx.x & 31) == 0) {
        atomicMax(&hdr->cb_cmax, __float_as_uint(cmax));
        atomicMax(&hdr->cb_hmax, __float_as_uint(hmax));
        atomicMax(&hdr->cb_qmax, __float_as_uint(qmax));
    }
}

// hdr->cb_craw = the codebook's largest norm (rounded up; NaN when a value is not
// finite), from which the operand scale beta is taken.
__global__ void __launch_bounds__(256) codebook_norm_tc_kernel(const float *__restrict__ C, int32_t K, Header *hdr) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    const float m = warp_max_bits(k < K ? codeword_norm_ru(C, k) : 0.f);
    if ((threadIdx.x & 31) == 0) atomicMax(&hdr->cb_craw, __float_as_uint(m));
}

// Packs beta C into tensor-core tiles (Kpad codewords, Kpad a multiple of TC_N) and
// reduces the scaled codebook bounds into hdr->cb_*; beta from hdr->cb_craw.
// cperm (nullable): position p holds codeword cperm[p]. Cprev, tdrift (nullable):
// tdrift[tile] = the largest |C[k] - Cprev[k]| (rounded up; NaN if not finite) over
// the tile's codewords (one CTA of 256 threads per tile).
__global__ void __launch_bounds__(256) pack_codebook_tc_kernel(const float *__restrict__ C, int32_t K, int32_t Kpad,
                                                               float *__restrict__ Cpk, Header *hdr,
                                                               const int32_t *__restrict__ cperm,
                                                               const float *__restrict__ Cprev,
                                                               float *__restrict__ tdrift) {
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    const float beta = tc_scale(__uint_as_float(__ldcg(&hdr->cb_craw)));
    float cmax = 0.f, hmax = 0.f, qmax = 0.f;
    const int32_t k = (cperm != nullptr && p < K) ? cperm[p] : p;
    if (p < Kpad) pack_codeword_tc(C, K, k, p, beta, Cpk, hdr, cmax, hmax, qmax);
    publish_bounds_tc(cmax, hmax, qmax, hdr);
    if (tdrift) {
        __shared__ float s_dr[8];
        float dr = 0.f;
        if (p < K) {
            float s2 = 0.f;
            bool ok = true;
#pragma unroll
            for (int u = 0; u < D; ++u) {
                const float dlt = C[(int64_t)k * D + u] - Cprev[(int64_t)k * D + u];
                ok &= isfinite(dlt);
                s2 = __fadd_ru(s2, __fmul_ru(dlt, dlt));
            }
            // |fl(a - b)| may be below |a - b| by half an ulp: one more ulp per coordinate
            dr = ok ? __fmul_ru(__fsqrt_ru(s2), 1.0000002384185791f) : __int_as_float(0x7fc00000);
        }
        dr = warp_max_bits(dr);
        if ((threadIdx.x & 31) == 0) s_dr[threadIdx.x >> 5] = dr;
        __syncthreads();
        if (threadIdx.x == 0) {
            float m = 0.f;
            for (int w = 0; w < 8; ++w) m = max_bits(m, s_dr[w]);
            tdrift[blockIdx.x] = m;
        }
    }
}

// Both steps in one CTA, for small codebooks (one launch instead of two).
constexpr int32_t TC_PACK_ONE_CTA = 2048;
constexpr int TC_PACK_SMALL_THREADS = 1024;
// The packing of a codebook of at most TC_PACK_ONE_CTA padded codewords by one CTA of
// TC_PACK_SMALL_THREADS threads (the bounds in hdr start from 0).
__device__ __forceinline__ void pack_small_body(const float *__restrict__ C, int32_t K, int32_t Kpad,
                                                float *__restrict__ Cpk, Header *hdr) {
    constexpr int WARPS = TC_PACK_SMALL_THREADS / 32;
    __shared__ float s_m[WARPS];
    float m = 0.f;
    for (int k = threadIdx.x; k < K; k += TC_PACK_SMALL_THREADS) m = max_bits(m, codeword_norm_ru(C, k));
    m = warp_max_bits(m);
    if ((threadIdx.x & 31) == 0) s_m[threadIdx.x >> 5] = m;
    __syncthreads();
    m = s_m[0];
#pragma unroll
    for (int w = 1; w < WARPS; ++w) m = max_bits(m, s_m[w]);
    if (threadIdx.x == 0) hdr->cb_craw = __float_as_uint(m);
    const float beta = tc_scale(m);
    float cmax = 0.f, hmax = 0.f, qmax = 0.f;
    for (int k = threadIdx.x; k < Kpad; k += TC_PACK_SMALL_THREADS) {
        float a, b, c;
        pack_codeword_tc(C, K, k, k, beta, Cpk, hdr, a, b, c);
        cmax = max_bits(cmax, a);
        hmax = max_bits(hmax, b);
        qmax = max_bits(qmax, c);
    }
    publish_bounds_tc(cmax, hmax, qmax, hdr);
}

__global__ void __launch_bounds__(TC_PACK_SMALL_THREADS) pack_codebook_tc_small_kernel(const float *__restrict__ C,
                                                                                       int32_t K, int32_t Kpad,
                                                                                       float *__restrict__ Cpk,
                                                                                       Header *hdr) {
    pack_small_body(C, K, Kpad, Cpk, hdr);
}

// One step of the fit for a small codebook (launch_finalize_pack_small): three
// launches (the objective's sum, the finalise, the packing) in one CTA.
__global__ void __launch_bounds__(TC_PACK_SMALL_THREADS)
finalize_pack_small_kernel(const double *__restrict__ blocksum, int nblocks, double *obj,
                           unsigned long long *__restrict__ acc, int32_t K, int32_t Kpad, Header *hdr,
                           const float *C_prev, float *C_next, int32_t *__restrict__ counts, float *__restrict__ Cpk) {
    __shared__ double wsum[8];
    if (obj) objective_sum_256(blocksum, nblocks, obj, wsum);  // block-uniform
    const int S = __ldcg(&hdr->upd_scale);
    for (int k = threadIdx.x; k < K; k += TC_PACK_SMALL_THREADS) finalize_codeword(acc, k, S, C_prev, C_next, counts, true);
    if (threadIdx.x == 0) {  // the packing's bounds start from 0
        atomicExch(&hdr->cb_cmax, 0u);
        atomicExch(&hdr->cb_hmax, 0u);
        atomicExch(&hdr->cb_qmax, 0u);
    }
    __syncthreads();  // C_next and the cleared bounds, for the whole CTA
    pack_small_body(C_next, K, Kpad, Cpk, hdr);
}

// The fit's finalise for larger codebooks (launch_finalize_norm_tc): finalize_kernel's
// work (one codeword per thread, CTA 0 also the objective) and the new codewords'
// largest norm into hdr->cb_craw (codebook_norm_tc_kernel's work), whose bounds the
// launcher cleared.
__global__ void __launch_bounds__(256)
finalize_norm_tc_kernel(const double *__restrict__ blocksum, int nblocks, double *obj,
                        unsigned long long *__restrict__ acc, int32_t K, Header *hdr, const float *C_prev,
                        float *C_next, int32_t *__restrict__ counts) {
    if (obj && blockIdx.x == 0) {
        __shared__ double wsum[8];
        objective_sum_256(blocksum, nblocks, obj, wsum);
    }
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k < K) finalize_codeword(acc, k, __ldcg(&hdr->upd_scale), C_prev, C_next, counts, true);
    const float m = warp_max_bits(k < K ? codeword_norm_ru(C_next, k) : 0.f);  // this thread's own write
    if ((threadIdx.x & 31) == 0) atomicMax(&hdr->cb_craw, __float_as_uint(m));
}

// Per-row constants of the test: k0 = X2lo - Qmax (rounded down), k1 = |x| Cmax +
// Hmax + |R| (rounded up), k2 = 2 x the absolute part of E (rounded up), and R.
struct RowConst {
    float k0, k1, k2, R;
};

// T' for a running best b (unscaled; beta2 = beta^2): with thr0 = (k0 - beta2 b /
// (1 - gamma_11)) / 2 (rounded down) and dT = thr0 - R (rounded down), T' = dT -
// 2^-15 (k1 + |dT|) - k2 rounded down to a normal fp16 value or 0. Then E(T') <
// thr0 - R - T' (|T'| <= (1 + 2^-10)(|dT| + margin) + 2^-14, and 2^-16 (k1 +
// that) + k2 / 2 stays below the margin since k2 >= 2^-10), so R + T' + E < thr0.
// Returns false (test every codeword) when any of it is not finite or |T'| would
// reach 2^14.
__device__ __forceinline__ bool tc_shift(const RowConst &rc, float b, float beta2, float &tp) {
    const float thr0 = __fmul_rd(__fsub_rd(rc.k0, __fmul_ru(__fmul_ru(b, beta2), INV_ONE_M_G11_TC)), 0.5f);
    const float dT = __fsub_rd(thr0, rc.R);
    const float margin = __fadd_ru(__fmul_ru(TWO_G_TC, __fadd_ru(rc.k1, fabsf(dT))), rc.k2);
    const float pre = __fsub_rd(dT, margin);
    if (!(fabsf(pre) < TC_T_LIMIT)) return false;
    tp = f16_rd_normal(pre);
    return true;
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
    unsigned long long full[TC_STAGES], empty[TC_STAGES], tfull[TC_RT], tempty[TC_RT], done;
    uint32_t tmem_base;
    uint32_t abort_flag;
    float xs[TC_ROWS][D];    // the CTA's kernels and test constants, read on the
    RowConst rc[TC_ROWS];    // rare exact path only (registers go to the tile values)
    float pbest[TC_ROWS];    // second half's result per row, merged at the end
    int32_t pidx[TC_ROWS];
    int32_t prow[TC_ROWS];   // kernel row of each slot (n for a slot without one)
    int32_t lslot[TC_ROWS];  // CTA-local grouping: the CTA row (0..255) slot s works on
    int32_t lhint[TC_ROWS];  // CTA-local grouping: the hint of each CTA row
    uint32_t lcnt[TC_LBINS];
    float rowbest[TC_ROWS];  // each CTA row's distance, for the objective's partial sum in row order
    F2 wsum[TC_EPI_WARPS / 2][TC_RT];  // per-warp partial sums (double-float)
};

// Shared layout of the pruned kernel (assign_tc_pruned_kernel); the per-row bound
// records follow it, TC_ROWS rows of stride + 4 bytes (the 4 put consecutive rows one
// bank apart).
struct __align__(16) TcPrunedShared {
    unsigned char a[TC_RT][TC_A_BYTES];
    unsigned char b[TC_STAGES_YY][TC_TILE_BYTES];
    unsigned long long full[TC_STAGES_YY], empty[TC_STAGES_YY], tfull[TC_RT], tempty[TC_RT], done;
    uint32_t tmem_base;
    uint32_t abort_flag;
    float xs[TC_ROWS][D];
    RowConst rc[TC_ROWS];
    int32_t prow[TC_ROWS];
    uint32_t mask[YY_MAX_TILES / 32];  // tiles this CTA processes
    int32_t nt;                        // their number
    int32_t pad_;
    uint16_t tl[YY_MAX_TILES];         // the tiles, in processing order
    uint32_t dq[YY_MAX_TILES / 4];     // per tile, a byte: its drift since the last pass in bound steps (rounded up)
    uint32_t msk[TC_ROWS][8];          // candidate masks of a row's chunks (rare: only those with candidates)
};

// Byte b of the result: bit b of bits (4 bits -> 4 bytes of 0 or 1).
__device__ __forceinline__ uint32_t bits_to_bytes01(uint32_t bits) { return (bits * 0x00204081u) & 0x01010101u; }
// Bit b of the result: byte b of v, which is 0 or 1 (4 bytes -> 4 bits).
__device__ __forceinline__ uint32_t bytes01_to_bits(uint32_t v) { return (v * 0x01020408u) >> 24; }
// min(255, ceil(x)) for x >= 0 as an integer; 255 for NaN or +inf, 0 for x <= 0.
__device__ __forceinline__ uint32_t ceil_byte(float x) {
    if (!(x < 255.f)) return 255u;
    return x > 0.f ? (uint32_t)ceilf(x) : 0u;
}

constexpr int YY_DELTA_SHIFT = 10;  // bound step: 2^(e - 10) for an initial codebook whose largest norm is f 2^e
constexpr float YY_ONE_M_G11 = 0.99999904632568359375f;  // 1 - 8 * 2^-23 <= 1 - gamma_11 <= 1 / (1 + gamma_11)
constexpr float TWO_M16 = 1.52587890625e-05f;            // 2^-16

// Record byte of a slack x (a lower bound of distance minus a distance reference,
// in units of the bound step: inv = 1 / step): floor(x / step) clamped to [0, 255],
// 0 for a negative or NaN x.
__device__ __forceinline__ uint32_t yy_encode(float x, float inv) {
    const float v = __fmul_rd(x, inv);
    if (!(v >= 1.f)) return 0u;
    return v >= 255.f ? 255u : (uint32_t)v;
}

// Bounds of sqrt(x) from rsqrtf (at most 2 ulp off) with a 2^-16 relative margin:
// below <= sqrt(x) <= above, for any x (0 / +inf outside [2^-100, 2^100]; NaN: 0 / +inf).
__device__ __forceinline__ float sqrt_below(float x) {
    if (!(x >= 7.888609052e-31f)) return 0.f;
    if (!(x <= 1.267650600e30f)) return 1.125899906842624e15f;  // 2^50
    return __fmul_rd(__fmul_rd(x, rsqrtf(x)), 0.9999847412109375f);
}
__device__ __forceinline__ float sqrt_above(float x) {
    if (!(x <= 1.267650600e30f)) return __int_as_float(0x7f800000);
    if (!(x >= 7.888609052e-31f)) return 8.881784197e-16f;  // 2^-50
    return __fmul_ru(__fmul_ru(x, rsqrtf(x)), 1.0000152587890625f);
}

// The part of a half row's lower bound that does not depend on the tile (scaled
// units): X2lo - Qmax - 2 (R + T'max + E), E = 2^-16 (k1 + |T'|max) + k2 / 2; the
// tile's bound is this minus twice the half's largest g (see the epilogue).
// The largest g for which a tile's byte saturates (slack >= 255 steps): with
// X = beta^2 (dref + 255 step)^2 rounded up, g <= (base - X) / 2 rounded down means
// base - 2 g >= X. -inf when any of it is not finite.
__device__ __forceinline__ float yy_saturation(float base, float dref, float step, float beta2) {
    const float dd = __fadd_ru(dref, __fmul_ru(255.f, step));
    const float r = __fmul_rd(__fsub_rd(base, __fmul_ru(beta2, __fmul_ru(dd, dd))), 0.5f);
    return r == r && r <= 3.402823466e38f ? r : __int_as_float(0xff800000);
}

__device__ __forceinline__ float yy_base(const RowConst &rq, float tmax, float tabs) {
    const float E = __fadd_ru(__fmul_ru(TWO_M16, __fadd_ru(rq.k1, tabs)), __fmul_ru(0.5f, rq.k2));
    return __fsub_rd(rq.k0, __fmul_ru(2.f, __fadd_ru(__fadd_ru(rq.R, tmax), E)));  // NaN for rows tested exactly
}

// Named barrier among the 256 epilogue threads (warps 3-10).
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

// The tile holding the hinted codeword of slot row0's row (the pruned kernel reading
// records streams it before the tile list is known); 0 without a usable hint.
__device__ __forceinline__ int yy_first_tile(const int32_t *hint, const int32_t *perm, int64_t row0, int64_t n,
                                             int32_t K, const int32_t *cpos) {
    const int64_t r0 = perm ? (int64_t)__ldg(perm + row0) : row0;
    const int32_t h = (hint != nullptr && (uint64_t)r0 < (uint64_t)n) ? hint[r0] : -1;
    return (uint32_t)h < (uint32_t)K ? __ldg(cpos + h) / TC_N : 0;
}

// TH: the instantiation with the failure-detection test hooks (kq_test_inject_wait_fault);
// the other keeps its wait limits compile-time constants, which its hot loops need.
template <bool TH>
__global__ void __launch_bounds__(TC_THREADS, 1)
assign_tc_kernel(const float *__restrict__ W, int64_t n, const float *__restrict__ C, const float *__restrict__ Cpk,
                 int32_t K, int32_t ntiles, const int32_t *hint, const int32_t *__restrict__ perm, int32_t *idx,
                 float *__restrict__ dist, double *__restrict__ blocksum, Header *hdr) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    TcShared &S = *reinterpret_cast<TcShared *>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile uint32_t *abort_flag = &S.abort_flag;
    uint32_t *status = &hdr->status;
    const float beta = tc_scale(__uint_as_float(__ldcg(&hdr->cb_craw)));  // as pack_codebook_tc_kernel
    const float beta2 = beta * beta;
    // failure-detection tests (kq_test_inject_wait_fault): shorter waits, tile stream cut
    const uint32_t tfault = TH ? __ldcg(&hdr->test_faults) : 0u;
    const uint32_t tlim = TH ? __ldcg(&hdr->test_wait_limit) : 0u;
    const long long wlim = (TH && tlim) ? (long long)tlim : TC_WAIT_LIMIT;

    // ---- barriers first: the producer starts streaming the first codeword tiles
    // while the epilogue threads set up their rows (the other roles wait for the
    // barriers only after the CTA barrier below)
    const int pre = ntiles < TC_STAGES ? ntiles : TC_STAGES;
    if (tid == 0) {
        for (int s = 0; s < TC_STAGES; ++s) {
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.full[s]), 1);
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.empty[s]), TC_EPI_WARPS);
        }
        for (int t = 0; t < TC_RT; ++t) {
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.tfull[t]), 1);
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.tempty[t]), TC_EPI_WARPS);
        }
        mbar_init((uint32_t)__cvta_generic_to_shared(&S.done), TC_RT);
        S.abort_flag = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // initialised barriers -> bulk copies
        for (int i = 0; i < pre; ++i) {
            const uint32_t fb = (uint32_t)__cvta_generic_to_shared(&S.full[i]);
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb), "r"(TC_TILE_BYTES)
                         : "memory");
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    (uint32_t)__cvta_generic_to_shared(S.b[i])),
                "l"(reinterpret_cast<const unsigned char *>(Cpk) + (int64_t)i * TC_TILE_BYTES), "r"(TC_TILE_BYTES),
                "r"(fb)
                : "memory");
        }
    }

    // ---- epilogue threads: one kernel in each row tile, one half of every tile
    const bool epi = warp >= TC_EPI_WARP0;
    const int q = warp & 3;                           // TMEM lane quarter this warp may access
    const int hsel = epi ? (warp - TC_EPI_WARP0) >> 2 : 0;  // codeword half (warps 3-6: first, 7-10: second)
    const int r = q * 32 + lane;                      // row within a row tile
    float best[TC_RT];
    int32_t bi[TC_RT], known[TC_RT];  // known: codeword whose exact distance is best[] (-1: none)
    uint32_t every = 0;               // bit t: half row in row tile t tests every codeword exactly
#pragma unroll
    for (int t = 0; t < TC_RT; ++t) {
        best[t] = __int_as_float(0x7f800000);
        bi[t] = 0;
        known[t] = -1;
    }
    const bool lgroup = hint != nullptr && perm == nullptr && K >= TC_LGROUP_MINK && K <= TC_LGROUP_MAXK;
    if (epi) {
        const int64_t row0 = (int64_t)blockIdx.x * TC_ROWS;
        if (lgroup) {
            // CTA-local grouping (counting sort of the CTA's rows by hint chunk; the
            // order within a chunk is free): a warp's rows then share a few chunks,
            // so the exact path for the hints' own columns is entered a few times
            // per warp instead of in nearly every chunk.
            if (hsel == 1)
                for (int b = r; b < TC_LBINS; b += TC_M) S.lcnt[b] = 0u;
            int32_t hh[TC_RT];
            if (hsel == 0) {
#pragma unroll
                for (int t = 0; t < TC_RT; ++t) {
                    const int64_t rw = row0 + t * TC_M + r;
                    hh[t] = rw < n ? hint[rw] : -1;
                    S.lhint[t * TC_M + r] = hh[t];
                }
            }
            epi_sync();
            uint32_t pos[TC_RT];
            int bin[TC_RT];
            if (hsel == 0) {
#pragma unroll
                for (int t = 0; t < TC_RT; ++t) {
                    bin[t] = (uint32_t)hh[t] < (uint32_t)K ? hh[t] >> 5 : TC_LBINS - 1;
                    pos[t] = atomicAdd(&S.lcnt[bin[t]], 1u);
                }
            }
            epi_sync();
            if (warp == TC_EPI_WARP0) {  // exclusive scan of the bin counts, 5 bins per lane
                uint32_t c[5], tot = 0;
#pragma unroll
                for (int u = 0; u < 5; ++u) {
                    const int b = lane * 5 + u;
                    c[u] = b < TC_LBINS ? S.lcnt[b] : 0u;
                    tot += c[u];
                }
                uint32_t inc = tot;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
                    if (lane >= o) inc += y;
                }
                uint32_t base = inc - tot;
#pragma unroll
                for (int u = 0; u < 5; ++u) {
                    const int b = lane * 5 + u;
                    if (b < TC_LBINS) S.lcnt[b] = base;
                    base += c[u];
                }
            }
            epi_sync();
            if (hsel == 0) {
#pragma unroll
                for (int t = 0; t < TC_RT; ++t) S.lslot[S.lcnt[bin[t]] + pos[t]] = t * TC_M + r;
            }
            epi_sync();
        }
        // Both rows' loads are issued before any of them is used (two dependent
        // rounds to global memory per thread instead of four): the kernels and their
        // hints, then the hinted codewords.
        int64_t row[TC_RT];
        float xw[TC_RT][D], ch[TC_RT][D];
        int32_t hv[TC_RT];
#pragma unroll
        for (int t = 0; t < TC_RT; ++t) {
            // slot -> kernel row (rows in the order of a global or CTA-local grouping, when given)
            const int loc = lgroup ? S.lslot[t * TC_M + r] : t * TC_M + r;
            const int64_t slot = row0 + loc;
            row[t] = slot < n ? (perm ? (int64_t)__ldg(perm + slot) : slot) : n;
        }
#pragma unroll
        for (int t = 0; t < TC_RT; ++t) {
#pragma unroll
            for (int j = 0; j < D; ++j) xw[t][j] = row[t] < n ? W[row[t] * D + j] : 0.f;
            hv[t] = (hint != nullptr && row[t] < n) ? (lgroup ? S.lhint[row[t] - row0] : hint[row[t]]) : -1;
        }
#pragma unroll
        for (int t = 0; t < TC_RT; ++t) {
            const bool hok = (uint32_t)hv[t] < (uint32_t)K;
#pragma unroll
            for (int j = 0; j < D; ++j) ch[t][j] = hok ? C[(int64_t)hv[t] * D + j] : 0.f;
        }
#pragma unroll
        for (int t = 0; t < TC_RT; ++t) {
            const int rloc = t * TC_M + r;
            float x[D], xs[D];  // the kernel, and beta times it (exact unless out of range)
#pragma unroll
            for (int j = 0; j < D; ++j) {
                x[j] = xw[t][j];
                xs[j] = beta * x[j];
            }
            bool ok = true;
#pragma unroll
            for (int j = 0; j < D; ++j) ok &= isfinite(x[j]);
            if (row[t] < n && !ok && hsel == 0) set_flag(status, KQ_FLAG_NONFINITE);
            const float cmax = __uint_as_float(__ldcg(&hdr->cb_cmax));  // scaled bounds
            const float hmax = __uint_as_float(__ldcg(&hdr->cb_hmax));
            const float qmax = __uint_as_float(__ldcg(&hdr->cb_qmax));
            float x2lo = 0.f, x2hi = 0.f;
#pragma unroll
            for (int j = 0; j < D; ++j) {
                x2lo = __fadd_rd(x2lo, __fmul_rd(xs[j], xs[j]));
                x2hi = __fadd_ru(x2hi, __fmul_ru(xs[j], xs[j]));
            }
            const float xn = __fsqrt_ru(x2hi);
            const bool inrange = xn <= TC_X_LIMIT;  // false for non-finite rows too
            RowConst rc;
            rc.R = inrange ? f16_rz(0.5f * x2lo) : 0.f;
            if (rc.R < F16_MIN_NORMAL) rc.R = 0.f;  // a normal fp16 operand or 0
            rc.k0 = inrange ? __fsub_rd(x2lo, qmax) : __int_as_float(0x7fc00000);  // NaN: never shifted
            rc.k1 = __fadd_ru(__fadd_ru(hmax, __fmul_ru(xn, cmax)), fabsf(rc.R));
            rc.k2 = __fmul_ru(TWO_ABS_TC, __fadd_ru(__fadd_ru(cmax, xn), 1.f));
            bool ev = true;
            float tp = 0.f;
            if ((uint32_t)hv[t] < (uint32_t)K) {
                const float d = direct_distance(x, ch[t]);
                if (d < best[t]) {
                    best[t] = d;
                    bi[t] = known[t] = hv[t];
                    ev = !tc_shift(rc, d, beta2, tp);
                }
            }
            every |= (ev ? 1u : 0u) << t;
            if (hsel == 0) {  // both halves start from the same state; one writes it
                S.prow[rloc] = (int32_t)row[t];
#pragma unroll
                for (int j = 0; j < D; ++j) S.xs[rloc][j] = x[j];
                S.rc[rloc] = rc;
                float a[TC_KD], xa[D];
#pragma unroll
                for (int j = 0; j < D; ++j) xa[j] = inrange ? xs[j] : 0.f;
                tc_row(xa, 1.f, true, a);
                a[TC_SLOT_T0] = a[TC_SLOT_T1] = ev ? TC_T_EVERY : -tp;
                a[TC_SLOT_R] = -rc.R;
                tc_store_row(S.a[t], r, a);
            }
        }
    }

    // ---- TMEM
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
        // ---- producer (lane 0)
        if (lane == 0) {
            const int nlast = (TH && (tfault & KQ_TEST_STOP_TILE_STREAM)) ? pre : ntiles;
            for (int i = pre; i < nlast; ++i) {  // tiles 0 .. pre - 1 are on their way
                const int s = i % TC_STAGES;
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.empty[s]), ((i / TC_STAGES) - 1) & 1, abort_flag,
                               status, wlim))
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
    } else if (warp <= TC_RT) {
        // ---- MMA issuer of row tile t = warp - 1 (lane 0)
        const int t = warp - 1;
        if (lane == 0) {
            constexpr uint32_t idesc = tc_idesc(TC_M, TC_N);
            const uint32_t a0 = (uint32_t)__cvta_generic_to_shared(S.a[t]);
            const uint32_t dcol = tmem + (uint32_t)(t * TC_N);
            for (int i = 0; i < ntiles; ++i) {
                const int s = i % TC_STAGES;
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.full[s]), (i / TC_STAGES) & 1, abort_flag, status, wlim))
                    break;
                // the accumulator is free once the epilogue read tile i - 1
                if (i >= 1 &&
                    !mbar_wait((uint32_t)__cvta_generic_to_shared(&S.tempty[t]), (i - 1) & 1, abort_flag, status, wlim))
                    break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t b0 = (uint32_t)__cvta_generic_to_shared(S.b[s]);
#pragma unroll
                for (int kb = 0; kb < TC_KD / 16; ++kb) {
                    const uint64_t ad = tc_smem_desc(a0 + kb * 2 * TC_LBO);
                    const uint64_t bd = tc_smem_desc(b0 + kb * 2 * TC_LBO);  // 16 fp16 of K per MMA
                    asm volatile(
                        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(dcol),
                        "l"(ad), "l"(bd), "r"(idesc), "r"((uint32_t)kb)
                        : "memory");
                }
                // row tile t's values are in TMEM once these MMAs complete (the epilogue
                // warps, which wait for that, also free the shared stage)
                asm volatile(
                    "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                        (uint32_t)__cvta_generic_to_shared(&S.tfull[t]))
                    : "memory");
            }
            // every MMA of both issuers has finished before TMEM can be freed (warp 1
            // frees it)
            const uint32_t db = (uint32_t)__cvta_generic_to_shared(&S.done);
            asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(db)
                         : "memory");
            if (t == 0) {
                for (long long it = 0; it < wlim; ++it) {
                    uint32_t ok;
                    asm volatile(
                        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
                        : "=r"(ok)
                        : "r"(db)
                        : "memory");
                    if (ok) break;
                    if (it + 1 == wlim) set_flag(status, KQ_FLAG_TIMEOUT);
                }
            }
        }
    } else {
        // ---- epilogue: per tile, for each row tile: load this thread's 128 values
        // with their chunk maxima (one wait), hand the accumulator back; a chunk
        // maximum without its sign bit means some codeword of that chunk may improve
        // or tie the running best.
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        bool go = true;
        for (int i = 0; i < ntiles && go; ++i) {
            const int st = i % TC_STAGES;
#pragma unroll
            for (int t = 0; t < TC_RT; ++t) {
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.tfull[t]), i & 1, abort_flag, status, wlim)) {
                    go = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t taddr = tmem + lane_base + (uint32_t)(t * TC_N + hsel * TC_HALF);
                uint32_t v[4][32];
                float cm[4];
#pragma unroll
                for (int c = 0; c < 4; ++c) tc_ld32_max(taddr + 32u * c, v[c], cm[c]);
                asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
                for (int c = 0; c < 4; ++c) tc_regs_ready(v[c], cm[c]);
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0)
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(
                                     (uint32_t)__cvta_generic_to_shared(&S.tempty[t]))
                                 : "memory");
                const bool ev = (every >> t) & 1u;
                const float m = fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3]));
                // Warp-uniform branches (votes) around the rare work: a lane-divergent
                // condition lets the compiler predicate all four chunks' mask builds
                // into every entry.
                if (__any_sync(0xffffffffu, !(__float_as_uint(m) >> 31) || ev)) {  // rare
                    const int rloc = t * TC_M + r;
                    const unsigned char *tile = S.b[st];
                    bool moved = false;
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const bool need = ev || !(__float_as_uint(cm[c]) >> 31);
                        if (!__any_sync(0xffffffffu, need)) continue;  // the whole chunk is ruled out in every lane
                        // candidate mask with static indexing, so v stays in registers;
                        // the running best itself needs no decision (in a warm start it
                        // is almost always the only codeword that passes)
                        uint32_t mask = !need ? 0u : (ev ? 0xffffffffu : ~sign_mask32(v[c]));
                        const int kloc = known[t] - (i * TC_N + hsel * TC_HALF + 32 * c);
                        if ((uint32_t)kloc < 32u) mask &= ~(1u << kloc);
                        while (mask) {
                            const int j = __ffs(mask) - 1;
                            mask &= mask - 1u;
                            const int kl = hsel * TC_HALF + 32 * c + j;
                            const int32_t k = i * TC_N + kl;
                            if (k >= K) break;
                            float xr[D], cw[D];
                            const float *c32 = reinterpret_cast<const float *>(tile + TC_TILE_H) + kl * D;
#pragma unroll
                            for (int u = 0; u < D; ++u) {
                                xr[u] = S.xs[rloc][u];
                                cw[u] = c32[u];
                            }
                            const float d = direct_distance(xr, cw);
                            if (d < best[t] || (d == best[t] && k < bi[t])) {
                                best[t] = d;
                                bi[t] = known[t] = k;
                                moved = true;
                            }
                        }
                    }
                    if (moved) {
                        float tp = 0.f;
                        const bool e2 = !tc_shift(S.rc[rloc], best[t], beta2, tp);
                        every = (every & ~(1u << t)) | ((e2 ? 1u : 0u) << t);
                        *reinterpret_cast<uint16_t *>(&S.a[t][tc_offset(r, hsel ? TC_SLOT_T1 : TC_SLOT_T0)]) =
                            (uint16_t)f16_bits(e2 ? TC_T_EVERY : -tp);
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // for later MMAs
                    }
                }
            }
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"((uint32_t)__cvta_generic_to_shared(&S.empty[st]))
                             : "memory");
        }
        if (hsel == 1) {
#pragma unroll
            for (int t = 0; t < TC_RT; ++t) {
                S.pbest[t * TC_M + r] = best[t];
                S.pidx[t * TC_M + r] = bi[t];
            }
        }
    }

    // ---- teardown (a CTA barrier first: see above); merge the halves (lowest index
    // on equal distances); objective partial sum in a fixed order
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (epi && hsel == 0) {
#pragma unroll
        for (int t = 0; t < TC_RT; ++t) {
            const int rloc = t * TC_M + r;
            const int64_t row = S.prow[rloc];
            const float ob = S.pbest[rloc];
            const int32_t oi = S.pidx[rloc];
            if (ob < best[t] || (ob == best[t] && oi < bi[t])) {
                best[t] = ob;
                bi[t] = oi;
            }
            if (row < n) {
                idx[row] = bi[t];
                if (dist) dist[row] = best[t];
            }
            // the partial sum runs over the CTA's rows in row order whatever the grouping
            S.rowbest[lgroup ? S.lslot[rloc] : rloc] = row < n ? best[t] : 0.f;
        }
        asm volatile("bar.sync 2, 128;" ::: "memory");  // the 128 threads of the first half
#pragma unroll
        for (int t = 0; t < TC_RT; ++t) {
            const F2 sum = f2_warp_sum(S.rowbest[t * TC_M + r]);
            if (lane == 0) S.wsum[warp - TC_EPI_WARP0][t] = sum;
        }
    }
    __syncthreads();
    if (tid == 0) {  // rows 0-31, 32-63, ... of the CTA in turn, as dist_block_sums_kernel
        F2 s{0.f, 0.f};
        for (int t = 0; t < TC_RT; ++t)
            for (int w = 0; w < TC_EPI_WARPS / 2; ++w) s = f2_add(s, S.wsum[w][t]);
        if (blocksum) blocksum[blockIdx.x] = f2_to_double(s);
    }
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TC_COLS) : "memory");
    }
}

// The pruned assignment of the fit (yy: its state). The codebook is packed in the
// order yy.cperm (tile g = positions [256 g, 256 g + 256)); indices and the tie rule
// stay those of the original numbering. Every row keeps a record of one byte per
// tile, q, with q * step + dprev <= its distance to every codeword of the tile, and
// dprev <= its distance to every codeword: written at the end of each pass and, in
// the next pass, lowered by the tile's drift (triangle inequality). A tile whose
// bound proves every codeword farther than the row's hinted codeword, for all 256
// rows of the CTA, is not streamed, multiplied or tested: the answer is the same,
// since no skipped codeword could improve or tie the row's best.
// Roles as in assign_tc_kernel (producer warp 0, MMA issuers warps 1-2, epilogue
// warps 3-10), except that an epilogue thread owns one whole row: warps 3-6 drain
// row tile 0 and warps 7-10 row tile 1, each thread reading all 256 columns of its
// row per tile (two batches of four reducing 32-column loads; the candidate masks
// are taken before the accumulator goes back). A row's best, threshold and bound
// over a tile then live in one thread, and the bound costs one fused multiply-add
// and a byte store per tile.
template <bool TH>  // as assign_tc_kernel
__global__ void __launch_bounds__(TC_THREADS, 1)
assign_tc_pruned_kernel(const float *__restrict__ W, int64_t n, const float *__restrict__ C,
                        const float *__restrict__ Cpk, int32_t K, int32_t ntiles, const int32_t *hint,
                        const int32_t *__restrict__ perm, int32_t *idx, float *__restrict__ dist, Header *hdr,
                        TcYy yy) {
    constexpr int NST = TC_STAGES_YY;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    TcPrunedShared &S = *reinterpret_cast<TcPrunedShared *>(smem_raw);
    unsigned char *yrec = smem_raw + sizeof(TcPrunedShared);
    const int ys = yy.stride + 4;  // record row pitch in shared memory
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile uint32_t *abort_flag = &S.abort_flag;
    uint32_t *status = &hdr->status;
    const float beta = tc_scale(__uint_as_float(__ldcg(&hdr->cb_craw)));  // as pack_codebook_tc_kernel
    const float beta2 = beta * beta;
    const float inv_beta = 1.f / beta;  // exact: a power of two
    const uint32_t tfault = TH ? __ldcg(&hdr->test_faults) : 0u;
    const uint32_t tlim = TH ? __ldcg(&hdr->test_wait_limit) : 0u;
    const long long wlim = (TH && tlim) ? (long long)tlim : TC_WAIT_LIMIT;
    const int64_t row0 = (int64_t)blockIdx.x * TC_ROWS;
    // bound step (fixed for the fit) and whether the records are valid
    float ystep = 0.f, yinv = 0.f;
    {
        const float cn = __uint_as_float(__ldcg(&hdr->yy_cnorm));
        if (cn > 0.f && cn <= 3.402823466e38f) {
            int e;
            frexpf(cn, &e);
            const int ex = max(-100, min(100, e - YY_DELTA_SHIFT));
            ystep = ldexpf(1.f, ex);
            yinv = ldexpf(1.f, -ex);
        }
    }
    const bool yread = yy.read != 0 && ystep > 0.f;

    // ---- barriers first; the first tiles stream while the rows are set up: a run of
    // NST consecutive tiles starting at (or just before) the one that holds the first
    // slot's hinted codeword (the kd order puts neighbouring tiles close together);
    // they are processed whatever the records say
    const int pre = ntiles < NST ? ntiles : NST;
    if (tid == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.full[s]), 1);
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.empty[s]), TC_EPI_WARPS);
        }
        for (int t = 0; t < TC_RT; ++t) {
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.tfull[t]), 1);
            mbar_init((uint32_t)__cvta_generic_to_shared(&S.tempty[t]), TC_EPI_WARPS / TC_RT);
        }
        mbar_init((uint32_t)__cvta_generic_to_shared(&S.done), TC_RT);
        S.abort_flag = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // initialised barriers -> bulk copies
        const int g0 = yread ? yy_first_tile(hint, perm, row0, n, K, yy.cpos) : 0;
        const int e0 = min(g0, ntiles - pre);
        for (int i = 0; i < pre; ++i) {
            const int g = e0 + i;
            const uint32_t fb = (uint32_t)__cvta_generic_to_shared(&S.full[i]);
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb), "r"(TC_TILE_BYTES)
                         : "memory");
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    (uint32_t)__cvta_generic_to_shared(S.b[i])),
                "l"(reinterpret_cast<const unsigned char *>(Cpk) + (int64_t)g * TC_TILE_BYTES), "r"(TC_TILE_BYTES),
                "r"(fb)
                : "memory");
        }
    }

    // ---- epilogue threads: one row each
    const bool epi = warp >= TC_EPI_WARP0;
    const int q = warp & 3;                                    // TMEM lane quarter this warp may access
    const int t = epi ? (warp - TC_EPI_WARP0) >> 2 : 0;       // its row tile
    const int r = q * 32 + lane;                               // row within the row tile
    const int sl = t * TC_M + r;                               // the row's CTA slot
    float best = __int_as_float(0x7f800000);
    int32_t bi = 0, known = -1;  // known: codebook position of the codeword whose distance is best (-1: none)
    bool ev = true;              // the row tests every codeword exactly
    float tmaxv = -TC_T_EVERY, tabsv = TC_T_EVERY;  // largest T' and |T'| any MMA may have read
    float ybase = __int_as_float(0x7fc00000), ydref = __int_as_float(0x7f800000);
    float ysat = __int_as_float(0xff800000);  // yy_saturation of the row
    float dpo = 0.f;  // the record's distance from the last pass
    int64_t row = n;
    if (epi) {
        {
            const int et = tid - TC_EPI_WARP0 * 32;
            if (et < YY_MAX_TILES / 32) S.mask[et] = 0u;
            if (et < YY_MAX_TILES / 4) {  // 4 tiles per word; tiles past the codebook never skip
                uint32_t wd = 0u;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int g = 4 * et + u;
                    const uint32_t b = (g < ntiles && yread) ? ceil_byte(__fmul_ru(__ldg(yy.tdrift + g), yinv)) : 255u;
                    wd |= b << (8 * u);
                }
                S.dq[et] = wd;
            }
        }
        const int64_t slot = row0 + sl;
        row = slot < n ? (int64_t)__ldg(perm + slot) : n;
        float x[D], ch[D];
        const int32_t hv = (hint != nullptr && row < n) ? hint[row] : -1;
        const bool hok = (uint32_t)hv < (uint32_t)K;
#pragma unroll
        for (int j = 0; j < D; ++j) x[j] = row < n ? W[row * D + j] : 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) ch[j] = hok ? C[(int64_t)hv * D + j] : 0.f;
        float xs[D];
#pragma unroll
        for (int j = 0; j < D; ++j) xs[j] = beta * x[j];
        bool ok = true;
#pragma unroll
        for (int j = 0; j < D; ++j) ok &= isfinite(x[j]);
        if (row < n && !ok) set_flag(status, KQ_FLAG_NONFINITE);
        const float cmax = __uint_as_float(__ldcg(&hdr->cb_cmax));  // scaled bounds
        const float hmax = __uint_as_float(__ldcg(&hdr->cb_hmax));
        const float qmax = __uint_as_float(__ldcg(&hdr->cb_qmax));
        float x2lo = 0.f, x2hi = 0.f;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            x2lo = __fadd_rd(x2lo, __fmul_rd(xs[j], xs[j]));
            x2hi = __fadd_ru(x2hi, __fmul_ru(xs[j], xs[j]));
        }
        const float xn = __fsqrt_ru(x2hi);
        const bool inrange = xn <= TC_X_LIMIT;  // false for non-finite rows too
        RowConst rc;
        rc.R = inrange ? f16_rz(0.5f * x2lo) : 0.f;
        if (rc.R < F16_MIN_NORMAL) rc.R = 0.f;
        rc.k0 = inrange ? __fsub_rd(x2lo, qmax) : __int_as_float(0x7fc00000);  // NaN: never shifted
        rc.k1 = __fadd_ru(__fadd_ru(hmax, __fmul_ru(xn, cmax)), fabsf(rc.R));
        rc.k2 = __fmul_ru(TWO_ABS_TC, __fadd_ru(__fadd_ru(cmax, xn), 1.f));
        float tp = 0.f;
        if (hok) {
            const float d = direct_distance(x, ch);
            if (d < best) {
                best = d;
                bi = hv;
                known = __ldg(yy.cpos + hv);
                ev = !tc_shift(rc, d, beta2, tp);
            }
        }
        S.prow[sl] = (int32_t)row;
#pragma unroll
        for (int j = 0; j < D; ++j) S.xs[sl][j] = x[j];
        S.rc[sl] = rc;
        {
            float a[TC_KD], xa[D];
#pragma unroll
            for (int j = 0; j < D; ++j) xa[j] = inrange ? xs[j] : 0.f;
            tc_row(xa, 1.f, true, a);
            a[TC_SLOT_T0] = a[TC_SLOT_T1] = ev ? TC_T_EVERY : -tp;
            a[TC_SLOT_R] = -rc.R;
            tc_store_row(S.a[t], r, a);
        }
        tmaxv = ev ? -TC_T_EVERY : tp;
        tabsv = ev ? TC_T_EVERY : fabsf(tp);
        ybase = yy_base(rc, tmaxv, tabsv);
        ydref = sqrt_above(__fmul_ru(best, INV_ONE_M_G11_TC));
        ysat = yy_saturation(ybase, ydref, ystep, beta2);

        // The tiles this CTA needs: tile g can be skipped for this row when its record's
        // bound, lowered by the tile's drift, proves every codeword of g farther than
        // the hinted codeword's distance (the row's best so far).
        epi_sync();  // mask cleared, drifts staged
        const bool all = !yread || !(best <= 3.402823466e38f);  // no valid record or no finite hint distance
        dpo = (yread && row < n) ? yy.dprev[row] : 0.f;
        const uint4 *src = reinterpret_cast<const uint4 *>(yy.rec + (row < n ? row : 0) * (int64_t)yy.stride);
        uint32_t *dst = reinterpret_cast<uint32_t *>(yrec + sl * ys);
        // the whole record in flight at once (one round trip to memory, not eight)
        uint4 rv[YY_MAX_TILES / 16];
#pragma unroll
        for (int c = 0; c < YY_MAX_TILES / 16; ++c)
            rv[c] = (row < n && !all && c * 16 < yy.stride) ? src[c] : make_uint4(0u, 0u, 0u, 0u);
        // Tile g is skipped for this row when q_g step + dprev - drift_g > S, S >= the
        // distance whose square times (1 - gamma_11) is the hint's distance (then every
        // codeword of g is farther, in the direct form, than the hinted one): in whole
        // steps, when q_g > base + dq_g (4 tiles per instruction, saturating at 255).
        const float Sr = sqrt_above(__fmul_ru(best, INV_ONE_M_G11_TC));
        const uint32_t base4 = ceil_byte(__fmul_ru(__fsub_ru(Sr, dpo), yinv)) * 0x01010101u;
#pragma unroll
        for (int w = 0; w < YY_MAX_TILES / 32; ++w) {
            if (32 * w >= ntiles) break;
            uint32_t need = 0u;
            if (row < n) {
                if (all) {
                    need = 0xffffffffu;
                } else {
#pragma unroll
                    for (int h2 = 0; h2 < 2; ++h2) {
                        const int c = 2 * w + h2;
                        if (c * 16 >= yy.stride) continue;  // a stride of 16 (mod 32) bytes
                        const uint4 v = rv[c];
                        dst[4 * c] = v.x;
                        dst[4 * c + 1] = v.y;
                        dst[4 * c + 2] = v.z;
                        dst[4 * c + 3] = v.w;
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint32_t qw = k == 0 ? v.x : k == 1 ? v.y : k == 2 ? v.z : v.w;
                            const uint32_t thr = __vaddus4(base4, S.dq[4 * c + k]);
                            const uint32_t skip = bytes01_to_bits(__vcmpgtu4(qw, thr) & 0x01010101u);
                            need |= ((~skip) & 0xfu) << (16 * h2 + 4 * k);
                        }
                    }
                }
                const int left = ntiles - 32 * w;
                if (left < 32) need &= (1u << left) - 1u;
            }
            need = __reduce_or_sync(0xffffffffu, need);
            if (lane == 0 && need) atomicOr(&S.mask[w], need);
        }
        epi_sync();
        if (warp == TC_EPI_WARP0) {
            // the list: the early tile first (records read), then the others in order;
            // lane l takes tiles 8 l .. 8 l + 7
            const int g0 = yread ? yy_first_tile(hint, perm, row0, n, K, yy.cpos) : 0;  // as streamed
            const int e0 = min(g0, ntiles - pre);
            uint32_t bits = (S.mask[lane >> 2] >> ((lane & 3) * 8)) & 0xffu;
#pragma unroll
            for (int b = 0; b < 8; ++b)  // the early run goes first
                if ((uint32_t)(lane * 8 + b - e0) < (uint32_t)pre) bits &= ~(1u << b);
            const int cnt = __popc(bits);
            int incl = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y2 = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y2;
            }
            int pos = pre + incl - cnt;
            while (bits) {
                const int b = __ffs(bits) - 1;
                bits &= bits - 1u;
                S.tl[pos++] = (uint16_t)(lane * 8 + b);
            }
            if (lane == 31) S.nt = pre + incl;
            if (lane < pre) {
                const int g = e0 + lane;
                S.tl[lane] = (uint16_t)g;
                atomicOr(&S.mask[g >> 5], 1u << (g & 31));  // the mask now marks every processed tile
            }
        }
    }

    // ---- TMEM
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
    const int nt = S.nt;

    if (warp == 0) {
        // ---- producer (lane 0)
        if (lane == 0) {
            const int nlast = (TH && (tfault & KQ_TEST_STOP_TILE_STREAM)) ? pre : nt;
            for (int i = pre; i < nlast; ++i) {  // list entries 0 .. pre - 1 are on their way
                const int s = i % NST;
                const int g = S.tl[i];
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.empty[s]), ((i / NST) - 1) & 1, abort_flag,
                               status, wlim))
                    break;
                const uint32_t fb = (uint32_t)__cvta_generic_to_shared(&S.full[s]);
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb), "r"(TC_TILE_BYTES)
                             : "memory");
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                        (uint32_t)__cvta_generic_to_shared(S.b[s])),
                    "l"(reinterpret_cast<const unsigned char *>(Cpk) + (int64_t)g * TC_TILE_BYTES), "r"(TC_TILE_BYTES),
                    "r"(fb)
                    : "memory");
            }
        }
    } else if (warp <= TC_RT) {
        // ---- MMA issuer of row tile warp - 1 (lane 0)
        const int ti = warp - 1;
        if (lane == 0) {
            constexpr uint32_t idesc = tc_idesc(TC_M, TC_N);
            const uint32_t a0 = (uint32_t)__cvta_generic_to_shared(S.a[ti]);
            const uint32_t dcol = tmem + (uint32_t)(ti * TC_N);
            for (int i = 0; i < nt; ++i) {
                const int s = i % NST;
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.full[s]), (i / NST) & 1, abort_flag, status, wlim))
                    break;
                // the accumulator is free once its row tile's epilogue warps read tile i - 1
                if (i >= 1 &&
                    !mbar_wait((uint32_t)__cvta_generic_to_shared(&S.tempty[ti]), (i - 1) & 1, abort_flag, status, wlim))
                    break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t b0 = (uint32_t)__cvta_generic_to_shared(S.b[s]);
#pragma unroll
                for (int kb = 0; kb < TC_KD / 16; ++kb) {
                    const uint64_t ad = tc_smem_desc(a0 + kb * 2 * TC_LBO);
                    const uint64_t bd = tc_smem_desc(b0 + kb * 2 * TC_LBO);
                    asm volatile(
                        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(dcol),
                        "l"(ad), "l"(bd), "r"(idesc), "r"((uint32_t)kb)
                        : "memory");
                }
                asm volatile(
                    "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                        (uint32_t)__cvta_generic_to_shared(&S.tfull[ti]))
                    : "memory");
            }
            const uint32_t db = (uint32_t)__cvta_generic_to_shared(&S.done);
            asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(db)
                         : "memory");
            if (ti == 0) {
                for (long long it = 0; it < wlim; ++it) {
                    uint32_t okd;
                    asm volatile(
                        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
                        : "=r"(okd)
                        : "r"(db)
                        : "memory");
                    if (okd) break;
                    if (it + 1 == wlim) set_flag(status, KQ_FLAG_TIMEOUT);
                }
            }
        }
    } else {
        // ---- epilogue: per tile, load the row's 256 values in two batches with their
        // chunk maxima, take the candidate masks of the chunks that may hold a codeword
        // improving or tying the best, hand the accumulator back, then test the
        // candidates exactly and record the row's bound for the tile
        const uint32_t taddr0 = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(t * TC_N);
        bool go = true;
        for (int i = 0; i < nt && go; ++i) {
            const int st = i % NST;
            const int gb = (int)S.tl[i] * TC_N;  // codebook position of the tile's first codeword
            if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&S.tfull[t]), i & 1, abort_flag, status, wlim)) {
                go = false;
                break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            uint32_t v[4][32];
            float cm[4];
            float m = __int_as_float(0xff800000);  // the row's largest g over the tile
            uint32_t anym = 0u;                     // bit c: chunk c has candidates (masks in S.msk)
#pragma unroll
            for (int hb = 0; hb < 2; ++hb) {  // columns 128 hb .. 128 hb + 127
#pragma unroll
                for (int c = 0; c < 4; ++c) tc_ld32_max(taddr0 + (uint32_t)(128 * hb + 32 * c), v[c], cm[c]);
                asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
                for (int c = 0; c < 4; ++c) tc_regs_ready(v[c], cm[c]);
                const float mb = fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3]));
                m = fmaxf(m, mb);
                // one warp vote on the way to the hand-back; the masks only in the rare case
                if (__any_sync(0xffffffffu, !(__float_as_uint(mb) >> 31) || ev)) {
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const bool need = ev || !(__float_as_uint(cm[c]) >> 31);
                        if (__any_sync(0xffffffffu, need) && need) {
                            S.msk[sl][4 * hb + c] = ev ? 0xffffffffu : ~sign_mask32(v[c]);
                            anym |= 1u << (4 * hb + c);
                        }
                    }
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(
                                 (uint32_t)__cvta_generic_to_shared(&S.tempty[t]))
                             : "memory");
            if (__any_sync(0xffffffffu, anym != 0u)) {  // rare: candidates
                const unsigned char *tile = S.b[st];
                bool moved = false;
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    uint32_t mask = ((anym >> c) & 1u) ? S.msk[sl][c] : 0u;
                    const int kloc = known - (gb + 32 * c);
                    if ((uint32_t)kloc < 32u) mask &= ~(1u << kloc);  // the best itself needs no test
                    while (mask) {
                        const int j = __ffs(mask) - 1;
                        mask &= mask - 1u;
                        const int kl = 32 * c + j;
                        const int32_t p = gb + kl;
                        if (p >= K) break;
                        float xr[D], cw[D];
                        const float *c32 = reinterpret_cast<const float *>(tile + TC_TILE_H) + kl * D;
#pragma unroll
                        for (int u = 0; u < D; ++u) {
                            xr[u] = S.xs[sl][u];
                            cw[u] = c32[u];
                        }
                        const float d = direct_distance(xr, cw);
                        if (d <= best) {
                            // the lowest original index wins a tie, whatever the packing order
                            const int32_t k = __ldg(yy.cperm + p);
                            if (d < best || k < bi) {
                                best = d;
                                bi = k;
                                known = p;
                                moved = true;
                            }
                        }
                    }
                }
                if (moved) {
                    float tp = 0.f;
                    const bool e2 = !tc_shift(S.rc[sl], best, beta2, tp);
                    ev = e2;
                    const uint16_t tb = (uint16_t)f16_bits(e2 ? TC_T_EVERY : -tp);
                    *reinterpret_cast<uint16_t *>(&S.a[t][tc_offset(r, TC_SLOT_T0)]) = tb;
                    *reinterpret_cast<uint16_t *>(&S.a[t][tc_offset(r, TC_SLOT_T1)]) = tb;
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // for later MMAs
                    const float tn = e2 ? -TC_T_EVERY : tp;
                    tmaxv = fmaxf(tmaxv, tn);
                    tabsv = fmaxf(tabsv, fabsf(tn));
                    ybase = yy_base(S.rc[sl], tmaxv, tabsv);
                    ydref = sqrt_above(__fmul_ru(best, INV_ONE_M_G11_TC));
                    ysat = yy_saturation(ybase, ydref, ystep, beta2);
                }
            }
            // the row's bound for this tile (D >= X2lo - Qmax - 2 e, e <= g + R + T' + E,
            // g <= m, scaled units), recorded as slack over its current best
            uint32_t qb = 255u;  // far tiles saturate: no square root
            if (!(m <= ysat)) {
                const float lb = __fmul_rd(sqrt_below(__fmaf_rd(-2.f, m, ybase)), inv_beta);
                qb = yy_encode(__fsub_rd(lb, ydref), yinv);
            }
            yrec[sl * ys + gb / TC_N] = (unsigned char)qb;
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"((uint32_t)__cvta_generic_to_shared(&S.empty[st]))
                             : "memory");
        }
    }

    // ---- teardown (a CTA barrier first)
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TC_COLS) : "memory");
    }
    if (tid == 0) {  // the work done against the work of an unpruned pass (kq_fit_prune_stats)
        atomicAdd(&hdr->yy_tiles_run, (unsigned long long)nt);
        atomicAdd(&hdr->yy_tiles_all, (unsigned long long)ntiles);
    }
    if (epi && row < n) {
        idx[row] = bi;
        if (dist) dist[row] = best;
        // the record for the next pass, relative to this pass's final best: processed
        // tiles keep this pass's byte (slack over a best at least the final one), the
        // others last pass's bound lowered by the tile's drift; after a wait gave up,
        // no bound (zeros)
        const bool fin = *abort_flag == 0u && best <= 3.402823466e38f;
        const float dpn = fin ? __fsqrt_rd(__fmul_rd(best, YY_ONE_M_G11)) : 0.f;  // <= the distance to any codeword
        const float dref = fin ? __fsqrt_ru(__fmul_ru(best, INV_ONE_M_G11_TC)) : __int_as_float(0x7f800000);
        const uint32_t *rs = reinterpret_cast<const uint32_t *>(yrec + sl * ys);
        uint4 *dstg = reinterpret_cast<uint4 *>(yy.rec + row * (int64_t)yy.stride);
        // unprocessed tiles: q - dq_g - cr (saturating), cr = the change of reference in
        // steps, rounded up: (q - dq - cr) step + dref <= q step + dprev - drift <= the
        // distance to the tile, and the next pass decodes with dpn <= dref
        const uint32_t cr4 = (fin ? ceil_byte(__fmul_ru(__fsub_ru(dref, dpo), yinv)) : 255u) * 0x01010101u;
        for (int c = 0; c < yy.stride / 16; ++c) {
            uint32_t wv[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int g0 = 16 * c + 4 * k;  // first of the word's 4 tiles
                const uint32_t qw = rs[4 * c + k];
                const uint32_t proc = bits_to_bytes01((S.mask[g0 >> 5] >> (g0 & 31)) & 0xfu) * 0xffu;
                const uint32_t adj = __vsubus4(qw, __vaddus4(S.dq[4 * c + k], cr4));
                wv[k] = fin ? ((qw & proc) | (adj & ~proc)) : 0u;
            }
            dstg[c] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
        }
        yy.dprev[row] = dpn;
    }
}

int32_t tc_kpad(int32_t K) { return (K + TC_N - 1) / TC_N * TC_N; }

bool tc_pack_small(int32_t K) { return tc_kpad(K) <= TC_PACK_ONE_CTA; }

cudaError_t launch_finalize_pack_small(const double *blocksum, int nblocks, double *obj, unsigned long long *acc,
                                       int32_t K, Header *hdr, const float *C_prev, float *C_next, int32_t *counts,
                                       float *Cpk, cudaStream_t s) {
    const int32_t Kpad = tc_kpad(K);
    if (Kpad > TC_PACK_ONE_CTA) return cudaErrorInvalidValue;
    launch_begin(s);
    finalize_pack_small_kernel<<<1, TC_PACK_SMALL_THREADS, 0, s>>>(blocksum, nblocks, obj, acc, K, Kpad, hdr, C_prev,
                                                                  C_next, counts, Cpk);
    launch_end(s, "finalize_pack_small_kernel");
    return cudaGetLastError();
}


// Which assignment kernel is faster, from measured costs on GB300: this kernel runs
// ceil(n / 256) CTAs, one per SM at a time, each ~12K cycles of setup and teardown
// plus ~1000 cycles per 256-codeword tile; the split-K CUDA-core kernel takes at
// least ~50 us at these sizes (e.g. 56 us for n = 4096, K = 1024) and ~1.4e12
// pairs/s beyond.
bool tc_eligible(int64_t n, int32_t K, int num_sms) {
    const double blocks = (double)((n + TC_ROWS - 1) / TC_ROWS);
    const double waves = (double)(int64_t)((blocks + num_sms - 1) / num_sms);
    const double tc_us = waves * (12000.0 + 1000.0 * ((K + TC_N - 1) / TC_N)) / 2070.0;
    const double cc_us = fmax(50.0, (double)n * K / 1.4e6);
    return n >= (int64_t)TC_ROWS * num_sms || tc_us < cc_us;
}

cudaError_t launch_finalize_norm_tc(const double *blocksum, int nblocks, double *obj, unsigned long long *acc,
                                    int32_t K, Header *hdr, const float *C_prev, float *C_next, int32_t *counts,
                                    cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(&hdr->cb_cmax, 0, 4 * sizeof(uint32_t), s);  // cb_cmax .. cb_craw
    if (e != cudaSuccess) return e;
    launch_begin(s);
    finalize_norm_tc_kernel<<<(K + 255) / 256, 256, 0, s>>>(blocksum, nblocks, obj, acc, K, hdr, C_prev, C_next,
                                                            counts);
    launch_end(s, "finalize_norm_tc_kernel");
    return cudaGetLastError();
}

cudaError_t launch_pack_codebook_tc(const float *C, int32_t K, float *Cpk, Header *hdr, cudaStream_t s,
                                    const int32_t *cperm, const float *Cprev, float *tdrift, bool normed) {
    cudaError_t e;
    const int32_t Kpad = tc_kpad(K);
    if (normed && Kpad > TC_PACK_ONE_CTA) {  // bounds cleared, largest norm in place
        launch_begin(s);
        pack_codebook_tc_kernel<<<(Kpad + 255) / 256, 256, 0, s>>>(C, K, Kpad, Cpk, hdr, cperm,
                                                                    tdrift ? Cprev : nullptr, Cprev ? tdrift : nullptr);
        launch_end(s, "pack_codebook_tc_kernel");
        return cudaGetLastError();
    }
    e = cudaMemsetAsync(&hdr->cb_cmax, 0, 4 * sizeof(uint32_t), s);  // cb_cmax .. cb_craw
    if (e != cudaSuccess) return e;
    if (Kpad <= TC_PACK_ONE_CTA && !cperm && !tdrift) {
        launch_begin(s);
        pack_codebook_tc_small_kernel<<<1, TC_PACK_SMALL_THREADS, 0, s>>>(C, K, Kpad, Cpk, hdr);
        launch_end(s, "pack_codebook_tc_small_kernel");
        return cudaGetLastError();
    }
    launch_begin(s);
    codebook_norm_tc_kernel<<<(K + 255) / 256, 256, 0, s>>>(C, K, hdr);
    launch_end(s, "codebook_norm_tc_kernel");
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    launch_begin(s);
    pack_codebook_tc_kernel<<<(Kpad + 255) / 256, 256, 0, s>>>(C, K, Kpad, Cpk, hdr, cperm, tdrift ? Cprev : nullptr,
                                                                Cprev ? tdrift : nullptr);
    launch_end(s, "pack_codebook_tc_kernel");
    return cudaGetLastError();
}

// ---- Warm starts: rows in the order of their hinted codeword. A warp's rows then
// share one hint, so the exact path that every row takes once (in the tile of its
// own running best, whose column the test cannot rule out) is entered once per warp
// instead of once per distinct hint. Results do not depend on the order.

// The group of hint h: cpos[h] (the codebook position) or h; K without a usable hint.
__device__ __forceinline__ int32_t hint_key(int32_t h, int32_t K, const int32_t *__restrict__ cpos) {
    if ((uint32_t)h >= (uint32_t)K) return K;
    return cpos ? __ldg(cpos + h) : h;
}

// cnt[key] = rows whose hint has that group key (see hint_key).
__global__ void __launch_bounds__(256) hint_histogram_kernel(const int32_t *__restrict__ hint, int64_t n, int32_t K,
                                                             const int32_t *__restrict__ cpos, int32_t *cnt) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        atomicAdd(cnt + hint_key(__ldcs(hint + i), K, cpos), 1);
}

// cursor[0..m) = exclusive prefix sum of cnt[0..m) (one CTA), where entries past
// mc read as 0 (so a K-entry count array can stand for K + 1 entries). Rounds of
// 4096 entries: coalesced 16-byte loads, a scan over the CTA, 16-byte stores, the
// round's total carried into the next. cursor may be cnt itself: each round reads
// all its entries before any are written.
constexpr int SCAN_THREADS = 1024;
// map (nullable): entry k reads cnt[map[k]] (counts per codeword scanned in
// codebook-position order).
__global__ void __launch_bounds__(SCAN_THREADS) scan_counts_kernel(const int32_t *cnt, int32_t mc, int32_t m,
                                                                   int32_t *cursor, const int32_t *__restrict__ map) {
    __shared__ int32_t wsum[SCAN_THREADS / 32];
    __shared__ int32_t s_carry;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) s_carry = 0;
    __syncthreads();
    for (int32_t base = 0; base < m; base += 4 * SCAN_THREADS) {
        const int32_t k0 = base + 4 * tid;
        int32_t c[4];
        if (!map && k0 + 3 < mc && ((reinterpret_cast<uintptr_t>(cnt + k0) & 15) == 0)) {
            const int4 v = *reinterpret_cast<const int4 *>(cnt + k0);
            c[0] = v.x; c[1] = v.y; c[2] = v.z; c[3] = v.w;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) c[u] = k0 + u < mc ? cnt[map ? map[k0 + u] : k0 + u] : 0;
        }
        const int32_t local = c[0] + c[1] + c[2] + c[3];
        int32_t incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int32_t w = wsum[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += y;
            }
            wsum[lane] = w;  // inclusive over the warps
        }
        __syncthreads();
        const int32_t carry = s_carry;
        int32_t run = carry + incl - local + (warp > 0 ? wsum[warp - 1] : 0);
        int32_t out[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            out[u] = run;
            run += c[u];
        }
        if (k0 + 3 < m && ((reinterpret_cast<uintptr_t>(cursor + k0) & 15) == 0)) {
            *reinterpret_cast<int4 *>(cursor + k0) = make_int4(out[0], out[1], out[2], out[3]);
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (k0 + u < m) cursor[k0 + u] = out[u];
        }
        __syncthreads();  // every thread has read s_carry and wsum
        if (tid == SCAN_THREADS - 1) s_carry = run;
        __syncthreads();
    }
}

// perm = the rows grouped by hint key (any order within a group).
// Four rows per thread step, so that four returning atomics are in flight at once.
constexpr int SCATTER_UNROLL = 4;
__global__ void __launch_bounds__(256) hint_scatter_kernel(const int32_t *__restrict__ hint, int64_t n, int32_t K,
                                                           const int32_t *__restrict__ cpos, int32_t *cursor,
                                                           int32_t *__restrict__ perm) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i0 < n; i0 += SCATTER_UNROLL * stride) {
        int32_t key[SCATTER_UNROLL], pos[SCATTER_UNROLL];
#pragma unroll
        for (int u = 0; u < SCATTER_UNROLL; ++u) {
            const int64_t i = i0 + u * stride;
            key[u] = i < n ? hint_key(__ldcs(hint + i), K, cpos) : -1;
        }
#pragma unroll
        for (int u = 0; u < SCATTER_UNROLL; ++u) pos[u] = key[u] >= 0 ? atomicAdd(cursor + key[u], 1) : -1;
#pragma unroll
        for (int u = 0; u < SCATTER_UNROLL; ++u)  // counts that do not match the hints: no stray write
            if ((uint32_t)pos[u] < (uint32_t)n) perm[pos[u]] = (int32_t)(i0 + u * stride);
    }
}

// blocksum[b] = sum of dist over rows [256 b, 256 b + 256) in a fixed order (double-float).
__global__ void __launch_bounds__(256) dist_block_sums_kernel(const float *__restrict__ dist, int64_t n,
                                                              double *__restrict__ blocksum) {
    __shared__ F2 ws[8];
    const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
    const F2 v = f2_warp_sum(i < n ? __ldcs(dist + i) : 0.f);
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        F2 t{0.f, 0.f};
        for (int w = 0; w < 8; ++w) t = f2_add(t, ws[w]);
        blocksum[blockIdx.x] = f2_to_double(t);
    }
}

// The same histogram and scatter for at most HINT_SMEM_BINS keys (e.g. the k-d
// leaves, 256 of them at 65,536 codewords, where millions of rows land on few keys
// and one global atomic per row contends on a handful of addresses): each CTA takes
// a contiguous run of rows, counts them per key in shared memory, and touches the
// global array once per key it holds. The scatter counts its run first, reserves
// one range per key with a single returning atomic, then places each row at that
// range's base plus its rank among the run's rows of the key (the order within a
// key is free).
constexpr int HINT_SMEM_BINS = 4096;
constexpr int HINT_SMEM_THREADS = 512;

__device__ __forceinline__ void hint_run(int64_t n, int64_t &r0, int64_t &r1) {
    const int64_t per = (n + gridDim.x - 1) / gridDim.x;
    r0 = min(n, (int64_t)blockIdx.x * per);
    r1 = min(n, r0 + per);
}

__global__ void __launch_bounds__(HINT_SMEM_THREADS) hint_histogram_smem_kernel(const int32_t *__restrict__ hint,
                                                                                int64_t n, int32_t K,
                                                                                const int32_t *__restrict__ cpos,
                                                                                int32_t *cnt) {
    __shared__ int32_t c[HINT_SMEM_BINS];
    const int m = K + 1;
    for (int b = threadIdx.x; b < m; b += HINT_SMEM_THREADS) c[b] = 0;
    __syncthreads();
    int64_t r0, r1;
    hint_run(n, r0, r1);
    for (int64_t i = r0 + threadIdx.x; i < r1; i += HINT_SMEM_THREADS) atomicAdd(&c[hint_key(__ldcs(hint + i), K, cpos)], 1);
    __syncthreads();
    for (int b = threadIdx.x; b < m; b += HINT_SMEM_THREADS)
        if (c[b]) atomicAdd(cnt + b, c[b]);
}

__global__ void __launch_bounds__(HINT_SMEM_THREADS) hint_scatter_smem_kernel(const int32_t *__restrict__ hint,
                                                                              int64_t n, int32_t K,
                                                                              const int32_t *__restrict__ cpos,
                                                                              int32_t *cursor, int32_t *__restrict__ perm) {
    __shared__ int32_t c[HINT_SMEM_BINS];     // the run's rows per key, then the rank counters
    __shared__ int32_t base[HINT_SMEM_BINS];  // the range reserved per key
    const int m = K + 1;
    for (int b = threadIdx.x; b < m; b += HINT_SMEM_THREADS) c[b] = 0;
    __syncthreads();
    int64_t r0, r1;
    hint_run(n, r0, r1);
    for (int64_t i = r0 + threadIdx.x; i < r1; i += HINT_SMEM_THREADS) atomicAdd(&c[hint_key(__ldcs(hint + i), K, cpos)], 1);
    __syncthreads();
    for (int b = threadIdx.x; b < m; b += HINT_SMEM_THREADS) {
        base[b] = c[b] ? atomicAdd(cursor + b, c[b]) : 0;
        c[b] = 0;
    }
    __syncthreads();
    for (int64_t i = r0 + threadIdx.x; i < r1; i += HINT_SMEM_THREADS) {
        const int32_t key = hint_key(__ldcs(hint + i), K, cpos);
        const int32_t pos = base[key] + atomicAdd(&c[key], 1);
        if ((uint32_t)pos < (uint32_t)n) perm[pos] = (int32_t)i;  // counts that do not match the hints: no stray write
    }
}

cudaError_t launch_hint_permutation(const int32_t *hint, int64_t n, int32_t K, const int32_t *cpos,
                                    const int32_t *cperm, const int32_t *hint_counts, int32_t *cnt, int32_t *perm,
                                    int num_sms, cudaStream_t s) {
    int64_t blocks = (n + 255) / 256;
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    // few keys: runs of at least 4096 rows per CTA, up to two CTAs per SM
    int64_t sblocks = (n + 4095) / 4096;
    if (sblocks > 2LL * num_sms) sblocks = 2LL * num_sms;
    if (sblocks < 1) sblocks = 1;
    if (hint_counts) {
        // the rows per hinted codeword are known (all hints valid): start offsets
        // straight from them, K + 1 entries with the last count 0
        launch_begin(s);
        scan_counts_kernel<<<1, SCAN_THREADS, 0, s>>>(hint_counts, K, K + 1, cnt, cpos ? cperm : nullptr);
        launch_end(s, "scan_counts_kernel");
    } else {
        cudaError_t e = cudaMemsetAsync(cnt, 0, (size_t)(K + 1) * sizeof(int32_t), s);
        if (e != cudaSuccess) return e;
        launch_begin(s);
        if (K + 1 <= HINT_SMEM_BINS) {
            hint_histogram_smem_kernel<<<(unsigned)sblocks, HINT_SMEM_THREADS, 0, s>>>(hint, n, K, cpos, cnt);
            launch_end(s, "hint_histogram_smem_kernel");
        } else {
            hint_histogram_kernel<<<(unsigned)blocks, 256, 0, s>>>(hint, n, K, cpos, cnt);
            launch_end(s, "hint_histogram_kernel");
        }
        // the scan turns cnt into start offsets in place
        launch_begin(s);
        scan_counts_kernel<<<1, SCAN_THREADS, 0, s>>>(cnt, K + 1, K + 1, cnt, nullptr);
        launch_end(s, "scan_counts_kernel");
    }
    launch_begin(s);
    if (K + 1 <= HINT_SMEM_BINS) {
        hint_scatter_smem_kernel<<<(unsigned)sblocks, HINT_SMEM_THREADS, 0, s>>>(hint, n, K, cpos, cnt, perm);
        launch_end(s, "hint_scatter_smem_kernel");
    } else {
        hint_scatter_kernel<<<(unsigned)blocks, 256, 0, s>>>(hint, n, K, cpos, cnt, perm);
        launch_end(s, "hint_scatter_kernel");
    }
    return cudaGetLastError();
}

// Seeds for a cold assignment with few codeword tiles: hint[i] = the nearest of
// codewords 0 .. S - 1 (fp32 direct form, first on ties; S <= SAMPLE_HINT_MAX), one
// thread per kernel. Without a seed the tensor-core pass tests every row's first
// tile exactly (no threshold yet); with it a row only meets the few codewords
// nearer than its seed. (When the codebook was drawn from the kernels, the first S
// codewords are a random sample of them.) The hints do not change the answer.
__global__ void __launch_bounds__(256) sample_hint_kernel(const float *__restrict__ W, int64_t n,
                                                          const float *__restrict__ C, int32_t S,
                                                          int32_t *__restrict__ hint) {
    __shared__ float cs[SAMPLE_HINT_MAX * D];
    for (int e = threadIdx.x; e < S * D; e += blockDim.x) cs[e] = C[e];
    __syncthreads();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        float x[D];
#pragma unroll
        for (int j = 0; j < D; ++j) x[j] = W[i * D + j];
        float best = __int_as_float(0x7f800000);
        int32_t bk = 0;
        for (int32_t k = 0; k < S; ++k) {
            const float d = direct_distance(x, cs + k * D);
            if (d < best) {
                best = d;
                bk = k;
            }
        }
        hint[i] = bk;
    }
}

cudaError_t launch_sample_hints(const float *W, int64_t n, const float *C, int32_t S, int32_t *hint, int num_sms,
                                cudaStream_t s) {
    if (S < 1 || S > SAMPLE_HINT_MAX) return cudaErrorInvalidValue;
    const int64_t want = (n + 255) / 256;
    const int64_t blocks = want < 8LL * num_sms ? want : 8LL * num_sms;
    launch_begin(s);
    sample_hint_kernel<<<(unsigned)blocks, 256, 0, s>>>(W, n, C, S, hint);
    launch_end(s, "sample_hint_kernel");
    return cudaGetLastError();
}

cudaError_t launch_dist_block_sums(const float *dist, int64_t n, double *blocksum, int *nblocksum, cudaStream_t s) {
    const int64_t blocks = (n + 255) / 256;
    launch_begin(s);
    dist_block_sums_kernel<<<(unsigned)blocks, 256, 0, s>>>(dist, n, blocksum);
    launch_end(s, "dist_block_sums_kernel");
    *nblocksum = (int)blocks;
    return cudaGetLastError();
}

cudaError_t launch_assign_tc(const float *W, int64_t n, const float *C, const float *Cpk, int32_t K,
                             const int32_t *hint, const int32_t *perm, int32_t *idx, float *dist, double *blocksum,
                             int *nblocksum, Header *hdr, cudaStream_t s, const TcYy *yy) {
    // One CTA per SM (it owns all of TMEM); the shared layout alone rules out a second.
    // (+ 1024: alignment slack of the dynamic base)
    constexpr size_t plain = sizeof(TcShared) + 1024;
    constexpr size_t pruned_max = sizeof(TcPrunedShared) + (size_t)TC_ROWS * (YY_MAX_TILES + 4) + 1024;
    static_assert(plain <= 227 * 1024 && pruned_max <= 227 * 1024, "shared layout too large");
    static_assert(plain > 114 * 1024 && sizeof(TcPrunedShared) + 1024 > 114 * 1024, "two CTAs per SM would share TMEM");
    static_assert(sizeof(TcPrunedShared) % 16 == 0, "record alignment");
    const int64_t blocks = (n + TC_ROWS - 1) / TC_ROWS;
    const int32_t ntiles = tc_kpad(K) / TC_N;
    cudaError_t e;
    if (yy) {
        if (ntiles > YY_MAX_TILES || yy->stride < ntiles || yy->stride % 16 != 0 || !perm || !dist)
            return cudaErrorInvalidValue;
        const int smem = (int)(sizeof(TcPrunedShared) + (size_t)TC_ROWS * (yy->stride + 4)) + 1024;
        auto kern = test_hooks(hdr) ? assign_tc_pruned_kernel<true> : assign_tc_pruned_kernel<false>;
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        launch_begin(s);
        kern<<<(unsigned)blocks, TC_THREADS, smem, s>>>(W, n, C, Cpk, K, ntiles, hint, perm, idx, dist, hdr, *yy);
        launch_end(s, "assign_tc_pruned_kernel");
    } else {
        auto kern = test_hooks(hdr) ? assign_tc_kernel<true> : assign_tc_kernel<false>;
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plain);
        if (e != cudaSuccess) return e;
        launch_begin(s);
        kern<<<(unsigned)blocks, TC_THREADS, (int)plain, s>>>(W, n, C, Cpk, K, ntiles, hint, perm, idx, dist, blocksum,
                                                             hdr);
        launch_end(s, "assign_tc_kernel");
    }
    *nblocksum = (int)blocks;
    return cudaGetLastError();
}

}  // namespace kq
