// kq_internal.cuh -- definitions shared by the libkq translation units (not part
// of the public ABI): workspace layout, device status bits, packed fp32x2 math.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <stddef.h>

#include "kq.h"

namespace kq {

constexpr int D = 9;             // omega^2 for 3x3 kernels (Sec. 3.1)
constexpr int LEVELS = 64;       // 6-bit codebook quantisation (Sec. 3.2)
constexpr int CD_FLOATS = 20;    // packed codeword for the assign kernel: 10 duplicated pairs
constexpr int CP_FLOATS = 12;    // padded codeword row for the reconstruct gather (48 B)
constexpr int ACC_WORDS = 16;    // int64 accumulator row per codeword: 9 sums, count, pad (128 B)
constexpr int ROW_BLOCK = 1024;  // kernels per assign CTA (128 threads x 8 rows)
constexpr int MAX_PART_BLOCKS = 512;  // bound on (row blocks x codeword splits) with split-K
// Tensor-core assign: a codeword tile is 256 codewords, streamed as 16 KiB of fp16
// operands (K = 32 per codeword) followed by the 256 codewords in fp32.
constexpr int TC_N = 256;
constexpr int TC_KD = 32;
constexpr int TC_TILE_H = TC_N * TC_KD * 2;
constexpr int TC_TILE_BYTES = TC_TILE_H + TC_N * D * 4;
// Pruned assignment in the fit (Yinyang-style tile bounds, kq_order.cu and
// kq_assign_tc.cu): codebooks of YY_MIN_K .. YY_MAX_K codewords (16 .. 256 tiles).
constexpr int32_t YY_MIN_K = 4096;
constexpr int32_t YY_MAX_K = 65536;
constexpr int YY_MAX_TILES = YY_MAX_K / TC_N;
inline bool yy_sizes(int32_t K) { return K >= YY_MIN_K && K <= YY_MAX_K; }
inline int32_t yy_stride(int32_t K) { return ((K + TC_N - 1) / TC_N + 15) / 16 * 16; }  // record bytes per kernel

// Split plane of an inner node of the codebook's k-d tree (kq_order.cu).
struct KdNode {
    float mean[D];
    float axis[D];
    float pivot;  // projections below go left
};

// Pruned assignment state (kq_assign_tc.cu): the codebook is packed in the order
// cperm (position -> codeword), and every kernel carries a record of one byte per
// tile, a lower bound on its distance to the tile's codewords (see kq_assign_tc.cu).
struct TcYy {
    const int32_t *cperm, *cpos;
    const float *tdrift;   // per tile: largest move of its codewords since the last pass
    unsigned char *rec;    // n x stride bytes
    float *dprev;          // n: lower bound on the kernel's distance to every codeword
    int32_t stride;
    int32_t read;          // 0: the records are not valid yet (every tile is processed)
};

// Fixed part of the workspace (first 4 KiB).
struct Header {
    uint32_t status;        // sticky KQ_FLAG_* bits
    // kq_test_inject_wait_fault (before the fields the entry points clear per call)
    uint32_t test_faults;       // KQ_TEST_* bits
    uint32_t test_wait_limit;   // poll limit of bounded waits (0: the normal ones)
    uint32_t maxabs_bits;   // max |W| as fp32 bits (update scale)
    uint32_t barrier;       // grid-barrier arrival counter (level fit)
    uint32_t abort;         // set when a bounded wait gives up
    uint32_t changed[3];    // level fit: "some code changed" per iteration (triple buffered)
    uint32_t fit_moved;     // fit (stop on stable): some row changed codeword in the last update
    uint32_t lo_w, lo_a;    // level fit: ordered-int minima over weighted / all scalars (init 0xff..)
    uint32_t hi_w, hi_a;    // level fit: ordered-int maxima over weighted / all scalars (init 0)
    uint32_t maxv_w;        // level fit: max |v| over weighted scalars (fp32 bits)
    uint32_t fit_moved1;    // one-launch fit (stop on stable): the same for odd iterations
    uint32_t cb_cmax, cb_hmax, cb_qmax;  // assign filter: codebook bounds (fp32 bits, see kq_assign.cu)
    uint32_t cb_craw;       // tensor-core assign: largest codeword norm before scaling (fp32 bits)
    uint32_t upd_bound;     // update: bound B on |W| the fixed-point scale was chosen for (fp32 bits)
    uint32_t upd_violation; // update: a |w| > B was seen (the exact fallback must run)
    int32_t upd_scale;      // update: the scale exponent S the accumulators hold
    int32_t fit_iters;      // one-launch fit: codebook updates performed
    unsigned long long wtotal;          // level fit: sum of weights
    unsigned long long lacc[3][LEVELS][2];  // level fit: (weight sum, fixed-point sum) per level
    double obj;                         // codebook-size search: objective of the last fit
    uint32_t yy_cnorm;                  // pruned fit: largest norm of the initial codebook (fp32 bits)
    unsigned long long yy_tiles_run;    // pruned fit: (row block, codeword tile) pairs processed, all passes
    unsigned long long yy_tiles_all;    // pruned fit: the pairs the same passes hold in all
};
static_assert(sizeof(Header) <= 4096, "header too large");
static_assert(offsetof(Header, yy_tiles_all) == offsetof(Header, yy_tiles_run) + 8,
              "kq_fit_prune_stats reads both counters with one copy");

struct WsLayout {
    size_t cd, acc, part, blocksum, cbuf0, cbuf1, cp, cq, cpk, dist, perm, pcnt, prev;
    // pruned fit (only when yy_sizes(K)): codebook order and its inverse, k-d tree
    // nodes and scratch, per-tile drift, per-kernel bound records and distances
    size_t cperm, cpos, kdtmp, kdkey, kdnode, tdrift, yrec, ydist, leaf, total;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

inline WsLayout ws_layout(int64_t n, int32_t K) {
    WsLayout L;
    size_t off = 4096;
    L.cd = off;       off = align_up(off + (size_t)K * CD_FLOATS * 4, 256);
    L.acc = off;      off = align_up(off + (size_t)K * ACC_WORDS * 8, 256);
    L.part = off;     off = align_up(off + (size_t)MAX_PART_BLOCKS * ROW_BLOCK * 8, 256);
    size_t nblk = (size_t)((n + 255) / 256) + MAX_PART_BLOCKS;  // >= CTAs of assign or combine
    L.blocksum = off; off = align_up(off + nblk * 8, 256);
    L.cbuf0 = off;    off = align_up(off + (size_t)K * D * 4, 256);
    L.cbuf1 = off;    off = align_up(off + (size_t)K * D * 4, 256);
    L.cp = off;       off = align_up(off + (size_t)K * CP_FLOATS * 4, 256);
    L.cq = off;       off = align_up(off + (size_t)K * 8, 256);
    L.cpk = off;      off = align_up(off + (size_t)((K + 255) / 256 * 256) * 128, 256);  // tensor-core codeword tiles
    L.dist = off;     off = align_up(off + (size_t)n * 4, 256);          // distances when the caller keeps none
    L.perm = off;     off = align_up(off + (size_t)n * 4, 256);          // rows in hint order
    L.pcnt = off;     off = align_up(off + (size_t)(K + 1) * 4, 256);    // per-hint counts / cursors
    L.prev = off;     off = align_up(off + (size_t)n * 4, 256);          // the fit's other assignment buffer
    const bool yy = yy_sizes(K);
    L.cperm = off;    off = align_up(off + (yy ? (size_t)K * 4 : 0), 256);
    L.cpos = off;     off = align_up(off + (yy ? (size_t)K * 4 : 0), 256);
    L.kdtmp = off;    off = align_up(off + (yy ? (size_t)K * 4 : 0), 256);
    L.kdkey = off;    off = align_up(off + (yy ? (size_t)K * 8 : 0), 256);
    L.kdnode = off;   off = align_up(off + (yy ? (size_t)2 * YY_MAX_TILES * sizeof(KdNode) : 0), 256);
    L.tdrift = off;   off = align_up(off + (yy ? (size_t)YY_MAX_TILES * 4 : 0), 256);
    L.yrec = off;     off = align_up(off + (yy ? (size_t)n * yy_stride(K) : 0), 256);
    L.ydist = off;    off = align_up(off + (yy ? (size_t)n * 4 : 0), 256);
    L.leaf = off;     off = align_up(off + (yy ? (size_t)n * 4 : 0), 256);
    L.total = off;
    return L;
}

// ---- packed fp32x2 arithmetic (sm_100+ PTX). Element 0 is the low 32 bits. ----
__device__ __forceinline__ unsigned long long pack2(float lo, float hi) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(unsigned long long v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ unsigned long long sub2(unsigned long long a, unsigned long long b) {
    unsigned long long d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ unsigned long long mul2(unsigned long long a, unsigned long long b) {
    unsigned long long d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ unsigned long long fma2(unsigned long long a, unsigned long long b,
                                                   unsigned long long c) {
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

// Order-preserving map of fp32 to uint32 (for atomicMin / atomicMax on floats).
__device__ __forceinline__ uint32_t f2ord(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord2f(uint32_t u) {
    return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}

// Scale exponent of exact fixed-point sums of n values bounded by B (B = max|W| of
// the fit): S = 62 - e with n B = f 2^e, f in [0.5, 1), so no sum reaches 2^62;
// 0 when B is zero or not finite (all-zero W: nothing to scale; non-finite W is
// flagged by the callers).
__device__ __forceinline__ int fit_sum_scale(float B, int64_t n) {
    if (!(B > 0.f) || !(B <= 3.402823466e38f)) return 0;
    int e;
    frexp((double)n * (double)B, &e);
    return 62 - e;
}

// rint(v * 2^S) as int64 (round half to even) for a finite fp32 v, using only
// integer operations: v = +-m * 2^(e - 150) (e the biased exponent, m with its
// implicit bit; subnormals m * 2^-149). Equal to rounding the exact product
// (double)v * 2^S to the nearest integer, ties to even. Callers choose S so that
// |v| * 2^S stays below 2^62; larger shifts are clamped (a finite-input bound
// violation only, reported elsewhere).
__device__ __forceinline__ long long fixed_rn(float v, int S) {
    const uint32_t u = __float_as_uint(v);
    const uint32_t e = (u >> 23) & 0xffu;
    uint32_t m = u & 0x7fffffu;
    int sh;
    if (e == 0) {
        sh = S - 149;
    } else {
        m |= 0x800000u;
        sh = (int)e - 150 + S;
    }
    unsigned long long q;
    if (sh >= 0) {
        q = (unsigned long long)m << (sh > 62 ? 62 : sh);
    } else if (sh <= -25) {
        q = 0;  // |v| * 2^S < 1/2
    } else {
        const int r = -sh;
        uint32_t qi = m >> r;
        const uint32_t rem = m & ((1u << r) - 1u);
        const uint32_t half = 1u << (r - 1);
        if (rem > half || (rem == half && (qi & 1u))) qi += 1u;
        q = qi;
    }
    return (u >> 31) ? -(long long)q : (long long)q;
}

__device__ __forceinline__ void set_flag(uint32_t *status, uint32_t bit) { atomicOr(status, bit); }

// ---- 6-bit encode (Sec. 3.2): nearest of 64 levels (used by the level fit and by
// the fused encode + recovery kernel)

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
// The code of v given cnt = #{l : L_l <= v} (levels sorted; see above).
__device__ __forceinline__ int nearest_from_count(float v, const float *L, int cnt) {
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

__device__ __forceinline__ int nearest_level_sorted(float v, const float *L) {
    if (v != v) return 0;  // NaN: no distance is below +inf
    int cnt = 0;           // number of levels <= v
#pragma unroll
    for (int step = 32; step > 0; step >>= 1)
        if (L[cnt + step - 1] <= v) cnt += step;
    cnt += L[cnt] <= v;  // cnt could only reach 63 above
    return nearest_from_count(v, L, cnt);
}

// Levels in non-decreasing order (and no NaN), so that nearest_level_sorted applies.
__device__ __forceinline__ bool levels_sorted(const float *L) {
    bool ok = true;
#pragma unroll 8
    for (int l = 0; l < LEVELS - 1; ++l) ok &= L[l] <= L[l + 1];
    return ok;
}


// Objective partial sums of a block of non-negative fp32 distances, in a fixed
// order and in double-float: an fp32 pair (hi, lo) holds the running sum hi + lo.
// One step: s = fl(a.hi + b.hi) with its exact rounding error (Knuth's TwoSum), the
// low parts added to that error, renormalised (Dekker's FastTwoSum). With every term
// non-negative each step is relatively accurate to ~2^-47, so a 256-term block sum is
// within ~1e-13 of the exact sum; fp32 operations with explicit rounding (no FMA
// contraction), far faster than GB300's fp64 pipe.
struct F2 {
    float hi, lo;
};
__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
    const float s = __fadd_rn(a.hi, b.hi);
    const float bb = __fsub_rn(s, a.hi);
    float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, bb)), __fsub_rn(b.hi, bb));
    e = __fadd_rn(e, __fadd_rn(a.lo, b.lo));
    const float hi = __fadd_rn(s, e);
    return F2{hi, __fsub_rn(e, __fsub_rn(hi, s))};
}
// a warp's 32 values (lane i holds v), summed by an xor butterfly: every lane ends
// with the same pair (each step is symmetric in its operands)
__device__ __forceinline__ F2 f2_warp_sum(float v) {
    F2 s{v, 0.f};
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const F2 t{__shfl_xor_sync(0xffffffffu, s.hi, o), __shfl_xor_sync(0xffffffffu, s.lo, o)};
        s = f2_add(s, t);
    }
    return s;
}
__device__ __forceinline__ double f2_to_double(F2 s) { return (double)s.hi + (double)s.lo; }

__device__ __forceinline__ bool finite9(const float *v) {
    bool ok = true;
#pragma unroll
    for (int j = 0; j < D; ++j) ok &= isfinite(v[j]);
    return ok;
}

// Bounded grid barrier for cooperative launches (all CTAs co-resident). The
// arrival counter hdr->barrier only grows (it must be zero at launch); barrier
// number `epoch` completes at epoch * nblocks arrivals. A wait that runs ~2 s sets
// KQ_FLAG_TIMEOUT and hdr->abort; every CTA then returns false and exits.
constexpr long long BARRIER_SPIN_LIMIT = 20000000;  // ~2 s of 100 ns naps
__device__ __forceinline__ bool grid_barrier(Header *h, unsigned nblocks, unsigned &epoch) {
    __shared__ int s_ok;
    __syncthreads();
    ++epoch;
    if (threadIdx.x == 0) {
        __threadfence();
        // (failure-detection tests: CTA 0 may be told not to arrive, and the limit shortened)
        if (!((h->test_faults & KQ_TEST_SKIP_ARRIVAL) && blockIdx.x == 0)) atomicAdd(&h->barrier, 1u);
        const long long limit = h->test_wait_limit ? (long long)h->test_wait_limit : BARRIER_SPIN_LIMIT;
        const unsigned target = epoch * nblocks;
        int ok = 1;
        for (long long spin = 0;; ++spin) {
            if (*(volatile unsigned *)&h->barrier >= target) break;
            if (*(volatile unsigned *)&h->abort) {
                ok = 0;
                break;
            }
            if (spin > limit) {
                atomicExch(&h->abort, 1u);
                set_flag(&h->status, KQ_FLAG_TIMEOUT);
                ok = 0;
                break;
            }
            __nanosleep(100);
        }
        __threadfence();
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
}

// Whether kq_test_inject_wait_fault has set test faults or a wait limit on the workspace
// whose header this is: the tensor-core assign kernels then run their instantiation
// with the test hooks (the normal one keeps its wait limits compile-time constants).
bool test_hooks(const Header *hdr);

// Every kernel launch is bracketed by launch_begin(s) before it and launch_end(s,
// name) after it (s: the launch stream, name: the kernel's, a string literal).
// launch_end counts the launch (kq_kernel_launches()); while a trace is on
// (kq_trace_start), the pair also records CUDA events around the kernel on s.
void launch_begin(cudaStream_t s);
void launch_end(cudaStream_t s, const char *name);

// ---- launchers (defined in the .cu files; all return cudaGetLastError()) ----
// Packs C for the assign kernel and computes the filter's codebook bounds into
// hdr->cb_* (which must be zero before the call; the launcher clears them).
cudaError_t launch_pack_codebook(const float *C, int32_t K, float *Cd, Header *hdr, cudaStream_t s);
// hint (nullable, may alias idx): a previous assignment used as a warm start.
cudaError_t launch_assign(const float *W, int64_t n, const float *Cd, const float *C, int32_t K, const int32_t *hint,
                          int32_t *idx, float *dist, double *blocksum, int *nblocksum, unsigned long long *part,
                          Header *hdr, int num_sms, cudaStream_t s);
// Tensor-core assignment (kq_assign_tc.cu): used where tc_eligible's cost estimate favours it.
bool tc_eligible(int64_t n, int32_t K, int num_sms);
// cperm (nullable): pack the codebook in that order; Cprev, tdrift (nullable): the
// largest codeword move per tile since Cprev.
// normed: the bounds are cleared and hdr->cb_craw holds C's largest norm already
// (launch_finalize_norm_tc).
cudaError_t launch_pack_codebook_tc(const float *C, int32_t K, float *Cpk, Header *hdr, cudaStream_t s,
                                    const int32_t *cperm = nullptr, const float *Cprev = nullptr,
                                    float *tdrift = nullptr, bool normed = false);
// yy (nullable): the pruned assignment over a codebook packed in yy->cperm order.
cudaError_t launch_assign_tc(const float *W, int64_t n, const float *C, const float *Cpk, int32_t K,
                             const int32_t *hint, const int32_t *perm, int32_t *idx, float *dist, double *blocksum,
                             int *nblocksum, Header *hdr, cudaStream_t s, const TcYy *yy = nullptr);
// The update's finalise of codeword k (sums at scale 2^S): c_k = (sum * 2^-S) / z_k
// in fp32 (C_prev when z_k = 0), counts[k] = z_k; the accumulator row is cleared
// unless keep. fp32 arithmetic (GB300's fp64 rate is low): sum -> fp32, exact
// power-of-two scaling, one IEEE division; within ~1.5 ulp of the exact mean.
__device__ __forceinline__ void finalize_codeword(unsigned long long *__restrict__ acc, int k, int S,
                                                  const float *C_prev, float *C_next, int32_t *__restrict__ counts,
                                                  bool keep) {
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
    if (keep) return;
    ulonglong2 *a2 = reinterpret_cast<ulonglong2 *>(a);
#pragma unroll
    for (int w = 0; w < ACC_WORDS / 2; ++w) a2[w] = make_ulonglong2(0ull, 0ull);
}

// The objective of an assignment from its block sums, in the order of
// sum_blocks_kernel: threads 0-255 take strided partial sums, xor butterflies within
// their warps, then thread 0 adds the eight warp sums in order. Every thread of the
// CTA calls it (a CTA barrier inside); wsum: 8 doubles of shared memory.
__device__ __forceinline__ void objective_sum_256(const double *__restrict__ blocksum, int nblocks, double *obj,
                                                  double *wsum) {
    if (threadIdx.x < 256) {
        double v = 0.0;
        for (int b = threadIdx.x; b < nblocks; b += 256) v += blocksum[b];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = v;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += wsum[w];
        *obj = t;
    }
}

// The fit's finalise for larger codebooks on the tensor-core path: launch_finalize
// (sums kept; obj nullable as there) that also reduces the new codebook's largest norm
// into hdr->cb_craw after clearing the packing bounds, so the next
// launch_pack_codebook_tc can skip both (normed).
cudaError_t launch_finalize_norm_tc(const double *blocksum, int nblocks, double *obj, unsigned long long *acc,
                                    int32_t K, Header *hdr, const float *C_prev, float *C_next, int32_t *counts,
                                    cudaStream_t s);
// Codebooks the tensor-core path packs in one CTA (at most 2048 padded codewords).
bool tc_pack_small(int32_t K);
// One step of the fit for such codebooks, one CTA: the objective of the assignment
// just made (obj nullable; the order of launch_sum_blocks), the update's finalise
// with the sums kept (as launch_finalize), and C_next packed for the next assignment
// (as launch_pack_codebook_tc).
cudaError_t launch_finalize_pack_small(const double *blocksum, int nblocks, double *obj, unsigned long long *acc,
                                       int32_t K, Header *hdr, const float *C_prev, float *C_next, int32_t *counts,
                                       float *Cpk, cudaStream_t s);
// Cold-start seeds: hint[i] = the nearest of codewords 0 .. S - 1, S <= SAMPLE_HINT_MAX.
constexpr int32_t SAMPLE_HINT_MAX = 64;
cudaError_t launch_sample_hints(const float *W, int64_t n, const float *C, int32_t S, int32_t *hint, int num_sms,
                                cudaStream_t s);
// Rows grouped by their hinted codeword (cnt: K + 1 ints of scratch, perm: n ints).
// cpos (nullable): groups ordered by cpos[hint] instead of the hint (the codebook's
// tile order); cperm is its inverse (needed with hint_counts). hint_counts: the
// number of rows per hinted codeword when the caller knows it (every hint then
// valid), else null (counted here).
cudaError_t launch_hint_permutation(const int32_t *hint, int64_t n, int32_t K, const int32_t *cpos,
                                    const int32_t *cperm, const int32_t *hint_counts, int32_t *cnt, int32_t *perm,
                                    int num_sms, cudaStream_t s);
// The k-d order of the codebook (kq_order.cu): cperm / cpos, tree nodes, and the
// initial codebook's largest norm in hdr->yy_cnorm.
cudaError_t launch_codebook_order(const float *C, int32_t K, int32_t *cperm, int32_t *cpos, int32_t *tmp,
                                  unsigned long long *keys, KdNode *nodes, Header *hdr, cudaStream_t s);
// First-pass hints: each kernel's nearest codeword within its k-d leaf tile
// (Cpk: the codebook packed in cperm order). leaf, cnt, perm: scratch.
cudaError_t launch_kd_hints(const float *W, int64_t n, const KdNode *nodes, int32_t K, const float *Cpk,
                            const int32_t *cperm, int32_t *leaf, int32_t *cnt, int32_t *perm, int32_t *hint,
                            int num_sms, cudaStream_t s);
// blocksum[b] = fp64 sum of dist over rows [256 b, 256 b + 256), in row order.
cudaError_t launch_dist_block_sums(const float *dist, int64_t n, double *blocksum, int *nblocksum, cudaStream_t s);
cudaError_t launch_sum_blocks(const double *blocksum, int nblocks, double *out, cudaStream_t s);

// Update step. Two ways to pick the fixed-point scale: `exact` takes B = max|W|
// (launch_maxabs first, as the fit does once); otherwise B is a guess from
// max|C_prev| checked against every value, with an exact fallback pass.
cudaError_t launch_maxabs(const float *W, int64_t count, uint32_t *maxabs_bits, uint32_t *status, int num_sms,
                          cudaStream_t s);
cudaError_t launch_update_prepare(const float *C_prev, int32_t K, unsigned long long *acc, Header *hdr,
                                  bool guess_from_codebook, cudaStream_t s);
cudaError_t launch_accumulate(const float *W, int64_t n, const int32_t *idx, int32_t K, Header *hdr,
                              unsigned long long *acc, bool guess, int num_sms, cudaStream_t s);
cudaError_t launch_update_fallback(const float *W, int64_t n, const int32_t *idx, int32_t K, Header *hdr,
                                   unsigned long long *acc, int num_sms, cudaStream_t s);
cudaError_t launch_histogram(const int32_t *idx, int64_t n, int32_t K, int32_t *counts, uint32_t *status,
                             int num_sms, cudaStream_t s);
// obj (nullable): also the objective, the sum of the nblocks block sums (as
// launch_sum_blocks, the same order).
cudaError_t launch_finalize(unsigned long long *acc, int32_t K, const Header *hdr, const float *C_prev,
                            float *C_next, int32_t *counts, cudaStream_t s, bool keep_sums = false,
                            const double *blocksum = nullptr, int nblocks = 0, double *obj = nullptr);
// The fit's update after its first iteration: the exact fixed-point sums of idx_old
// (held in acc) become those of idx_new by moving only the rows whose codeword changed.
// moved (nullable): set to 1 when some row's codeword changed. dist (nullable): also
// the per-256-row sums of dist into blocksum (as launch_dist_block_sums), their count
// into *nblocksum.
cudaError_t launch_accumulate_delta(const float *W, int64_t n, const int32_t *idx_old, const int32_t *idx_new,
                                    int32_t K, Header *hdr, unsigned long long *acc, int num_sms, cudaStream_t s,
                                    uint32_t *moved = nullptr, const float *dist = nullptr,
                                    double *blocksum = nullptr, int *nblocksum = nullptr);
// obj[j] = obj[from] for from < j <= to (the objective of a fit stopped at a fixed point).
cudaError_t launch_fill_objective(double *obj, int32_t from, int32_t to, cudaStream_t s);

// The whole k-means fit in one cooperative launch, for small codebooks (K <= 512).
bool small_fit_eligible(int64_t n, int32_t K);
// stop_on_stable: end at the first assignment equal to the previous one (the
// outputs are then those of all iters; hdr->fit_iters receives the updates made).
cudaError_t launch_small_fit(const float *W, int64_t n, const float *C0, int32_t K, int32_t iters, float *C_out,
                             int32_t *idx, int32_t *counts, double *objective, unsigned long long *acc, float *cbuf0,
                             float *cbuf1, double *blocksum, int max_blocksum, Header *hdr, int num_sms,
                             cudaStream_t s, bool stop_on_stable = false);

// shared_gpu: other work runs beside this fit (kq_fit_layers), so the one-cluster
// kernel is taken wherever it fits; alone, only where it is also the faster one.
cudaError_t launch_level_fit(const float *C, int64_t N, const int32_t *counts, int32_t max_iters, float *levels,
                             uint8_t *codes, int32_t *iters_run, Header *hdr, int num_sms, cudaStream_t s,
                             bool shared_gpu = false);
// kq_quantize_codebook_6bit with that choice (kq_api.cu)
kq_status quantize_codebook(const float *C, int32_t K, const int32_t *counts, int32_t max_iters, float *levels,
                            uint8_t *codes, int32_t *iters_run, void *ws, size_t ws_bytes, cudaStream_t s,
                            bool shared_gpu);

// Retraining with averaged gradients (Eq. 2): codebook finalise over the update's
// accumulators, and the 64-level segment mean of the quantised codebook.
cudaError_t launch_grad_finalize(unsigned long long *acc, int32_t K, const Header *hdr, float lr, const float *C,
                                 float *C_next, int32_t *counts, cudaStream_t s);
cudaError_t launch_level_grad(const float *G, int64_t n, const int32_t *idx, int32_t K, const uint8_t *codes,
                              float lr, const float *levels, float *levels_next, int64_t *counts, Header *hdr,
                              int num_sms, cudaStream_t s);

// Recovery. K only: C is re-laid as 48-byte rows (Cp) and gathered. K+C: the
// codes are packed 9 x 6 bits per codeword (Cq, 8 bytes) and decoded on the fly.
cudaError_t launch_decode_codebook(const float *C, int32_t K, const uint8_t *codes, float *Cp,
                                   unsigned long long *Cq, uint32_t *status, cudaStream_t s);
cudaError_t launch_gather_rows(const int32_t *idx, int64_t n, const float *Cp, const unsigned long long *Cq,
                               const float *levels, int32_t K, float *W_out, uint32_t *status, int num_sms,
                               cudaStream_t s);
cudaError_t launch_init_codebook(const float *W, int64_t n, const int64_t *sel, int32_t K, float *C0,
                                 uint32_t *status, cudaStream_t s);
// Fused 6-bit encode of the codebook against given levels + K+C recovery (one
// cooperative launch with a bounded grid barrier).
cudaError_t launch_encode_gather(const float *C, int32_t K, const float *levels, uint8_t *codes,
                                 unsigned long long *Cq, const int32_t *idx, int64_t n, float *W_out, Header *hdr,
                                 int num_sms, cudaStream_t s);

}  // namespace kq
