// kq_quant.cu -- 6-bit quantisation by 64-level 1-D k-means (Sec. 3.2) on sm_103a:
// of the kernel codebook (the K*9 codebook scalars, weight of a scalar = appearance
// count z_k of its codeword) and of fully-connected layers (any m scalars, weight 1).
//
// One cooperative launch runs the whole iteration: each CTA assigns a grid-stride
// slice of scalars to the nearest level (levels held in shared memory),
// accumulates per-level (weight, weight * fixed-point value) sums in per-warp
// shared int64 atomics, flushes them with global int64 atomics, and meets the
// other CTAs at a bounded grid barrier; after it every CTA computes the same new
// levels from the same integer sums. Integer sums make the result independent of
// the order of the atomics, so the levels and codes are bit-identical from run to
// run and to an exact-arithmetic CPU reference.
//
// Per-iteration global state is triple buffered (iteration it accumulates into
// slot it%3 while CTA 0 clears slot (it+1)%3, last read two barriers earlier),
// so one grid barrier per iteration suffices.
#include <type_traits>

#include "kq_internal.cuh"

namespace kq {

struct LevelArgs {
    const float *C;  // the N scalars
    int64_t N;
    const int32_t *counts;  // weight of scalar m: counts[m / 9], or 1 for every scalar when null
    int32_t max_iters;
    float *levels;
    uint8_t *codes;
    int32_t *iters_run;
    Header *hdr;
    int use_table;  // many scalars per thread: find codes through the bucket table
};

// nearest_level_sorted with the count found from a table instead of a binary
// search: Tb[b] is the number of levels at or below a point of bucket b of a
// uniform grid over [L_0, L_63] (inv_w buckets per unit), and the two walks make
// it the exact count for v whatever the guess; in most buckets no level lies,
// so each walk stops at its first test.
constexpr int Q_TABLE = 1024;
__device__ __forceinline__ int nearest_level_table(float v, const float *L, const uint8_t *Tb, float lo, float inv_w) {
    if (v != v) return 0;
    const float x = fminf(fmaxf((v - lo) * inv_w, 0.f), (float)(Q_TABLE - 1));
    int c = Tb[(int)x];
    while (c < LEVELS && L[c] <= v) ++c;
    while (c > 0 && L[c - 1] > v) --c;
    return nearest_from_count(v, L, c);
}


// Per-lane private accumulators: lane l of warp w adds into column l of its
// warp's [level][lane] arrays with plain read-modify-writes (no atomics; a 64-bit
// add would otherwise be a compare-and-swap loop, and lanes of a warp often share
// a level). Weight sums are 32-bit per lane; one that would overflow is first
// moved into the 64-bit global total of its level (only with very large counts).
constexpr int Q_THREADS = 256;
constexpr int Q_WARPS = Q_THREADS / 32;
struct LevelBins {
    unsigned long long q[Q_WARPS][LEVELS][32];  // sum of weight * fixed-point value
    uint32_t w[Q_WARPS][LEVELS][32];            // sum of weights
};

constexpr int Q_UNROLL = 4;  // scalars per thread whose loads are in flight together

// After the levels change (all threads): whether they are sorted, and if so the
// bucket table of nearest_level_table over [L_0, L_63].
__device__ __forceinline__ void build_table(const float *L, uint8_t *Tb, int &s_sorted, float &s_tlo, float &s_tinv,
                                            bool use_table) {
    if (threadIdx.x == 0) {
        const bool srt = levels_sorted(L);
        s_sorted = srt;
        const float lo = L[0], span = L[LEVELS - 1] - L[0];
        s_tlo = lo;
        // buckets per unit; 0 (every value in bucket 0) when the span is empty or not finite
        s_tinv = (srt && span > 0.f && span <= 3.402823466e38f) ? (float)Q_TABLE / span : 0.f;
    }
    __syncthreads();
    if (!use_table) return;
    const float lo = s_tlo, inv = s_tinv;
    const float w = inv > 0.f ? 1.f / inv : 0.f;
    for (int b = threadIdx.x; b < Q_TABLE; b += blockDim.x) {
        const float x = lo + ((float)b + 0.5f) * w;  // a point of bucket b (any guess is corrected)
        int cnt = 0;
#pragma unroll
        for (int step = 32; step > 0; step >>= 1)
            if (L[cnt + step - 1] <= x) cnt += step;
        cnt += L[cnt] <= x;
        Tb[b] = (uint8_t)cnt;
    }
    __syncthreads();
}

template <bool UNIT>
__global__ void __launch_bounds__(Q_THREADS, 1) level_fit_kernel(LevelArgs a) {
    constexpr int NP = Q_THREADS / LEVELS;  // reducer threads per level
    extern __shared__ __align__(16) unsigned char q_smem[];
    LevelBins &B = *reinterpret_cast<LevelBins *>(q_smem);
    __shared__ float L[LEVELS];
    __shared__ uint8_t Tb[Q_TABLE];
    __shared__ float s_tlo, s_tinv;
    __shared__ unsigned long long red_q[NP][LEVELS], red_w[NP][LEVELS];
    __shared__ int s_changed;
    __shared__ int s_stop;
    __shared__ int s_sorted;
    Header *h = a.hdr;
    const int64_t N = a.N;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t tid0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    unsigned epoch = 0;

    // Phase 0: value ranges, max |v| and total weight.
    {
        float lo_w = __int_as_float(0x7f800000), hi_w = -lo_w, lo_a = lo_w, hi_a = -lo_w, mv = 0.f;
        unsigned long long wt = 0;
        bool ok = true, badc = false;
        for (int64_t m = tid0; m < N; m += stride) {
            const float v = a.C[m];
            int32_t z = UNIT ? 1 : a.counts[(uint32_t)m / D];
            if (z < 0) {
                badc = true;
                z = 0;
            }
            if (!isfinite(v)) {
                ok = false;
                continue;
            }
            lo_a = fminf(lo_a, v);
            hi_a = fmaxf(hi_a, v);
            if (z > 0) {
                lo_w = fminf(lo_w, v);
                hi_w = fmaxf(hi_w, v);
                mv = fmaxf(mv, fabsf(v));
                wt += (unsigned long long)z;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            lo_w = fminf(lo_w, __shfl_xor_sync(0xffffffffu, lo_w, o));
            hi_w = fmaxf(hi_w, __shfl_xor_sync(0xffffffffu, hi_w, o));
            lo_a = fminf(lo_a, __shfl_xor_sync(0xffffffffu, lo_a, o));
            hi_a = fmaxf(hi_a, __shfl_xor_sync(0xffffffffu, hi_a, o));
            mv = fmaxf(mv, __shfl_xor_sync(0xffffffffu, mv, o));
            wt += __shfl_xor_sync(0xffffffffu, wt, o);
        }
        const bool all_ok = __all_sync(0xffffffffu, ok), any_bad = __any_sync(0xffffffffu, badc);
        if (lane == 0) {
            atomicMin(&h->lo_w, f2ord(lo_w));
            atomicMax(&h->hi_w, f2ord(hi_w));
            atomicMin(&h->lo_a, f2ord(lo_a));
            atomicMax(&h->hi_a, f2ord(hi_a));
            atomicMax(&h->maxv_w, __float_as_uint(mv));
            if (wt) atomicAdd(&h->wtotal, wt);
            if (!all_ok) set_flag(&h->status, KQ_FLAG_NONFINITE);
            if (any_bad) set_flag(&h->status, KQ_FLAG_INDEX_RANGE);
        }
    }
    for (int l = 0; l < LEVELS; ++l) {
        B.q[warp][l][lane] = 0ull;
        B.w[warp][l][lane] = 0;
    }
    if (!grid_barrier(h, gridDim.x, epoch)) return;

    // Phase 1: initial levels linspace(lo, hi, 64) in fp64, and the fixed-point scale.
    const unsigned long long A = __ldcg(&h->wtotal);
    const bool any = A > 0;
    const float lo = ord2f(__ldcg(any ? &h->lo_w : &h->lo_a));
    const float hi = ord2f(__ldcg(any ? &h->hi_w : &h->hi_a));
    const float M = __uint_as_float(__ldcg(&h->maxv_w));
    int S = 0;
    if (any && M > 0.f) {
        int e;
        frexp(__dmul_rn(__ull2double_rn(A), (double)M), &e);
        S = 62 - e;
    }
    const double down = ldexp(1.0, -S);
    if (threadIdx.x < LEVELS) {
        const double t = __ddiv_rn(__dmul_rn(__dsub_rn((double)hi, (double)lo), (double)threadIdx.x), 63.0);
        L[threadIdx.x] = __double2float_rn(__dadd_rn((double)lo, t));
    }
    __syncthreads();
    const bool use_table = a.use_table;
    build_table(L, Tb, s_sorted, s_tlo, s_tinv, use_table);

    int32_t updates = 0;
    for (int32_t it = 0; it < a.max_iters; ++it) {
        const int buf = it % 3, nxt = (it + 1) % 3;
        if (threadIdx.x == 0) s_changed = 0;
        if (blockIdx.x == 0) {
            if (threadIdx.x < 2 * LEVELS) (&h->lacc[nxt][0][0])[threadIdx.x] = 0ull;
            if (threadIdx.x == 0) h->changed[nxt] = 0u;
        }
        __syncthreads();
        bool changed = false;
        const bool sorted = s_sorted;
        const float tlo = s_tlo, tinv = s_tinv;
        for (int64_t m0 = tid0; m0 < N; m0 += Q_UNROLL * stride) {
            float v[Q_UNROLL];
            int32_t z[Q_UNROLL];
            uint32_t old[Q_UNROLL];
#pragma unroll
            for (int u = 0; u < Q_UNROLL; ++u) {
                const int64_t m = m0 + u * stride;
                const bool in = m < N;
                v[u] = in ? __ldg(a.C + m) : 0.f;
                z[u] = in ? (UNIT ? 1 : __ldg(a.counts + (uint32_t)m / D)) : 0;
                old[u] = (in && it > 0) ? a.codes[m] : 0u;
            }
#pragma unroll
            for (int u = 0; u < Q_UNROLL; ++u) {
                const int64_t m = m0 + u * stride;
                if (m >= N) break;
                const int code = !sorted     ? nearest_level(v[u], L)
                                 : use_table ? nearest_level_table(v[u], L, Tb, tlo, tinv)
                                             : nearest_level_sorted(v[u], L);
                changed |= it > 0 && old[u] != (uint32_t)code;
                a.codes[m] = (uint8_t)code;
                if (z[u] > 0) {
                    const long long q = fixed_rn(v[u], S);
                    B.q[warp][code][lane] += (unsigned long long)((long long)z[u] * q);
                    const uint32_t w0 = B.w[warp][code][lane];
                    if (!UNIT && w0 > 0xffffffffu - (uint32_t)z[u]) {  // would overflow: move to the total
                        atomicAdd(&h->lacc[buf][code][0], (unsigned long long)w0);
                        B.w[warp][code][lane] = (uint32_t)z[u];
                    } else {
                        B.w[warp][code][lane] = w0 + (uint32_t)z[u];
                    }
                }
            }
        }
        if (__any_sync(0xffffffffu, changed) && lane == 0) s_changed = 1;
        __syncthreads();
        {  // CTA totals per level: NP threads per level, 2 warps' columns each; bins cleared as read
            const int l = threadIdx.x % LEVELS, part = threadIdx.x / LEVELS;
            unsigned long long sq = 0ull, sw = 0ull;
            for (int w = 2 * part; w < 2 * part + 2; ++w)
#pragma unroll 8
                for (int j = 0; j < 32; ++j) {
                    const int ln = (j + l) & 31;  // lanes of a warp read 32 different banks
                    sq += B.q[w][l][ln];
                    sw += (unsigned long long)B.w[w][l][ln];
                    B.q[w][l][ln] = 0ull;
                    B.w[w][l][ln] = 0u;
                }
            red_q[part][l] = sq;
            red_w[part][l] = sw;
        }
        __syncthreads();
        if (threadIdx.x < LEVELS) {
            unsigned long long sq = 0ull, sw = 0ull;
#pragma unroll
            for (int p = 0; p < NP; ++p) {
                sq += red_q[p][threadIdx.x];
                sw += red_w[p][threadIdx.x];
            }
            if (sw) {
                atomicAdd(&h->lacc[buf][threadIdx.x][0], sw);
                atomicAdd(&h->lacc[buf][threadIdx.x][1], sq);
            }
        }
        if (threadIdx.x == 0 && s_changed) atomicOr(&h->changed[buf], 1u);
        if (!grid_barrier(h, gridDim.x, epoch)) return;
        if (threadIdx.x == 0) s_stop = (it > 0) && (__ldcg(&h->changed[buf]) == 0u);
        __syncthreads();
        if (s_stop) break;
        if (threadIdx.x < LEVELS) {
            const unsigned long long Wl = __ldcg(&h->lacc[buf][threadIdx.x][0]);
            const long long Ql = (long long)__ldcg(&h->lacc[buf][threadIdx.x][1]);
            if (Wl > 0)
                L[threadIdx.x] =
                    __double2float_rn(__ddiv_rn(__dmul_rn(__ll2double_rn(Ql), down), __ull2double_rn(Wl)));
        }
        __syncthreads();
        build_table(L, Tb, s_sorted, s_tlo, s_tinv, use_table);
        ++updates;
    }

    // Codes of the final levels.
    __syncthreads();
    const bool sorted = s_sorted;
    const float tlo = s_tlo, tinv = s_tinv;
    for (int64_t m0 = tid0; m0 < N; m0 += Q_UNROLL * stride) {
        float v[Q_UNROLL];
#pragma unroll
        for (int u = 0; u < Q_UNROLL; ++u) {
            const int64_t m = m0 + u * stride;
            v[u] = m < N ? __ldg(a.C + m) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < Q_UNROLL; ++u) {
            const int64_t m = m0 + u * stride;
            if (m < N)
                a.codes[m] = (uint8_t)(!sorted     ? nearest_level(v[u], L)
                                       : use_table ? nearest_level_table(v[u], L, Tb, tlo, tinv)
                                                   : nearest_level_sorted(v[u], L));
        }
    }
    if (blockIdx.x == 0) {
        if (threadIdx.x < LEVELS) a.levels[threadIdx.x] = L[threadIdx.x];
        if (threadIdx.x == 0 && a.iters_run) *a.iters_run = updates;
    }
}

template <bool UNIT>
cudaError_t launch_level_fit_t(const LevelArgs &args, int num_sms, cudaStream_t s) {
    constexpr int T = Q_THREADS;
    const int smem = (int)sizeof(LevelBins);
    static_assert(sizeof(LevelBins) <= 200 * 1024, "level bins too large");
    cudaError_t e = cudaFuncSetAttribute(level_fit_kernel<UNIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, level_fit_kernel<UNIT>, T, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    int64_t blocks = (args.N + T - 1) / T;
    if (blocks > (int64_t)num_sms) blocks = num_sms;  // one CTA per SM: co-resident by construction
    if (blocks < 1) blocks = 1;
    // a lane's 32-bit count of unit weights stays below 2^31
    if (UNIT && args.N / (blocks * T) >= (1LL << 31)) return cudaErrorInvalidValue;
    LevelArgs a = args;
    a.use_table = args.N / (blocks * T) >= 64;  // the table pays for itself from ~64 scalars per thread
    void *params[] = {&a};
    launch_begin(s);
    e = cudaLaunchCooperativeKernel((const void *)level_fit_kernel<UNIT>, dim3((unsigned)blocks), dim3(T), params,
                                    smem, s);
    if (e != cudaSuccess) return e;
    launch_end(s, "level_fit_kernel");
    return cudaGetLastError();
}

// ---- The same level fit on one thread-block cluster, for up to LFC_MAX_CL x
// ~13K scalars (a codebook of up to ~23K codewords): every CTA of the cluster keeps
// its slice of the scalars in shared memory for the whole fit (value, weight x
// fixed-point value, code; the weights per codeword), the per-level integer sums
// of the CTAs are exchanged through distributed shared memory, and the CTAs meet at
// the cluster's hardware barrier instead of a grid barrier in global memory. Every
// per-scalar decision and every sum is the grid kernel's (the same nearest-level
// functions, the same fixed-point values, exact integer sums), so levels, codes
// and iteration count are bit-identical to it. It occupies LFC_MAX_CL SMs or fewer,
// so other work (another layer's fit) runs beside it.
constexpr int LFC_THREADS = 1024;
constexpr int LFC_WARPS = LFC_THREADS / 32;
constexpr int LFC_MAX_CL = 16;
constexpr int64_t LFC_MIN_PER_CTA = 4096;  // fewer CTAs while each would hold fewer scalars than this
constexpr int64_t LFC_ALONE_MAX_N = 9 * 8192;  // scalars up to which it also wins alone on the GPU

struct LfcPhase0 {
    uint32_t lo_w, hi_w, lo_a, hi_a, maxv_w;  // ordered-int minima / maxima (maxv_w: fp32 bits)
    uint32_t flags;
    unsigned long long wt;
};

struct LfcShared {
    uint32_t bins[LFC_WARPS][LEVELS][4];         // per warp: q lo, q hi, w lo, w hi (carry-propagated)
    unsigned long long red[16][LEVELS][2];       // CTA reduction partials (w, q)
    unsigned long long tot[2][LEVELS][2];        // CTA totals per level (w, q), by iteration parity
    uint32_t chg[2];                             // "a code of this CTA changed", by parity
    LfcPhase0 p0, all;                           // this CTA's phase-0 figures, and the cluster's
    float L[LEVELS];
    uint8_t Tb[Q_TABLE];
    float tlo, tinv;
    int sorted, any_changed;
};

// unsigned 64-bit add into a (lo, hi) pair of 32-bit shared words with two 32-bit
// atomics: the carry out of the low word is the add's own (exact under any order)
__device__ __forceinline__ void add64_carry(uint32_t *lohi, unsigned long long x) {
    const uint32_t xl = (uint32_t)x;
    const uint32_t old = atomicAdd(lohi, xl);
    const uint32_t carry = (old + xl) < old ? 1u : 0u;
    const uint32_t xh = (uint32_t)(x >> 32) + carry;
    if (xh) atomicAdd(lohi + 1, xh);
}

__device__ __forceinline__ uint32_t cluster_map(const void *p, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"((uint32_t)__cvta_generic_to_shared(p)), "r"(rank));
    return r;
}
__device__ __forceinline__ unsigned long long dsmem_ld64(uint32_t a) {
    unsigned long long v;
    asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t dsmem_ld32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

constexpr size_t LFC_HDR = (sizeof(LfcShared) + 15) / 16 * 16;

// per: codewords (or, UNIT, scalars) per CTA; len_max = scalars per CTA at most.
// Grid = one cluster. Shared memory: LfcShared, then the slice's weight x fixed-point
// values (8 B), values (4 B), weights per codeword (4 B per 9) and codes (1 B).
template <bool UNIT>
__global__ void __launch_bounds__(LFC_THREADS, 1) level_fit_cluster_kernel(LevelArgs a, int64_t per, int64_t len_max) {
    extern __shared__ __align__(16) unsigned char lfc_smem[];
    LfcShared &S = *reinterpret_cast<LfcShared *>(lfc_smem);
    unsigned long long *zq = reinterpret_cast<unsigned long long *>(lfc_smem + LFC_HDR);
    float *vv = reinterpret_cast<float *>(zq + len_max);
    int32_t *zz = reinterpret_cast<int32_t *>(vv + len_max);
    uint8_t *cc = reinterpret_cast<uint8_t *>(zz + (UNIT ? 0 : len_max / D));
    Header *h = a.hdr;
    const int64_t N = a.N;
    const uint32_t rank = blockIdx.x, cl = gridDim.x;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int64_t e0, e1;  // this CTA's scalars
    if (UNIT) {
        e0 = min(N, (int64_t)rank * per);
        e1 = min(N, e0 + per);
    } else {
        const int64_t K = N / D, k0 = min(K, (int64_t)rank * per), k1 = min(K, k0 + per);
        e0 = k0 * D;
        e1 = k1 * D;
    }
    const int len = (int)(e1 - e0);

    // Phase 0 (as the grid kernel): value ranges, max |v|, total weight; the slice
    // is loaded into shared memory on the way.
    if (tid == 0) {
        S.p0 = LfcPhase0{0xffffffffu, 0u, 0xffffffffu, 0u, 0u, 0u, 0ull};
        S.all = S.p0;
    }
    __syncthreads();
    {
        float lo_w = __int_as_float(0x7f800000), hi_w = -lo_w, lo_a = lo_w, hi_a = -lo_w, mv = 0.f;
        unsigned long long wt = 0;
        bool ok = true, badc = false;
        for (int i = tid; i < len; i += LFC_THREADS) {
            const float v = a.C[e0 + i];
            vv[i] = v;
            int32_t z = UNIT ? 1 : a.counts[(e0 + i) / D];
            if (z < 0) {
                badc = true;
                z = 0;
            }
            if (!UNIT && i % D == 0) zz[i / D] = z;
            if (!isfinite(v)) {
                ok = false;
                continue;
            }
            lo_a = fminf(lo_a, v);
            hi_a = fmaxf(hi_a, v);
            if (z > 0) {
                lo_w = fminf(lo_w, v);
                hi_w = fmaxf(hi_w, v);
                mv = fmaxf(mv, fabsf(v));
                wt += (unsigned long long)z;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            lo_w = fminf(lo_w, __shfl_xor_sync(0xffffffffu, lo_w, o));
            hi_w = fmaxf(hi_w, __shfl_xor_sync(0xffffffffu, hi_w, o));
            lo_a = fminf(lo_a, __shfl_xor_sync(0xffffffffu, lo_a, o));
            hi_a = fmaxf(hi_a, __shfl_xor_sync(0xffffffffu, hi_a, o));
            mv = fmaxf(mv, __shfl_xor_sync(0xffffffffu, mv, o));
            wt += __shfl_xor_sync(0xffffffffu, wt, o);
        }
        const bool all_ok = __all_sync(0xffffffffu, ok), any_bad = __any_sync(0xffffffffu, badc);
        if (lane == 0) {
            atomicMin(&S.p0.lo_w, f2ord(lo_w));
            atomicMax(&S.p0.hi_w, f2ord(hi_w));
            atomicMin(&S.p0.lo_a, f2ord(lo_a));
            atomicMax(&S.p0.hi_a, f2ord(hi_a));
            atomicMax(&S.p0.maxv_w, __float_as_uint(mv));
            if (wt) atomicAdd(&S.p0.wt, wt);
            if (!all_ok) set_flag(&h->status, KQ_FLAG_NONFINITE);
            if (any_bad) set_flag(&h->status, KQ_FLAG_INDEX_RANGE);
        }
    }
    cluster_sync_all();
    if (tid < (int)cl) {  // the cluster's figures from every CTA's
        const uint32_t r = cluster_map(&S.p0, (uint32_t)tid);
        const uint32_t lw = dsmem_ld32(r), hw = dsmem_ld32(r + 4), la = dsmem_ld32(r + 8), ha = dsmem_ld32(r + 12),
                       mx = dsmem_ld32(r + 16);
        const unsigned long long wt = dsmem_ld64(r + 24);
        atomicMin(&S.all.lo_w, lw);
        atomicMax(&S.all.hi_w, hw);
        atomicMin(&S.all.lo_a, la);
        atomicMax(&S.all.hi_a, ha);
        atomicMax(&S.all.maxv_w, mx);
        if (wt) atomicAdd(&S.all.wt, wt);
    }
    __syncthreads();

    // Initial levels and the fixed-point scale (as the grid kernel)
    const unsigned long long A = S.all.wt;
    const bool any = A > 0;
    const float lo = ord2f(any ? S.all.lo_w : S.all.lo_a);
    const float hi = ord2f(any ? S.all.hi_w : S.all.hi_a);
    const float M = __uint_as_float(S.all.maxv_w);
    int Sx = 0;
    if (any && M > 0.f) {
        int e;
        frexp(__dmul_rn(__ull2double_rn(A), (double)M), &e);
        Sx = 62 - e;
    }
    const double down = ldexp(1.0, -Sx);
    if (tid < LEVELS) {
        const double t = __ddiv_rn(__dmul_rn(__dsub_rn((double)hi, (double)lo), (double)tid), 63.0);
        S.L[tid] = __double2float_rn(__dadd_rn((double)lo, t));
    }
    for (int i = tid; i < len; i += LFC_THREADS) {
        const int32_t z = UNIT ? 1 : zz[i / D];
        zq[i] = z > 0 ? (unsigned long long)((long long)z * fixed_rn(vv[i], Sx)) : 0ull;
    }
    __syncthreads();
    build_table(S.L, S.Tb, S.sorted, S.tlo, S.tinv, true);

    int32_t updates = 0;
    for (int32_t it = 0; it < a.max_iters; ++it) {
        const int par = it & 1;
        uint32_t *wb = &S.bins[warp][0][0];
        for (int e = lane; e < LEVELS * 4; e += 32) wb[e] = 0u;
        if (tid == 0) {
            S.chg[par] = 0u;  // last read by the other CTAs before the previous cluster barrier
            S.any_changed = 0;
        }
        __syncthreads();
        bool changed = false;
        const bool sorted = S.sorted;
        const float tlo = S.tlo, tinv = S.tinv;
        for (int i = tid; i < len; i += LFC_THREADS) {
            const int code = sorted ? nearest_level_table(vv[i], S.L, S.Tb, tlo, tinv) : nearest_level(vv[i], S.L);
            changed |= it > 0 && cc[i] != (uint8_t)code;
            cc[i] = (uint8_t)code;
            const int32_t z = UNIT ? 1 : zz[i / D];
            if (z > 0) {
                add64_carry(&S.bins[warp][code][0], zq[i]);
                add64_carry(&S.bins[warp][code][2], (unsigned long long)z);
            }
        }
        if (__any_sync(0xffffffffu, changed) && lane == 0) atomicOr(&S.chg[par], 1u);
        __syncthreads();
        {  // CTA totals per level: 16 partials of 2 warps each, then their sum
            const int l = tid & (LEVELS - 1), part = tid >> 6;
            unsigned long long sq = 0ull, sw = 0ull;
#pragma unroll
            for (int w = 2 * part; w < 2 * part + 2; ++w) {
                const uint4 b = *reinterpret_cast<const uint4 *>(&S.bins[w][l][0]);
                sq += ((unsigned long long)b.y << 32) | b.x;
                sw += ((unsigned long long)b.w << 32) | b.z;
            }
            S.red[part][l][0] = sw;
            S.red[part][l][1] = sq;
        }
        __syncthreads();
        if (tid < LEVELS) {
            unsigned long long sw = 0ull, sq = 0ull;
#pragma unroll
            for (int p = 0; p < 16; ++p) {
                sw += S.red[p][tid][0];
                sq += S.red[p][tid][1];
            }
            S.tot[par][tid][0] = sw;
            S.tot[par][tid][1] = sq;
        }
        cluster_sync_all();
        // the cluster's totals (each CTA sums every CTA's, in the same exact integers):
        // thread (r, l) fetches CTA r's totals of level l (S.red is free again)
        {
            const int l = tid & (LEVELS - 1), r = tid >> 6;
            if (r < (int)cl) {
                const uint32_t ra = cluster_map(&S.tot[par][l][0], (uint32_t)r);
                S.red[r][l][0] = dsmem_ld64(ra);
                S.red[r][l][1] = dsmem_ld64(ra + 8);
                if (l == 0 && dsmem_ld32(cluster_map(&S.chg[par], (uint32_t)r))) atomicOr(&S.any_changed, 1);
            }
        }
        __syncthreads();
        unsigned long long Wl = 0ull, Ql = 0ull;
        if (tid < LEVELS)
            for (int r = 0; r < (int)cl; ++r) {
                Wl += S.red[r][tid][0];
                Ql += S.red[r][tid][1];
            }
        if (it > 0 && S.any_changed == 0) break;  // the same decision in every CTA
        if (tid < LEVELS && Wl > 0)
            S.L[tid] = __double2float_rn(__ddiv_rn(__dmul_rn(__ll2double_rn((long long)Ql), down), __ull2double_rn(Wl)));
        __syncthreads();
        build_table(S.L, S.Tb, S.sorted, S.tlo, S.tinv, true);
        ++updates;
    }

    // codes of the final levels
    __syncthreads();
    {
        const bool sorted = S.sorted;
        const float tlo = S.tlo, tinv = S.tinv;
        for (int i = tid; i < len; i += LFC_THREADS)
            a.codes[e0 + i] =
                (uint8_t)(sorted ? nearest_level_table(vv[i], S.L, S.Tb, tlo, tinv) : nearest_level(vv[i], S.L));
    }
    if (rank == 0) {
        if (tid < LEVELS) a.levels[tid] = S.L[tid];
        if (tid == 0 && a.iters_run) *a.iters_run = updates;
    }
    cluster_sync_all();  // no CTA leaves while another may still read its shared memory
}

// Launches the cluster kernel when the fit fits one cluster; *launched = false
// (and nothing enqueued) otherwise.
template <bool UNIT>
cudaError_t launch_level_fit_cluster_t(const LevelArgs &args, cudaStream_t s, bool *launched) {
    *launched = false;
    const int64_t units = UNIT ? args.N : args.N / D;  // scalars, or codewords of 9 scalars
    const int64_t unit_len = UNIT ? 1 : D;
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    auto kern = level_fit_cluster_kernel<UNIT>;
    for (int cap = LFC_MAX_CL; cap >= 8; cap /= 2) {
        int cl = 1;
        while (cl < cap && (units + cl - 1) / cl * unit_len > LFC_MIN_PER_CTA) cl *= 2;
        const int64_t per = (units + cl - 1) / cl;
        const int64_t len_max = per * unit_len;
        const size_t smem = LFC_HDR + (size_t)len_max * (8 + 4 + 1) + (UNIT ? 0 : (size_t)per * 4);
        if (smem > (size_t)optin) return cudaSuccess;  // too large for one cluster: the grid kernel
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e == cudaSuccess && cl > 8) e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)cl);
        cfg.blockDim = dim3(LFC_THREADS);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = (unsigned)cl;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int nclusters = 0;
        if (cudaOccupancyMaxActiveClusters(&nclusters, kern, &cfg) != cudaSuccess || nclusters < 1) {
            (void)cudaGetLastError();  // not schedulable at this size: try a smaller cluster
            continue;
        }
        LevelArgs a = args;
        launch_begin(s);
        e = cudaLaunchKernelEx(&cfg, kern, a, per, len_max);
        if (e != cudaSuccess) return e;
        launch_end(s, "level_fit_cluster_kernel");
        *launched = true;
        return cudaGetLastError();
    }
    return cudaSuccess;
}

cudaError_t launch_level_fit(const float *C, int64_t N, const int32_t *counts, int32_t max_iters, float *levels,
                             uint8_t *codes, int32_t *iters_run, Header *hdr, int num_sms, cudaStream_t s,
                             bool shared_gpu) {
    // Clear everything but the sticky status word; minima start at the top of the order.
    cudaError_t e = cudaMemsetAsync(&hdr->maxabs_bits, 0, sizeof(Header) - offsetof(Header, maxabs_bits), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(&hdr->lo_w, 0xff, 2 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    const LevelArgs args{C, N, counts, max_iters, levels, codes, iters_run, hdr, 0};
    // Alone on the GPU the cluster kernel is the faster one up to ~8K codewords (per
    // iteration at K = 512 / 4096 / 16384: 5.1 / 6.3 / 11.1 us against the grid
    // kernel's 6.2 / 6.9 / 9.4 us); beside other work it always is, as it leaves
    // all but 16 SMs free. (The failure-detection tests exercise the grid kernel's
    // bounded barrier.)
    if ((shared_gpu || N <= LFC_ALONE_MAX_N) && !test_hooks(hdr)) {
        bool launched = false;
        e = counts ? launch_level_fit_cluster_t<false>(args, s, &launched)
                   : launch_level_fit_cluster_t<true>(args, s, &launched);
        if (e != cudaSuccess || launched) return e;
    }
    return counts ? launch_level_fit_t<false>(args, num_sms, s) : launch_level_fit_t<true>(args, num_sms, s);
}

}  // namespace kq
