// kq_reconstruct.cu -- test-time recovery (Sec. 3.2, last paragraph) and the
// codeword initialisation gather, on sm_103a.
//
// Recovery runs in the paper's order: first the kernel codebook is decoded once
// per codeword (C_hat[k][j] = levels[codes[k][j]], or C itself without codes) into
// 48-byte rows that are 16-byte aligned, then the weight tensor is gathered,
// W'[i] = C_hat[idx[i]]. The gather is HBM-bound (4 B of index read and 36 B of
// weights written per kernel); the decoded codebook (<= a few MB) stays in L2.
// The gather kernel is described above its definition.
#include "kq_internal.cuh"

namespace kq {

constexpr int R_THREADS = 256;

// K only: C into 48-byte rows (Cp). K+C: the 9 codes of a codeword into one
// 64-bit word (Cq), 7 bits each so an out-of-range code (>= 64) stays visible and
// decodes to 0.
__global__ void __launch_bounds__(256)
decode_codebook_kernel(const float *__restrict__ C, int32_t K, const uint8_t *__restrict__ codes,
                       float *__restrict__ Cp, unsigned long long *__restrict__ Cq, uint32_t *status) {
    // the K+C gather is launched as a programmatic dependent of this kernel: let it
    // start its prologue now (it waits for this grid before reading Cq)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    if (codes) {
        unsigned long long q = 0;
        bool bad = false;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            const uint32_t c = codes[(int64_t)k * D + j];
            bad |= c >= LEVELS;
            q |= (unsigned long long)(c < LEVELS ? c : LEVELS) << (7 * j);
        }
        if (bad) set_flag(status, KQ_FLAG_CODE_RANGE);
        Cq[k] = q;
        return;
    }
    float c[CP_FLOATS];
#pragma unroll
    for (int j = 0; j < D; ++j) c[j] = C[(int64_t)k * D + j];
#pragma unroll
    for (int j = D; j < CP_FLOATS; ++j) c[j] = 0.f;
    float4 *dst = reinterpret_cast<float4 *>(Cp + (int64_t)k * CP_FLOATS);
    dst[0] = make_float4(c[0], c[1], c[2], c[3]);
    dst[1] = make_float4(c[4], c[5], c[6], c[7]);
    dst[2] = make_float4(c[8], c[9], c[10], c[11]);
}

// Each warp owns groups of G_CHUNKS x 32 consecutive kernels. All index loads of
// a group are issued first, then all codebook-row gathers (three 16-byte loads per
// kernel), so a warp keeps a whole group of requests in flight. The rows go into a
// per-warp shared tile (kernel i at float offset 9i, conflict-free), which the warp
// then writes out with coalesced streaming float4 stores.
constexpr int G_CHUNKS = 2;
constexpr unsigned long long ALL_CODES_OUT_OF_RANGE = 0x4081020408102040ull;  // nine 7-bit fields = 64
constexpr int G_ROWS = 32 * G_CHUNKS;
constexpr int G_TILE_FLOATS = G_ROWS * D;
constexpr int R_WARPS = R_THREADS / 32;

__global__ void __launch_bounds__(R_THREADS)
gather_rows_kernel(const int32_t *__restrict__ idx, int64_t n, const float *__restrict__ Cp, int32_t K,
                   float *__restrict__ W_out, uint32_t *status) {
    __shared__ __align__(16) float tile[R_WARPS][G_TILE_FLOATS];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t ngroups = n / G_ROWS;  // full groups; the ragged end is handled below
    bool bad = false;
    float *t = tile[warp];
    for (int64_t g = (int64_t)blockIdx.x * R_WARPS + warp; g < ngroups; g += (int64_t)gridDim.x * R_WARPS) {
        const int64_t r0 = g * G_ROWS;
        int32_t k[G_CHUNKS];
#pragma unroll
        for (int c = 0; c < G_CHUNKS; ++c) k[c] = __ldcs(idx + r0 + c * 32 + lane);
        float4 v[G_CHUNKS][3];
#pragma unroll
        for (int c = 0; c < G_CHUNKS; ++c) {
            const bool ok = (uint32_t)k[c] < (uint32_t)K;
            bad |= !ok;
            const float4 *src = reinterpret_cast<const float4 *>(Cp + (int64_t)(ok ? k[c] : 0) * CP_FLOATS);
            v[c][0] = __ldg(src);
            v[c][1] = __ldg(src + 1);
            v[c][2] = __ldg(src + 2);
            if (!ok) v[c][0] = v[c][1] = v[c][2] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int c = 0; c < G_CHUNKS; ++c) {
            float *row = t + (c * 32 + lane) * D;
            row[0] = v[c][0].x; row[1] = v[c][0].y; row[2] = v[c][0].z; row[3] = v[c][0].w;
            row[4] = v[c][1].x; row[5] = v[c][1].y; row[6] = v[c][1].z; row[7] = v[c][1].w;
            row[8] = v[c][2].x;
        }
        __syncwarp();
        const float4 *t4 = reinterpret_cast<const float4 *>(t);
        float4 *d4 = reinterpret_cast<float4 *>(W_out + r0 * D);
#pragma unroll
        for (int v2 = lane; v2 < G_TILE_FLOATS / 4; v2 += 32) __stcs(d4 + v2, t4[v2]);
        __syncwarp();
    }

    // ragged end (fewer than G_ROWS kernels): CTA 0, plain loads and stores
    if (blockIdx.x == 0) {
        for (int64_t i = ngroups * G_ROWS + threadIdx.x; i < n; i += R_THREADS) {
            const int32_t kk = idx[i];
            const bool ok = (uint32_t)kk < (uint32_t)K;
            bad |= !ok;
#pragma unroll
            for (int j = 0; j < D; ++j) W_out[i * D + j] = ok ? Cp[(int64_t)kk * CP_FLOATS + j] : 0.f;
        }
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) set_flag(status, KQ_FLAG_INDEX_RANGE);
}

// Index loads of chunk pair c2 (two chunks of 32 kernels, the second only when it
// exists) and the code-word gathers of a loaded pair.
__device__ __forceinline__ void gc_load_idx(const int32_t *__restrict__ idx, int64_t nch, int64_t c2, int lane,
                                            int32_t (&k)[2]) {
    k[0] = __ldcs(idx + 2 * c2 * 32 + lane);
    k[1] = 2 * c2 + 1 < nch ? __ldcs(idx + (2 * c2 + 1) * 32 + lane) : 0;
}
__device__ __forceinline__ void gc_gather(const unsigned long long *__restrict__ Cq, int32_t K, const int32_t (&k)[2],
                                          bool two, unsigned long long (&q)[2], bool &bad) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const bool ok = (uint32_t)k[h] < (uint32_t)K;
        bad |= !ok && (h == 0 || two);
        q[h] = ok ? __ldg(Cq + k[h]) : ALL_CODES_OUT_OF_RANGE;
    }
}

// A lane's float4 slots of a 32-kernel chunk (288 floats, 72 float4): float4 lane
// and lane + 32 of every chunk (slots 0, 1), and float4 64 + (lane & 7) of the
// first chunk of a pair (lanes 0-7) or of the second (lanes 8-15) (slot 2, both
// chunks' last eight float4 in one pass). A slot's first element is code j0 of the
// chunk's kernel ra; elements e < split belong to ra, the rest are codes 0-2 of
// kernel ra + 1 (all in the low word of its code word).
struct GcSlots {
    int ra[3], j0[3], split[3];
};
__device__ __forceinline__ GcSlots gc_slots(int lane) {
    GcSlots g;
#pragma unroll
    for (int s = 0; s < 3; ++s) {
        const int v = s < 2 ? lane + 32 * s : 64 + (lane & 7);
        g.ra[s] = (4 * v) / D;
        g.j0[s] = 4 * v - D * g.ra[s];
        g.split[s] = D - g.j0[s];
    }
    return g;
}
// The four weights of a slot: qa the code word of kernel ra, qb the low word of
// kernel ra + 1's; lv the replicated level table.
__device__ __forceinline__ float4 gc_decode(unsigned long long qa, uint32_t qb, int j0, int split,
                                            const float (*lv)[32], int lane) {
    float r[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const bool first = e < split;
        const int j = first ? j0 + e : e - split;
        r[e] = lv[((first ? qa : (unsigned long long)qb) >> (7 * j)) & 127u][lane];
    }
    return make_float4(r[0], r[1], r[2], r[3]);
}

// A warp's place in the loop of gather_codes_rows: its first chunk pair and the
// indices of its first two pairs, loaded by gc_start (before the code words exist).
struct GcPipe {
    int64_t c2;
    int32_t k[2], kn[2];
};
__device__ __forceinline__ void gc_start(const int32_t *__restrict__ idx, int64_t n, int64_t cta, int64_t ncta,
                                         GcPipe &p) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nch = n / 32;
    const int64_t npairs = nch / 2 + (nch & 1);
    const int64_t step = ncta * R_WARPS;
    p.c2 = cta * R_WARPS + warp;
    p.k[0] = p.k[1] = p.kn[0] = p.kn[1] = 0;
    if (p.c2 < npairs) {
        gc_load_idx(idx, nch, p.c2, lane, p.k);
        if (p.c2 + step < npairs) gc_load_idx(idx, nch, p.c2 + step, lane, p.kn);
    }
}

// The loop of gather_codes_kernel over the chunk pairs of CTA `cta` of `ncta` (and
// the ragged end in CTA 0), from the state gc_start left; lv is the replicated level
// table. Software-pipelined by one pair: while pair c2 is decoded and stored, the
// code words of the warp's next pair and the indices of the one after are already in
// flight, so a warp waits for neither the index read from DRAM nor the gather from
// L2. Returns whether this thread saw an index outside [0, K).
__device__ __forceinline__ bool gather_codes_rows(const int32_t *__restrict__ idx, int64_t n,
                                                  const unsigned long long *__restrict__ Cq, int32_t K,
                                                  float *__restrict__ W_out, const float (*lv)[32], const GcSlots &sl,
                                                  GcPipe p, int64_t cta, int64_t ncta) {
    const int lane = threadIdx.x & 31;
    bool bad = false;
    const int64_t nch = n / 32;
    const int64_t npairs = nch / 2 + (nch & 1);
    const int64_t step = ncta * R_WARPS;
    int64_t c2 = p.c2;
    int32_t kn[2] = {p.kn[0], p.kn[1]};
    unsigned long long q[2] = {0ull, 0ull};
    if (c2 < npairs) gc_gather(Cq, K, p.k, 2 * c2 + 1 < nch, q, bad);
    // slot 2 reads kernels 28-31 of both chunks from lanes 28-31 (first chunk) and
    // 12-15 (second chunk, moved there by one shuffle pair)
    const int off2 = lane < 8 ? 0 : 16;
    const int sa2 = sl.ra[2] - off2, sb2 = min(sl.ra[2] + 1, 31) - off2;
    for (; c2 < npairs; c2 += step) {
        const int64_t c2n = c2 + step;
        unsigned long long qn[2] = {0ull, 0ull};
        int32_t knn[2] = {0, 0};
        if (c2n < npairs) gc_gather(Cq, K, kn, 2 * c2n + 1 < nch, qn, bad);
        if (c2n + step < npairs) gc_load_idx(idx, nch, c2n + step, lane, knn);
        const bool two = 2 * c2 + 1 < nch;
        float4 *d4[2] = {reinterpret_cast<float4 *>(W_out + 2 * c2 * 32 * D),
                         reinterpret_cast<float4 *>(W_out + (2 * c2 + 1) * 32 * D)};
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            if (h == 1 && !two) break;
            const uint32_t qlo = (uint32_t)q[h], qhi = (uint32_t)(q[h] >> 32);
#pragma unroll
            for (int s = 0; s < 2; ++s) {
                const int rb = min(sl.ra[s] + 1, 31);
                const unsigned long long qa = ((unsigned long long)__shfl_sync(0xffffffffu, qhi, sl.ra[s]) << 32) |
                                              __shfl_sync(0xffffffffu, qlo, sl.ra[s]);
                const uint32_t qb = __shfl_sync(0xffffffffu, qlo, rb);
                __stcs(d4[h] + lane + 32 * s, gc_decode(qa, qb, sl.j0[s], sl.split[s], lv, lane));
            }
        }
        {
            const uint32_t t_lo = __shfl_sync(0xffffffffu, (uint32_t)q[1], (lane + 16) & 31);
            const uint32_t t_hi = __shfl_sync(0xffffffffu, (uint32_t)(q[1] >> 32), (lane + 16) & 31);
            const uint32_t wlo = lane >= 16 ? (uint32_t)q[0] : t_lo;
            const uint32_t whi = lane >= 16 ? (uint32_t)(q[0] >> 32) : t_hi;
            const unsigned long long qa = ((unsigned long long)__shfl_sync(0xffffffffu, whi, sa2) << 32) |
                                          __shfl_sync(0xffffffffu, wlo, sa2);
            const uint32_t qb = __shfl_sync(0xffffffffu, wlo, sb2);
            const float4 v = gc_decode(qa, qb, sl.j0[2], sl.split[2], lv, lane);
            if (lane < 8)
                __stcs(d4[0] + 64 + lane, v);
            else if (lane < 16 && two)
                __stcs(d4[1] + 56 + lane, v);  // float4 64 + (lane - 8)
        }
        q[0] = qn[0];
        q[1] = qn[1];
        kn[0] = knn[0];
        kn[1] = knn[1];
    }
    // ragged end (< 32 kernels): CTA 0, plain loads and stores
    if (cta == 0) {
        for (int64_t i = nch * 32 + threadIdx.x; i < n; i += R_THREADS) {
            const int32_t kk = idx[i];
            const bool ok = (uint32_t)kk < (uint32_t)K;
            bad |= !ok;
            const unsigned long long q = ok ? Cq[kk] : ALL_CODES_OUT_OF_RANGE;
#pragma unroll
            for (int j = 0; j < D; ++j) W_out[i * D + j] = lv[(q >> (7 * j)) & 127u][0];
        }
    }
    return bad;
}

// K+C recovery. A warp owns pairs of 32-kernel chunks (1152 output bytes = 72
// float4 each). Each lane fetches the packed codes of its own kernel (one 8-byte
// word, instead of a 36-byte row), then produces output float4 number lane and
// lane + 32 of each chunk, and lanes 0-15 the last eight float4 of both chunks
// (gc_slots), directly: the at most two kernels a float4 spans send their code
// words by shuffle, and every code is looked up in a level table replicated across
// the 32 shared-memory banks (level l for lane L at [l][L]: no bank conflicts). The
// stores are coalesced streaming float4 stores; one resident wave of CTAs, each
// warp's loop software-pipelined (gather_codes_rows). Launched as a programmatic
// dependent of decode_codebook_kernel (the launch, the first index loads and the
// level table overlap the decode; Cq is read after griddepcontrol.wait). Stress
// layer (n = 4,194,304), whole kq_reconstruct call, minimum of 30 calls: 42.9 us with
// two waves and no pipelining, 41.8 us pipelined, 40.3 us as here; decoding each
// lane's own kernel into a staging tile instead of the shuffles was slower.
__global__ void __launch_bounds__(R_THREADS, 4)
gather_codes_kernel(const int32_t *__restrict__ idx, int64_t n, const unsigned long long *__restrict__ Cq,
                    const float *__restrict__ levels, int32_t K, float *__restrict__ W_out, uint32_t *status) {
    __shared__ float lv[LEVELS + 1][32];  // row LEVELS decodes out-of-range codes to 0
    const int lane = threadIdx.x & 31;
    // the first indices are in flight while the level table is built (the decode
    // kernel does not write them; everything before it has completed)
    GcPipe p;
    gc_start(idx, n, blockIdx.x, gridDim.x, p);
    for (int e = threadIdx.x; e < (LEVELS + 1) * 32; e += R_THREADS)
        lv[e / 32][e % 32] = e / 32 < LEVELS ? levels[e / 32] : 0.f;
    const GcSlots sl = gc_slots(lane);
    __syncthreads();
    asm volatile("griddepcontrol.wait;" ::: "memory");  // Cq is written by the decode kernel
    const bool bad = gather_codes_rows(idx, n, Cq, K, W_out, lv, sl, p, blockIdx.x, gridDim.x);
    if (__any_sync(0xffffffffu, bad) && lane == 0) set_flag(status, KQ_FLAG_INDEX_RANGE);
}

// Fused 6-bit encode + K+C recovery (Sec. 3.2: the codebook scalars are encoded
// to their nearest levels, and the weights are the decoded codebook rows at the
// kernel indices), one cooperative launch: every CTA encodes a grid-stride share of
// the codewords into the packed code words of gather_codes_kernel (and the code
// bytes, when asked for), all CTAs meet at a bounded grid barrier, then gather.
__global__ void __launch_bounds__(R_THREADS, 3)
encode_gather_kernel(const float *__restrict__ C, int32_t K, const float *__restrict__ levels,
                     uint8_t *__restrict__ codes, unsigned long long *__restrict__ Cq, const int32_t *__restrict__ idx,
                     int64_t n, float *__restrict__ W_out, Header *hdr) {
    __shared__ float L[LEVELS];
    __shared__ float lv[LEVELS + 1][32];
    __shared__ int s_sorted;
    for (int e = threadIdx.x; e < (LEVELS + 1) * 32; e += R_THREADS)
        lv[e / 32][e % 32] = e / 32 < LEVELS ? levels[e / 32] : 0.f;
    if (threadIdx.x < LEVELS) L[threadIdx.x] = levels[threadIdx.x];
    __syncthreads();
    if (threadIdx.x == 0) s_sorted = levels_sorted(L);
    __syncthreads();
    const bool sorted = s_sorted;
    bool nonfinite = false;
    for (int64_t k = (int64_t)blockIdx.x * R_THREADS + threadIdx.x; k < K; k += (int64_t)gridDim.x * R_THREADS) {
        float v[D];
#pragma unroll
        for (int j = 0; j < D; ++j) v[j] = __ldg(C + k * D + j);
        unsigned long long q = 0;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            nonfinite |= !isfinite(v[j]);
            const int c = sorted ? nearest_level_sorted(v[j], L) : nearest_level(v[j], L);
            q |= (unsigned long long)c << (7 * j);
            if (codes) codes[k * D + j] = (uint8_t)c;
        }
        Cq[k] = q;
    }
    if (nonfinite) set_flag(&hdr->status, KQ_FLAG_NONFINITE);
    unsigned epoch = 0;
    if (!grid_barrier(hdr, gridDim.x, epoch)) return;
    const int lane = threadIdx.x & 31;
    GcPipe p;
    gc_start(idx, n, blockIdx.x, gridDim.x, p);
    const bool bad = gather_codes_rows(idx, n, Cq, K, W_out, lv, gc_slots(lane), p, blockIdx.x, gridDim.x);
    if (__any_sync(0xffffffffu, bad) && lane == 0) set_flag(&hdr->status, KQ_FLAG_INDEX_RANGE);
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

cudaError_t launch_decode_codebook(const float *C, int32_t K, const uint8_t *codes, float *Cp,
                                   unsigned long long *Cq, uint32_t *status, cudaStream_t s) {
    launch_begin(s);
    decode_codebook_kernel<<<(K + 255) / 256, 256, 0, s>>>(C, K, codes, Cp, Cq, status);
    launch_end(s, "decode_codebook_kernel");
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const int32_t *idx, int64_t n, const float *Cp, const unsigned long long *Cq,
                               const float *levels, int32_t K, float *W_out, uint32_t *status, int num_sms,
                               cudaStream_t s) {
    if (Cq) {
        // one resident wave (the loop is pipelined across a warp's pairs)
        int per_sm = 0;
        cudaError_t e0 = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_codes_kernel, R_THREADS, 0);
        if (e0 != cudaSuccess) return e0;
        if (per_sm < 1) per_sm = 1;
        int64_t blocks = ((n / 32 + 1) / 2 + R_WARPS - 1) / R_WARPS;
        if (blocks > (int64_t)per_sm * num_sms) blocks = (int64_t)per_sm * num_sms;
        if (blocks < 1) blocks = 1;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)blocks);
        cfg.blockDim = dim3(R_THREADS);
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // after decode_codebook_kernel
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        launch_begin(s);
        const cudaError_t e = cudaLaunchKernelEx(&cfg, gather_codes_kernel, idx, n, Cq, levels, K, W_out, status);
        launch_end(s, "gather_codes_kernel");
        return e != cudaSuccess ? e : cudaGetLastError();
    }
    const int64_t groups = n / G_ROWS;
    int64_t blocks = (groups + R_WARPS - 1) / R_WARPS;
    if (blocks > 8LL * num_sms) blocks = 8LL * num_sms;
    if (blocks < 1) blocks = 1;
    launch_begin(s);
    gather_rows_kernel<<<(unsigned)blocks, R_THREADS, 0, s>>>(idx, n, Cp, K, W_out, status);
    launch_end(s, "gather_rows_kernel");
    return cudaGetLastError();
}

cudaError_t launch_encode_gather(const float *C, int32_t K, const float *levels, uint8_t *codes,
                                 unsigned long long *Cq, const int32_t *idx, int64_t n, float *W_out, Header *hdr,
                                 int num_sms, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(&hdr->barrier, 0, 2 * sizeof(uint32_t), s);  // barrier counter, abort word
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, encode_gather_kernel, R_THREADS, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    int64_t blocks = ((n / 32 + 1) / 2 + R_WARPS - 1) / R_WARPS;
    const int64_t enc_blocks = ((int64_t)K + R_THREADS - 1) / R_THREADS;
    if (blocks < enc_blocks) blocks = enc_blocks;
    if (blocks > (int64_t)per_sm * num_sms) blocks = (int64_t)per_sm * num_sms;  // co-resident by construction
    if (blocks < 1) blocks = 1;
    void *params[] = {(void *)&C, (void *)&K, (void *)&levels, (void *)&codes, (void *)&Cq,
                      (void *)&idx, (void *)&n, (void *)&W_out, (void *)&hdr};
    launch_begin(s);
    e = cudaLaunchCooperativeKernel((const void *)encode_gather_kernel, dim3((unsigned)blocks), dim3(R_THREADS),
                                    params, 0, s);
    if (e != cudaSuccess) return e;
    launch_end(s, "encode_gather_kernel");
    return cudaGetLastError();
}

cudaError_t launch_init_codebook(const float *W, int64_t n, const int64_t *sel, int32_t K, float *C0,
                                 uint32_t *status, cudaStream_t s) {
    const int64_t total = (int64_t)K * D;
    launch_begin(s);
    init_codebook_kernel<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(W, n, sel, K, C0, status);
    launch_end(s, "init_codebook_kernel");
    return cudaGetLastError();
}

}  // namespace kq
