// kq_order.cu -- spatial order of the codebook for the pruned assignment of the
// k-means fit (Sec. 3.1, Eq. 1). The paper speeds its clustering up with Yinyang
// k-means (Sec. 4.1), whose group bounds rule out codewords without changing the
// result; the tensor-core assignment applies the same idea to whole 256-codeword
// tiles, and for a bound over a tile to rule it out, the tile's codewords have to
// lie close together. This file orders the codebook so that they do.
//
// A k-d tree over the K codewords, built top down one level per launch: a node
// covering tiles [ta, tb) splits its codewords at rank 256 (tm - ta) along their
// principal axis (top eigenvector of the node's covariance, by power iteration),
// tm the middle tile, so both children hold whole tiles; a node of one tile is a
// leaf. The codewords of leaf t are the codebook positions [256 t, 256 t + 256).
//
// The same tree seeds the first assignment of a fit: a kernel descends to its
// leaf along the split planes and takes the nearest codeword of that leaf tile
// (exact fp32 direct form). These hints only change how fast the exact
// assignment that follows runs, never its result.
#include "kq_internal.cuh"

namespace kq {

constexpr int KD_THREADS = 512;
constexpr int KD_WARPS = KD_THREADS / 32;
constexpr int KD_COV = D * (D + 1) / 2;  // distinct entries of the 9 x 9 covariance
constexpr int KD_POWER_ITERS = 24;

__device__ __forceinline__ int kd_tile_at(int64_t j, int32_t T, int level) { return (int)((j * T) >> level); }

// One level of the tree: CTA j splits node (level, j). cur: codeword at each
// position before the split (nullptr: the identity); nxt: after it.
__global__ void __launch_bounds__(KD_THREADS) kd_split_kernel(const float *__restrict__ C, int32_t K, int32_t T,
                                                              int level, const int32_t *__restrict__ cur,
                                                              int32_t *__restrict__ nxt,
                                                              unsigned long long *__restrict__ keys,
                                                              KdNode *__restrict__ nodes) {
    const int j = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ta = kd_tile_at(j, T, level), tb = kd_tile_at(j + 1, T, level);
    const int64_t ea = (int64_t)ta * 256, eb = min((int64_t)tb * 256, (int64_t)K);
    if (tb - ta <= 1) {  // a leaf: its codewords keep their order
        for (int64_t e = ea + tid; e < eb; e += KD_THREADS) nxt[e] = cur ? cur[e] : (int32_t)e;
        return;
    }
    const int tm = kd_tile_at(2 * (int64_t)j + 1, T, level + 1);
    const int64_t r = (int64_t)(tm - ta) * 256;  // codewords that go left: whole tiles
    const float cnt = (float)(eb - ea);

    __shared__ float s_red[KD_WARPS][KD_COV];
    __shared__ float s_mean[D], s_cov[KD_COV], s_axis[D];
    __shared__ unsigned int hist[256];
    __shared__ unsigned long long s_prefix, s_mask;
    __shared__ long long s_rank;
    __shared__ unsigned int s_left, s_right;
    __shared__ int s_unique;

    // mean (fixed summation order: per thread, then xor-shuffle tree, then warps in order)
    float acc[KD_COV];
#pragma unroll
    for (int u = 0; u < D; ++u) acc[u] = 0.f;
    for (int64_t e = ea + tid; e < eb; e += KD_THREADS) {
        const int64_t k = cur ? cur[e] : e;
#pragma unroll
        for (int u = 0; u < D; ++u) acc[u] += C[k * D + u];
    }
#pragma unroll
    for (int u = 0; u < D; ++u) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[u] += __shfl_xor_sync(0xffffffffu, acc[u], o);
        if (lane == 0) s_red[warp][u] = acc[u];
    }
    __syncthreads();
    if (tid < D) {
        float s = 0.f;
        for (int w = 0; w < KD_WARPS; ++w) s += s_red[w][tid];
        s_mean[tid] = s / cnt;
    }
    __syncthreads();
    // covariance (upper triangle)
    float m[D];
#pragma unroll
    for (int u = 0; u < D; ++u) m[u] = s_mean[u];
#pragma unroll
    for (int u = 0; u < KD_COV; ++u) acc[u] = 0.f;
    for (int64_t e = ea + tid; e < eb; e += KD_THREADS) {
        const int64_t k = cur ? cur[e] : e;
        float d[D];
#pragma unroll
        for (int u = 0; u < D; ++u) d[u] = C[k * D + u] - m[u];
        int q = 0;
#pragma unroll
        for (int a = 0; a < D; ++a)
#pragma unroll
            for (int b = a; b < D; ++b) acc[q++] += d[a] * d[b];
    }
    __syncthreads();  // s_red is reused
#pragma unroll
    for (int u = 0; u < KD_COV; ++u) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[u] += __shfl_xor_sync(0xffffffffu, acc[u], o);
        if (lane == 0) s_red[warp][u] = acc[u];
    }
    __syncthreads();
    if (tid < KD_COV) {
        float s = 0.f;
        for (int w = 0; w < KD_WARPS; ++w) s += s_red[w][tid];
        s_cov[tid] = s;
    }
    __syncthreads();
    if (warp == 0) {  // principal axis by power iteration: lane a < 9 holds row a and v[a]
        float Arow[D];
#pragma unroll
        for (int b = 0; b < D; ++b) {
            const int lo = min(lane, b), hi = max(lane, b);  // upper-triangle index of (lo, hi)
            Arow[b] = lane < D ? s_cov[lo * D - lo * (lo - 1) / 2 + (hi - lo)] : 0.f;
        }
        float v = lane < D ? 1.f + 0.01f * lane : 0.f;  // not orthogonal to a dominant axis in practice
        bool ok = true;
        for (int it = 0; it < KD_POWER_ITERS; ++it) {
            float w = 0.f;
#pragma unroll
            for (int b = 0; b < D; ++b) w = fmaf(Arow[b], __shfl_sync(0xffffffffu, v, b), w);
            float nrm = w * w;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) nrm += __shfl_xor_sync(0xffffffffu, nrm, o);
            if (!(nrm > 1e-36f) || !(nrm < 1e36f)) {  // degenerate or out of range: keep the last axis
                ok = it > 0;
                break;
            }
            v = w * rsqrtf(nrm);
        }
        if (lane < D) s_axis[lane] = ok ? v : (lane == 0 ? 1.f : 0.f);
    }
    __syncthreads();
    float ax[D];
#pragma unroll
    for (int u = 0; u < D; ++u) ax[u] = s_axis[u];
    // keys: projection (order-preserving bits) above the codeword index, all distinct
    for (int64_t e = ea + tid; e < eb; e += KD_THREADS) {
        const int64_t k = cur ? cur[e] : e;
        float p = 0.f;
#pragma unroll
        for (int u = 0; u < D; ++u) p = fmaf(C[k * D + u] - m[u], ax[u], p);
        keys[e] = ((unsigned long long)f2ord(p) << 32) | (unsigned long long)(uint32_t)k;
    }
    if (tid == 0) {
        s_prefix = 0ull;
        s_mask = 0ull;
        s_rank = r;
        s_unique = 0;
    }
    __syncthreads();
    // radix select of the key of rank r, 8 bits at a time from the top; it stops as
    // soon as one key alone carries the selected prefix: that key is the one of rank
    // r, and comparing with the prefix (lower bits 0) puts exactly the r keys below
    // it on the left
    for (int shift = 56; shift >= 0 && !s_unique; shift -= 8) {
        for (int i = tid; i < 256; i += KD_THREADS) hist[i] = 0u;
        __syncthreads();
        const unsigned long long pre = s_prefix, msk = s_mask;
        for (int64_t e0 = ea; e0 < eb; e0 += KD_THREADS) {  // warp-uniform trip count
            const int64_t e = e0 + tid;
            unsigned int dg = 256u;  // no bin
            if (e < eb) {
                const unsigned long long key = keys[e];
                if ((key & msk) == pre) dg = (unsigned int)(key >> shift) & 255u;
            }
            // lanes with the same digit add once (keys of a node cluster in few bins)
            const unsigned int peers = __match_any_sync(0xffffffffu, dg);
            if (dg < 256u && lane == __ffs(peers) - 1) atomicAdd(&hist[dg], (unsigned int)__popc(peers));
        }
        __syncthreads();
        if (tid == 0) {
            long long rk = s_rank, cum = 0;
            int d = 255;
            for (int b = 0; b < 256; ++b) {
                if (rk < cum + (long long)hist[b]) {
                    d = b;
                    break;
                }
                cum += hist[b];
            }
            s_prefix = pre | ((unsigned long long)d << shift);
            s_mask = msk | (0xffull << shift);
            s_rank = rk - cum;
            s_left = 0u;
            s_right = 0u;
            s_unique = hist[d] == 1u;
        }
        __syncthreads();
    }
    const unsigned long long pivot = s_prefix;  // exactly r keys are below it (lower bits 0 after an early stop)
    for (int64_t e0 = ea; e0 < eb; e0 += KD_THREADS) {  // warp-uniform trip count
        const int64_t e = e0 + tid;
        const bool in = e < eb;
        const unsigned long long key = in ? keys[e] : 0ull;
        const bool left = in && key < pivot;
        // one atomic per warp and side, lanes placed by their rank within the warp
        const unsigned int bl = __ballot_sync(0xffffffffu, left), br = __ballot_sync(0xffffffffu, in && !left);
        unsigned int basel = 0u, baser = 0u;
        if (lane == 0) {
            if (bl) basel = atomicAdd(&s_left, (unsigned int)__popc(bl));
            if (br) baser = atomicAdd(&s_right, (unsigned int)__popc(br));
        }
        basel = __shfl_sync(0xffffffffu, basel, 0);
        baser = __shfl_sync(0xffffffffu, baser, 0);
        const unsigned int below = (1u << lane) - 1u;
        if (in) {
            const int32_t k = (int32_t)(uint32_t)key;
            if (left) {
                const unsigned int s = basel + __popc(bl & below);
                if ((int64_t)s < r) nxt[ea + s] = k;
            } else {
                const unsigned int s = baser + __popc(br & below);
                if (ea + r + (int64_t)s < eb) nxt[ea + r + s] = k;
            }
        }
    }
    if (tid == 0) {
        KdNode &nd = nodes[(1 << level) + j];
        for (int u = 0; u < D; ++u) {
            nd.mean[u] = m[u];
            nd.axis[u] = ax[u];
        }
        nd.pivot = ord2f((uint32_t)(pivot >> 32));
    }
}

// cpos[cperm[p]] = p, and the largest codeword norm (rounded up; NaN when a value
// is not finite) into hdr->yy_cnorm. identity: the tree had no split (one tile).
__global__ void __launch_bounds__(256) kd_finish_kernel(const float *__restrict__ C, int32_t K, int32_t *cperm,
                                                        int32_t *__restrict__ cpos, Header *hdr, bool identity) {
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    float nrm = 0.f;
    if (p < K) {
        if (identity) cperm[p] = p;
        const int32_t k = cperm[p];
        if ((uint32_t)k < (uint32_t)K) cpos[k] = p;
        bool ok = (uint32_t)k < (uint32_t)K;
        float s = 0.f;
#pragma unroll
        for (int u = 0; u < D; ++u) {
            const float c = ok ? C[(int64_t)k * D + u] : 0.f;
            ok &= isfinite(c);
            s = __fadd_ru(s, __fmul_ru(c, c));
        }
        nrm = ok ? __fsqrt_ru(s) : __int_as_float(0x7fc00000);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        nrm = __uint_as_float(max(__float_as_uint(nrm), __shfl_xor_sync(0xffffffffu, __float_as_uint(nrm), o)));
    if ((threadIdx.x & 31) == 0) atomicMax(&hdr->yy_cnorm, __float_as_uint(nrm));
}

// leaf[i] = the tile of the leaf that kernel i descends to.
__global__ void __launch_bounds__(256) kd_leaf_kernel(const float *__restrict__ W, int64_t n,
                                                      const KdNode *__restrict__ nodes, int32_t T,
                                                      int32_t *__restrict__ leaf) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    float x[D];
#pragma unroll
    for (int u = 0; u < D; ++u) x[u] = W[i * D + u];
    int level = 0;
    int64_t j = 0;
    for (;;) {
        const int ta = kd_tile_at(j, T, level), tb = kd_tile_at(j + 1, T, level);
        if (tb - ta <= 1) {
            leaf[i] = ta;
            return;
        }
        const KdNode &nd = nodes[(1 << level) + j];
        float p = 0.f;
#pragma unroll
        for (int u = 0; u < D; ++u) p = fmaf(x[u] - nd.mean[u], nd.axis[u], p);
        j = 2 * j + (p >= nd.pivot ? 1 : 0);
        ++level;
    }
}

// hint[row] = the nearest codeword of row's leaf tile (fp32 direct form, first
// position on ties), rows taken in the order of perm (grouped by leaf, so a CTA's
// rows read the same few tiles). The tile's codewords are the fp32 part of the
// packed tensor-core tile. A thread takes LS_ROWS consecutive slots: when they
// share a leaf (all but the slots at a leaf boundary) each codeword is loaded once
// for all of them. (The hints only seed the tensor-core pass; any choice gives the
// same assignment.)
constexpr int LS_ROWS = 4;
__global__ void __launch_bounds__(256) kd_leaf_search_kernel(const float *__restrict__ W, int64_t n,
                                                             const int32_t *__restrict__ perm,
                                                             const int32_t *__restrict__ leaf,
                                                             const unsigned char *__restrict__ Cpk,
                                                             const int32_t *__restrict__ cperm, int32_t K,
                                                             int32_t *__restrict__ hint) {
    // The CTA's slots mostly share one leaf (rows are grouped by leaf): that of its first
    // slot's row is staged in shared memory coordinate by coordinate (cs[u][kl], +inf
    // past the tile's codewords), so a pair of codewords' coordinate u is one 8-byte load.
    __shared__ __align__(16) float cs[D][256];
    const int64_t cta0 = (int64_t)blockIdx.x * blockDim.x * LS_ROWS;
    int gh = -1;
    {
        const int64_t r0 = perm[cta0];  // cta0 < n: the grid covers n slots
        if ((uint64_t)r0 < (uint64_t)n) gh = leaf[r0];
    }
    if (gh >= 0) {
        const float *cw = reinterpret_cast<const float *>(Cpk + (int64_t)gh * TC_TILE_BYTES + TC_TILE_H);
        const int cntw = min(256, K - gh * 256);
        for (int e = threadIdx.x; e < D * 256; e += blockDim.x) {
            const int kl = e / D, u = e - kl * D;  // coalesced reads of the tile's rows
            cs[u][kl] = kl < cntw ? __ldg(cw + e) : __int_as_float(0x7f800000);
        }
    }
    __syncthreads();
    const int64_t s0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * LS_ROWS;
    if (s0 >= n) return;
    int64_t row[LS_ROWS];
    int32_t g[LS_ROWS];
    bool same = true;
#pragma unroll
    for (int r = 0; r < LS_ROWS; ++r) {
        const int64_t s = s0 + r;
        row[r] = s < n ? perm[s] : -1;
        if ((uint64_t)row[r] >= (uint64_t)n) row[r] = -1;
        g[r] = row[r] >= 0 ? leaf[row[r]] : -1;
        same &= row[r] >= 0 && g[r] == g[0];
    }
    if (same) {
        // two codewords per packed fp32x2 operation (each half the scalar sequence)
        unsigned long long x2[LS_ROWS][D];
        float best[LS_ROWS];
        int bk[LS_ROWS];
#pragma unroll
        for (int r = 0; r < LS_ROWS; ++r) {
#pragma unroll
            for (int u = 0; u < D; ++u) {
                const float v = W[row[r] * D + u];
                x2[r][u] = pack2(v, v);
            }
            best[r] = __int_as_float(0x7f800000);
            bk[r] = 0;
        }
        const float *cw = reinterpret_cast<const float *>(Cpk + (int64_t)g[0] * TC_TILE_BYTES + TC_TILE_H);
        const int cntw = min(256, K - g[0] * 256);
        const bool staged = g[0] == gh;
        for (int kl = 0; kl < cntw; kl += 2) {
            const bool two = kl + 1 < cntw;  // an odd last codeword pairs with +inf (never chosen)
            unsigned long long c2[D];
            if (staged) {
#pragma unroll
                for (int u = 0; u < D; ++u) c2[u] = *reinterpret_cast<const unsigned long long *>(&cs[u][kl]);
            } else {
#pragma unroll
                for (int u = 0; u < D; ++u)
                    c2[u] = pack2(__ldg(cw + kl * D + u),
                                  two ? __ldg(cw + (kl + 1) * D + u) : __int_as_float(0x7f800000));
            }
#pragma unroll
            for (int r = 0; r < LS_ROWS; ++r) {
                unsigned long long t = sub2(x2[r][0], c2[0]);
                unsigned long long acc = mul2(t, t);
#pragma unroll
                for (int u = 1; u < D; ++u) {
                    t = sub2(x2[r][u], c2[u]);
                    acc = fma2(t, t, acc);
                }
                float d0, d1;
                unpack2(acc, d0, d1);
                if (d0 < best[r]) {
                    best[r] = d0;
                    bk[r] = kl;
                }
                if (d1 < best[r]) {
                    best[r] = d1;
                    bk[r] = kl + 1;
                }
            }
        }
#pragma unroll
        for (int r = 0; r < LS_ROWS; ++r) hint[row[r]] = cperm[g[0] * 256 + bk[r]];
        return;
    }
#pragma unroll
    for (int r = 0; r < LS_ROWS; ++r) {  // a leaf boundary or the end: row by row
        if (row[r] < 0) continue;
        float x[D];
#pragma unroll
        for (int u = 0; u < D; ++u) x[u] = W[row[r] * D + u];
        const float *cw = reinterpret_cast<const float *>(Cpk + (int64_t)g[r] * TC_TILE_BYTES + TC_TILE_H);
        const int cntw = min(256, K - g[r] * 256);
        float best = __int_as_float(0x7f800000);
        int bk = 0;
        for (int kl = 0; kl < cntw; ++kl) {
            float acc = 0.f;
#pragma unroll
            for (int u = 0; u < D; ++u) {
                const float t = x[u] - __ldg(cw + kl * D + u);
                acc = fmaf(t, t, acc);
            }
            if (acc < best) {
                best = acc;
                bk = kl;
            }
        }
        hint[row[r]] = cperm[g[r] * 256 + bk];
    }
}

int kd_levels(int32_t T) {
    int L = 0;
    while ((1 << L) < T) ++L;
    return L;
}

cudaError_t launch_codebook_order(const float *C, int32_t K, int32_t *cperm, int32_t *cpos, int32_t *tmp,
                                  unsigned long long *keys, KdNode *nodes, Header *hdr, cudaStream_t s) {
    const int32_t T = (K + 255) / 256;
    const int L = kd_levels(T);
    cudaError_t e = cudaMemsetAsync(&hdr->yy_cnorm, 0, sizeof(uint32_t), s);
    if (e != cudaSuccess) return e;
    const int32_t *src = nullptr;
    for (int l = 0; l < L; ++l) {
        int32_t *dst = ((L - 1 - l) % 2 == 0) ? cperm : tmp;  // the last level writes cperm
        launch_begin(s);
        kd_split_kernel<<<1u << l, KD_THREADS, 0, s>>>(C, K, T, l, src, dst, keys, nodes);
        launch_end(s, "kd_split_kernel");
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        src = dst;
    }
    launch_begin(s);
    kd_finish_kernel<<<(K + 255) / 256, 256, 0, s>>>(C, K, cperm, cpos, hdr, L == 0);
    launch_end(s, "kd_finish_kernel");
    return cudaGetLastError();
}

cudaError_t launch_kd_hints(const float *W, int64_t n, const KdNode *nodes, int32_t K, const float *Cpk,
                            const int32_t *cperm, int32_t *leaf, int32_t *cnt, int32_t *perm, int32_t *hint,
                            int num_sms, cudaStream_t s) {
    const int32_t T = (K + 255) / 256;
    const unsigned blocks = (unsigned)((n + 255) / 256);
    launch_begin(s);
    kd_leaf_kernel<<<blocks, 256, 0, s>>>(W, n, nodes, T, leaf);
    launch_end(s, "kd_leaf_kernel");
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // rows grouped by leaf tile (the leaf numbers stand in for hints over T "codewords")
    if ((e = launch_hint_permutation(leaf, n, T, nullptr, nullptr, nullptr, cnt, perm, num_sms, s)) != cudaSuccess)
        return e;
    launch_begin(s);
    kd_leaf_search_kernel<<<(unsigned)((n + 256 * LS_ROWS - 1) / (256 * LS_ROWS)), 256, 0, s>>>(
        W, n, perm, leaf, reinterpret_cast<const unsigned char *>(Cpk), cperm, K, hint);
    launch_end(s, "kd_leaf_search_kernel");
    return cudaGetLastError();
}

}  // namespace kq
