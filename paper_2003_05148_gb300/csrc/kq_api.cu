// kq_api.cu -- the extern "C" entry points of libkq declared in include/kq.h:
// argument validation, workspace carving and kernel sequencing. No device memory
// is allocated here; every buffer is the caller's or a slice of its workspace.
#include <stddef.h>

#include <atomic>
#include <cmath>
#include <mutex>
#include <unordered_map>
#include <unordered_set>
#include <vector>

#include "kq_internal.cuh"

using namespace kq;

namespace kq {
static std::atomic<unsigned long long> g_launches{0};

// Kernel trace (kq_trace_*): event pairs created up front, filled in launch order.
struct TraceRec {
    const char *name;
    cudaEvent_t begin, end;
};
static std::mutex g_trace_mu;
static std::vector<TraceRec> g_trace;
static size_t g_trace_used = 0;
static std::atomic<bool> g_trace_on{false};

void launch_begin(cudaStream_t s) {
    if (!g_trace_on.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lock(g_trace_mu);
    if (g_trace_on && g_trace_used < g_trace.size()) cudaEventRecord(g_trace[g_trace_used].begin, s);
}

void launch_end(cudaStream_t s, const char *name) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (!g_trace_on.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lock(g_trace_mu);
    if (g_trace_on && g_trace_used < g_trace.size()) {
        cudaEventRecord(g_trace[g_trace_used].end, s);
        g_trace[g_trace_used].name = name;
        ++g_trace_used;
    }
}
// Workspaces with test faults or a wait limit set (kq_test_inject_wait_fault).
static std::mutex g_hooks_mu;
static std::unordered_set<const void *> g_hooks;
bool test_hooks(const Header *hdr) {
    std::lock_guard<std::mutex> lock(g_hooks_mu);
    return !g_hooks.empty() && g_hooks.count(hdr) != 0;
}

// kq_test_inject_wait_fault: the header words that the bounded waits read.
__global__ void test_inject_kernel(Header *h, uint32_t faults, uint32_t limit) {
    h->test_faults = faults;
    h->test_wait_limit = limit;
}
}  // namespace kq

namespace {

constexpr int32_t KQ_ABI_VERSION = 7;
constexpr int32_t HINT_ORDER_MIN_K = 4096;  // warm starts in hint order from 16 codeword tiles on
// Cold assignments with many codeword tiles start from a pilot pass: rows against the
// first K / COLD_PILOT_DIV codewords (a random sample when the codebook was drawn from
// the kernels), whose answers then serve as warm-start hints for the full pass.
constexpr int32_t COLD_PILOT_MIN_K = 16384;
constexpr int32_t COLD_PILOT_DIV = 16;
constexpr double KD_HINT_MIN_PAIRS = 1e10;  // cold starts of at least this many kernel x codeword pairs: k-d hints

inline bool aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

inline kq_status cuda_status(cudaError_t e) { return e == cudaSuccess ? KQ_OK : KQ_ERR_CUDA; }

#define KQ_TRY(expr)                                  \
    do {                                              \
        cudaError_t e_ = (expr);                      \
        if (e_ != cudaSuccess) return KQ_ERR_CUDA;    \
    } while (0)

// Supported problem sizes (see kq.h, "Sizes").
inline bool sizes_ok(int64_t n, int32_t K) {
    return n >= 1 && n < (1LL << 31) && K >= 1 && (int64_t)K <= n && (int64_t)K * D < (1LL << 31);
}

// Entry points that only use the fixed 4 KiB header of the workspace.
kq_status check_ws_header(void *ws, size_t ws_bytes) {
    if (!ws) return KQ_ERR_WORKSPACE;
    if (!aligned(ws, 256)) return KQ_ERR_ALIGNMENT;
    if (ws_bytes < 4096) return KQ_ERR_WORKSPACE;
    return KQ_OK;
}

kq_status check_ws(void *ws, size_t ws_bytes, int64_t n, int32_t K) {
    if (!ws) return KQ_ERR_WORKSPACE;
    if (!aligned(ws, 256)) return KQ_ERR_ALIGNMENT;
    if (ws_bytes < ws_layout(n, K).total) return KQ_ERR_WORKSPACE;
    return KQ_OK;
}

kq_status num_sms(int *out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return KQ_ERR_CUDA;
    if (cudaDeviceGetAttribute(out, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return KQ_ERR_CUDA;
    return KQ_OK;
}

struct Ws {
    Header *hdr;
    float *cd;
    unsigned long long *acc;
    unsigned long long *part;
    double *blocksum;
    float *cbuf0, *cbuf1, *cp;
    unsigned long long *cq;
    float *cpk;
    float *dist;
    int32_t *perm, *pcnt, *prev;
    // pruned fit (yy_cap: the largest codebook the regions hold, 0 when absent)
    int32_t yy_cap;
    int32_t *cperm, *cpos, *kdtmp, *leaf;
    unsigned long long *kdkey;
    KdNode *nodes;
    float *tdrift, *ydist;
    unsigned char *yrec;
};

Ws carve(void *ws, int64_t n, int32_t K) {
    const WsLayout L = ws_layout(n, K);
    char *b = static_cast<char *>(ws);
    Ws w;
    w.hdr = reinterpret_cast<Header *>(b);
    w.cd = reinterpret_cast<float *>(b + L.cd);
    w.acc = reinterpret_cast<unsigned long long *>(b + L.acc);
    w.part = reinterpret_cast<unsigned long long *>(b + L.part);
    w.blocksum = reinterpret_cast<double *>(b + L.blocksum);
    w.cbuf0 = reinterpret_cast<float *>(b + L.cbuf0);
    w.cbuf1 = reinterpret_cast<float *>(b + L.cbuf1);
    w.cp = reinterpret_cast<float *>(b + L.cp);
    w.cq = reinterpret_cast<unsigned long long *>(b + L.cq);
    w.cpk = reinterpret_cast<float *>(b + L.cpk);
    w.dist = reinterpret_cast<float *>(b + L.dist);
    w.perm = reinterpret_cast<int32_t *>(b + L.perm);
    w.pcnt = reinterpret_cast<int32_t *>(b + L.pcnt);
    w.prev = reinterpret_cast<int32_t *>(b + L.prev);
    w.yy_cap = yy_sizes(K) ? K : 0;
    w.cperm = reinterpret_cast<int32_t *>(b + L.cperm);
    w.cpos = reinterpret_cast<int32_t *>(b + L.cpos);
    w.kdtmp = reinterpret_cast<int32_t *>(b + L.kdtmp);
    w.kdkey = reinterpret_cast<unsigned long long *>(b + L.kdkey);
    w.nodes = reinterpret_cast<KdNode *>(b + L.kdnode);
    w.tdrift = reinterpret_cast<float *>(b + L.tdrift);
    w.yrec = reinterpret_cast<unsigned char *>(b + L.yrec);
    w.ydist = reinterpret_cast<float *>(b + L.ydist);
    w.leaf = reinterpret_cast<int32_t *>(b + L.leaf);
    return w;
}

// One assignment, on the kernel tc_eligible picks. hint_counts: rows per hinted
// codeword, when known (the fit's previous update counted them), or null.
// packed: the workspace already holds C packed for the tensor cores (the fit's fused
// step for small codebooks packs each new codebook). sums: where the objective's block
// sums (w.blocksum) come from when the rows were processed in hint order: SUMS_NOW
// (dist_block_sums_kernel), SUMS_NONE (nobody reads them), or SUMS_DEFER (the caller
// sums *defer_dist itself; set to null when the block sums are already there).
enum BlockSums { SUMS_NOW, SUMS_NONE, SUMS_DEFER };
// normed: the packing bounds are cleared and C's largest norm is in place
// (launch_finalize_norm_tc).
kq_status run_assign(const float *W, int64_t n, const float *C, int32_t K, const int32_t *hint, int32_t *idx,
                     float *dist, int *nb, const Ws &w, int sms, cudaStream_t s, const int32_t *hint_counts = nullptr,
                     bool packed = false, BlockSums sums = SUMS_NOW, const float **defer_dist = nullptr,
                     bool normed = false) {
    if (defer_dist) *defer_dist = nullptr;
    if (tc_eligible(n, K, sms)) {
        // A cold start with many tiles gets hints, written into idx (each row's hint is
        // read before its own answer is written, by the same CTA): on large problems
        // (4096 to 65536 codewords, n K >= KD_HINT_MIN_PAIRS) each kernel's nearest
        // codeword in its leaf of a k-d tree over the codebook (kq_order.cu; the
        // workspace holds the tree), otherwise from 16384 codewords a pilot pass against
        // the first K / 16 codewords. (The tree costs about 0.4-1.2 ms: on ResNet-18's
        // 256 -> 256 layer, n = 65,536 and K = 16,384, it made the fit 12% slower; on
        // the 2048 x 2048 layer, 7% faster.)
        if (!hint && K <= w.yy_cap && yy_sizes(K) && (double)n * (double)K >= KD_HINT_MIN_PAIRS) {
            KQ_TRY(launch_codebook_order(C, K, w.cperm, w.cpos, w.kdtmp, w.kdkey, w.nodes, w.hdr, s));
            KQ_TRY(launch_pack_codebook_tc(C, K, w.cpk, w.hdr, s, w.cperm));
            KQ_TRY(launch_kd_hints(W, n, w.nodes, K, w.cpk, w.cperm, w.leaf, w.pcnt, w.perm, idx, sms, s));
            hint = idx;
            hint_counts = nullptr;
        }
        if (!packed) KQ_TRY(launch_pack_codebook_tc(C, K, w.cpk, w.hdr, s, nullptr, nullptr, nullptr, normed));
        if (!hint && K < COLD_PILOT_MIN_K) {
            // fewer codewords: each row seeded with the nearest of the first few (one
            // CUDA-core pass), instead of testing its whole first tile exactly
            KQ_TRY(launch_sample_hints(W, n, C, K < SAMPLE_HINT_MAX ? K : SAMPLE_HINT_MAX, idx, sms, s));
            hint = idx;
            hint_counts = nullptr;
        }
        if (!hint && K >= COLD_PILOT_MIN_K) {
            int nbp = 0;
            KQ_TRY(launch_assign_tc(W, n, C, w.cpk, K / COLD_PILOT_DIV, nullptr, nullptr, idx, nullptr, nullptr, &nbp,
                                    w.hdr, s));
            hint = idx;
            hint_counts = nullptr;
        }
        // Warm start with many codeword tiles: rows grouped by hint (see
        // kq_assign_tc.cu); the objective's block sums are then taken over the
        // distances in row order, whatever the grouping. With few tiles the four extra
        // launches cost more than they save, and rows stay in order.
        if (hint && K >= HINT_ORDER_MIN_K) {
            KQ_TRY(launch_hint_permutation(hint, n, K, nullptr, nullptr, hint_counts, w.pcnt, w.perm, sms, s));
            float *d = dist ? dist : w.dist;
            KQ_TRY(launch_assign_tc(W, n, C, w.cpk, K, hint, w.perm, idx, d, nullptr, nb, w.hdr, s));
            if (sums == SUMS_NOW) KQ_TRY(launch_dist_block_sums(d, n, w.blocksum, nb, s));
            if (sums == SUMS_DEFER) *defer_dist = d;
        } else {
            KQ_TRY(launch_assign_tc(W, n, C, w.cpk, K, hint, nullptr, idx, dist, w.blocksum, nb, w.hdr, s));
        }
    } else {
        KQ_TRY(launch_pack_codebook(C, K, w.cd, w.hdr, s));
        KQ_TRY(launch_assign(W, n, w.cd, C, K, hint, idx, dist, w.blocksum, nb, w.part, w.hdr, sms, s));
    }
    return KQ_OK;
}

// One assignment of a pruned fit (kq_assign_tc.cu, kq_order.cu): the codebook
// packed in k-d order, rows grouped by the codebook position of their hint, tiles
// ruled out by the rows' bound records. read: the records are those of the
// previous pass, whose codebook is Cprev (tile drifts from it); otherwise every
// tile is processed and the records are written fresh. Without a hint (the fit's
// first pass) the hints come from the k-d leaves, written into idx.
kq_status run_assign_pruned(const float *W, int64_t n, const float *C, int32_t K, const int32_t *hint, int32_t *idx,
                            int *nb, const Ws &w, int sms, cudaStream_t s, const int32_t *hint_counts,
                            const float *Cprev, bool read, BlockSums sums = SUMS_NOW,
                            const float **defer_dist = nullptr) {
    if (defer_dist) *defer_dist = nullptr;
    const TcYy st{w.cperm, w.cpos, w.tdrift, w.yrec, w.ydist, yy_stride(w.yy_cap), read ? 1 : 0};
    KQ_TRY(launch_pack_codebook_tc(C, K, w.cpk, w.hdr, s, w.cperm, read ? Cprev : nullptr,
                                   read ? w.tdrift : nullptr));
    if (!hint) {
        KQ_TRY(launch_kd_hints(W, n, w.nodes, K, w.cpk, w.cperm, w.leaf, w.pcnt, w.perm, idx, sms, s));
        hint = idx;
        hint_counts = nullptr;
    }
    KQ_TRY(launch_hint_permutation(hint, n, K, w.cpos, w.cperm, hint_counts, w.pcnt, w.perm, sms, s));
    KQ_TRY(launch_assign_tc(W, n, C, w.cpk, K, hint, w.perm, idx, w.dist, nullptr, nb, w.hdr, s, &st));
    if (sums == SUMS_NOW) KQ_TRY(launch_dist_block_sums(w.dist, n, w.blocksum, nb, s));
    if (sums == SUMS_DEFER) *defer_dist = w.dist;
    return KQ_OK;
}

// The k-means fit of kq_fit_codebook on carved workspace regions (sized for at
// least K codewords). objective: iters + 1 device doubles or null; final_obj: one
// device double receiving the objective of the final assignment, or null.
// stop_on_stable: after every incremental update, read on the host whether any row
// changed codeword; if none did, the fit is at a fixed point (the next update would
// rebuild the same codebook from the same sets, bit for bit, and every later
// assignment would repeat this one), so the outputs of the remaining iterations are
// written directly. iters_run (host, nullable): the codebook updates performed.
kq_status run_fit(const float *W, int64_t n, int32_t K, const float *C_init, int32_t iters, float *C_out,
                  int32_t *idx, int32_t *counts, double *objective, double *final_obj, const Ws &w, int sms,
                  cudaStream_t s, bool stop_on_stable = false, int32_t *iters_run = nullptr, bool prune = false) {
    const size_t cbytes = (size_t)K * D * sizeof(float);
    kq_status st;
    KQ_TRY(launch_update_prepare(nullptr, K, w.acc, w.hdr, false, s));
    KQ_TRY(launch_maxabs(W, n * D, &w.hdr->maxabs_bits, &w.hdr->status, sms, s));  // the scale, once per fit
    KQ_TRY(cudaMemcpyAsync(w.cbuf0, C_init, cbytes, cudaMemcpyDeviceToDevice, s));
    float *cur = w.cbuf0, *nxt = w.cbuf1;
    int nb = 0;
    // pruned assignments: the codebook's k-d order is taken once, from C_init
    const bool pruned = prune && K <= w.yy_cap && yy_sizes(K) && tc_eligible(n, K, sms);
    if (pruned) KQ_TRY(launch_codebook_order(cur, K, w.cperm, w.cpos, w.kdtmp, w.kdkey, w.nodes, w.hdr, s));
    // small codebooks on the tensor-core path: the objective's sum, the finalise and the
    // next codebook's packing in one launch per iteration
    const bool fused = !pruned && !stop_on_stable && tc_eligible(n, K, sms) && tc_pack_small(K);
    bool packed = false;  // cur is packed in the workspace
    // larger codebooks on the tensor-core path: the finalise also takes the new
    // codebook's largest norm (the packing's first step)
    const bool fnorm = !pruned && !stop_on_stable && tc_eligible(n, K, sms) && !tc_pack_small(K);
    bool normed = false;  // cur's largest norm is in place
    // the block sums of an assignment made in hint order: summed by the delta update
    // that follows it (one launch fewer), when the objective is wanted and that update runs
    const bool want_sums = objective || final_obj;
    const float *ddist = nullptr;  // the distances whose block sums the next delta update takes
    auto assign = [&](int32_t t, const int32_t *hint, int32_t *out, const int32_t *hint_counts) -> kq_status {
        const BlockSums bs = !want_sums ? SUMS_NONE : (t >= 1 && t < iters && !stop_on_stable) ? SUMS_DEFER : SUMS_NOW;
        if (pruned)
            return run_assign_pruned(W, n, cur, K, hint, out, &nb, w, sms, s, hint_counts, nxt, t > 0, bs, &ddist);
        return run_assign(W, n, cur, K, hint, out, nullptr, &nb, w, sms, s, hint_counts, packed, bs, &ddist, normed);
    };
    // Assignment t goes to idx when iters - t is even, else to the workspace's other
    // index buffer, so the final one lands in idx. Iteration t > 0 starts every row
    // from assignment t - 1 (warm start; the update wrote its cluster sizes), and its
    // update moves only the rows whose codeword changed (the sums stay in place).
    auto buf = [&](int32_t t) -> int32_t * { return ((iters - t) & 1) ? w.prev : idx; };
    for (int32_t t = 0; t < iters; ++t) {
        int32_t *out = buf(t);
        const int32_t *hint = t > 0 ? buf(t - 1) : nullptr;
        if ((st = assign(t, hint, out, t > 0 ? counts : nullptr)) != KQ_OK) return st;
        // the objective of assignment t: with the finalise below (one launch fewer), or
        // here when the fit may stop before it
        if (objective && stop_on_stable) KQ_TRY(launch_sum_blocks(w.blocksum, nb, objective + t, s));
        if (t == 0) {
            KQ_TRY(launch_accumulate(W, n, out, K, w.hdr, w.acc, false, sms, s));
        } else if (!stop_on_stable) {
            KQ_TRY(launch_accumulate_delta(W, n, hint, out, K, w.hdr, w.acc, sms, s, nullptr, ddist, w.blocksum, &nb));
        } else {
            KQ_TRY(cudaMemsetAsync(&w.hdr->fit_moved, 0, sizeof(uint32_t), s));
            KQ_TRY(launch_accumulate_delta(W, n, hint, out, K, w.hdr, w.acc, sms, s, &w.hdr->fit_moved));
            uint32_t moved = 1;
            KQ_TRY(cudaMemcpyAsync(&moved, &w.hdr->fit_moved, sizeof(moved), cudaMemcpyDeviceToHost, s));
            KQ_TRY(cudaStreamSynchronize(s));
            if (!moved) {  // assignment t repeats assignment t - 1: C_t is the fixed point
                if (out != idx) KQ_TRY(cudaMemcpyAsync(idx, out, (size_t)n * sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
                if (objective) KQ_TRY(launch_fill_objective(objective, t, iters, s));
                if (final_obj) KQ_TRY(launch_sum_blocks(w.blocksum, nb, final_obj, s));
                KQ_TRY(launch_histogram(idx, n, K, counts, &w.hdr->status, sms, s));
                KQ_TRY(cudaMemcpyAsync(C_out, cur, cbytes, cudaMemcpyDeviceToDevice, s));
                if (iters_run) *iters_run = t;
                return KQ_OK;
            }
        }
        if (fused) {
            KQ_TRY(launch_finalize_pack_small(w.blocksum, nb, objective ? objective + t : nullptr, w.acc, K, w.hdr, cur,
                                              nxt, counts, w.cpk, s));
            packed = true;
        } else if (fnorm) {
            KQ_TRY(launch_finalize_norm_tc(w.blocksum, nb, objective ? objective + t : nullptr, w.acc, K, w.hdr, cur,
                                           nxt, counts, s));
            normed = true;
        } else {
            KQ_TRY(launch_finalize(w.acc, K, w.hdr, cur, nxt, counts, s, true, w.blocksum, nb,
                                   objective && !stop_on_stable ? objective + t : nullptr));
        }
        float *tmp = cur;
        cur = nxt;
        nxt = tmp;
    }
    if ((st = assign(iters, iters > 0 ? buf(iters - 1) : nullptr, idx, iters > 0 ? counts : nullptr)) != KQ_OK)
        return st;
    if (objective) KQ_TRY(launch_sum_blocks(w.blocksum, nb, objective + iters, s));
    if (final_obj) KQ_TRY(launch_sum_blocks(w.blocksum, nb, final_obj, s));
    KQ_TRY(launch_histogram(idx, n, K, counts, &w.hdr->status, sms, s));
    KQ_TRY(cudaMemcpyAsync(C_out, cur, cbytes, cudaMemcpyDeviceToDevice, s));
    if (iters_run) *iters_run = iters;
    return KQ_OK;
}

// SplitMix64 finaliser (Steele, Lea and Flood, OOPSLA 2014).
uint64_t splitmix_mix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

int ceil_log2_i64(int64_t k) {
    int b = 0;
    while ((1LL << b) < k) ++b;
    return b;
}

}  // namespace

namespace kq {
kq_status quantize_codebook(const float *C, int32_t K, const int32_t *counts, int32_t max_iters, float *levels,
                            uint8_t *codes, int32_t *iters_run, void *ws, size_t ws_bytes, cudaStream_t s,
                            bool shared_gpu) {
    if (K < 1 || (int64_t)K * D >= (1LL << 31) || !C || !counts || !levels || !codes) return KQ_ERR_INVALID_ARG;
    if (max_iters < 0 || max_iters > 100000) return KQ_ERR_INVALID_ARG;
    if (!aligned(C, 4) || !aligned(counts, 4) || !aligned(levels, 4) || !aligned(iters_run, 4))
        return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws_header(ws, ws_bytes);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    Header *h = static_cast<Header *>(ws);
    return cuda_status(
        launch_level_fit(C, (int64_t)K * D, counts, max_iters, levels, codes, iters_run, h, sms, s, shared_gpu));
}
}  // namespace kq

extern "C" {

const char *kq_status_string(kq_status s) {
    switch (s) {
        case KQ_OK: return "KQ_OK";
        case KQ_ERR_INVALID_ARG: return "KQ_ERR_INVALID_ARG";
        case KQ_ERR_ALIGNMENT: return "KQ_ERR_ALIGNMENT";
        case KQ_ERR_NONFINITE: return "KQ_ERR_NONFINITE";
        case KQ_ERR_CUDA: return "KQ_ERR_CUDA";
        case KQ_ERR_DEVICE_CHECK: return "KQ_ERR_DEVICE_CHECK";
        case KQ_ERR_WORKSPACE: return "KQ_ERR_WORKSPACE";
        case KQ_ERR_TIMEOUT: return "KQ_ERR_TIMEOUT";
    }
    return "KQ_ERR_UNKNOWN";
}

int32_t kq_abi_version(void) { return KQ_ABI_VERSION; }

uint64_t kq_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

kq_status kq_trace_start(int32_t capacity) {
    if (capacity < 1 || capacity > (1 << 20)) return KQ_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> lock(g_trace_mu);
    g_trace_on = false;
    // events belong to the device current when they were made: remake them all
    for (TraceRec &r : g_trace) {
        cudaEventDestroy(r.begin);
        cudaEventDestroy(r.end);
    }
    g_trace.clear();
    g_trace_used = 0;
    g_trace.reserve((size_t)capacity);
    for (int32_t i = 0; i < capacity; ++i) {
        TraceRec r{nullptr, nullptr, nullptr};
        if (cudaEventCreate(&r.begin) != cudaSuccess) return KQ_ERR_CUDA;
        if (cudaEventCreate(&r.end) != cudaSuccess) {
            cudaEventDestroy(r.begin);
            return KQ_ERR_CUDA;
        }
        g_trace.push_back(r);
    }
    g_trace_on = true;
    return KQ_OK;
}

kq_status kq_trace_stop(void) {
    std::lock_guard<std::mutex> lock(g_trace_mu);
    g_trace_on = false;
    return KQ_OK;
}

int32_t kq_trace_count(void) {
    std::lock_guard<std::mutex> lock(g_trace_mu);
    return (int32_t)g_trace_used;
}

kq_status kq_trace_get(int32_t i, const char **name, float *ms) {
    std::lock_guard<std::mutex> lock(g_trace_mu);
    if (i < 0 || (size_t)i >= g_trace_used || !name || !ms) return KQ_ERR_INVALID_ARG;
    const TraceRec &r = g_trace[(size_t)i];
    if (cudaEventSynchronize(r.end) != cudaSuccess) return KQ_ERR_CUDA;
    if (cudaEventElapsedTime(ms, r.begin, r.end) != cudaSuccess) return KQ_ERR_CUDA;
    *name = r.name;
    return KQ_OK;
}

size_t kq_workspace_bytes(int64_t n, int32_t K) {
    if (!sizes_ok(n, K)) return 0;
    return ws_layout(n, K).total;
}

kq_status kq_device_status(void *ws, size_t ws_bytes, kq_stream_t stream, uint32_t *flags_out) {
    if (!ws) return KQ_ERR_WORKSPACE;
    if (!aligned(ws, 256)) return KQ_ERR_ALIGNMENT;
    if (ws_bytes < sizeof(Header)) return KQ_ERR_WORKSPACE;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Header *h = static_cast<Header *>(ws);
    uint32_t flags = 0;
    KQ_TRY(cudaMemcpyAsync(&flags, &h->status, sizeof(flags), cudaMemcpyDeviceToHost, s));
    KQ_TRY(cudaMemsetAsync(&h->status, 0, sizeof(uint32_t), s));
    KQ_TRY(cudaStreamSynchronize(s));
    if (flags_out) *flags_out = flags;
    if (flags & KQ_FLAG_TIMEOUT) return KQ_ERR_TIMEOUT;
    if (flags & (KQ_FLAG_INDEX_RANGE | KQ_FLAG_CODE_RANGE)) return KQ_ERR_DEVICE_CHECK;
    if (flags & KQ_FLAG_NONFINITE) return KQ_ERR_NONFINITE;
    return KQ_OK;
}

kq_status kq_fit_prune_stats(void *ws, size_t ws_bytes, uint64_t *tiles_run, uint64_t *tiles_all,
                             kq_stream_t stream) {
    if (!tiles_run || !tiles_all) return KQ_ERR_INVALID_ARG;
    kq_status st = check_ws_header(ws, ws_bytes);
    if (st != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Header *h = static_cast<Header *>(ws);
    unsigned long long v[2] = {0ull, 0ull};  // yy_tiles_run, yy_tiles_all (adjacent)
    KQ_TRY(cudaMemcpyAsync(v, &h->yy_tiles_run, sizeof(v), cudaMemcpyDeviceToHost, s));
    KQ_TRY(cudaStreamSynchronize(s));
    *tiles_run = v[0];
    *tiles_all = v[1];
    return KQ_OK;
}

kq_status kq_test_inject_wait_fault(void *ws, size_t ws_bytes, uint32_t faults, uint32_t wait_limit,
                                    kq_stream_t stream) {
    if ((faults & ~(KQ_TEST_SKIP_ARRIVAL | KQ_TEST_STOP_TILE_STREAM)) != 0u) return KQ_ERR_INVALID_ARG;
    kq_status st = check_ws_header(ws, ws_bytes);
    if (st != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    {
        std::lock_guard<std::mutex> lock(g_hooks_mu);
        if (faults != 0u || wait_limit != 0u)
            g_hooks.insert(ws);
        else
            g_hooks.erase(ws);
    }
    launch_begin(s);
    test_inject_kernel<<<1, 1, 0, s>>>(static_cast<Header *>(ws), faults, wait_limit);
    launch_end(s, "test_inject_kernel");
    return cuda_status(cudaGetLastError());
}

kq_status kq_init_codebook(const float *W, int64_t n, const int64_t *sel, int32_t K, float *C0, void *ws,
                           size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !W || !sel || !C0) return KQ_ERR_INVALID_ARG;
    if (!aligned(W, 4) || !aligned(sel, 8) || !aligned(C0, 4)) return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws_header(ws, ws_bytes);
    if (st != KQ_OK) return st;
    Header *h = static_cast<Header *>(ws);
    return cuda_status(launch_init_codebook(W, n, sel, K, C0, &h->status, reinterpret_cast<cudaStream_t>(stream)));
}

kq_status kq_assign(const float *W, int64_t n, const float *C, int32_t K, const int32_t *hint, int32_t *idx,
                    float *dist, void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !W || !C || !idx) return KQ_ERR_INVALID_ARG;
    if (!aligned(W, 16) || !aligned(C, 4) || !aligned(idx, 4) || !aligned(dist, 4) || !aligned(hint, 4))
        return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws(ws, ws_bytes, n, K);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Ws w = carve(ws, n, K);
    int nb = 0;
    return run_assign(W, n, C, K, hint, idx, dist, &nb, w, sms, s, nullptr, false, SUMS_NONE);  // no objective out
}

kq_status kq_update_centroids(const float *W, int64_t n, const int32_t *idx, int32_t K, const float *C_prev,
                              float *C_next, int32_t *counts, void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !W || !idx || !C_prev || !C_next || !counts) return KQ_ERR_INVALID_ARG;
    if (!aligned(W, 16) || !aligned(idx, 4) || !aligned(C_prev, 4) || !aligned(C_next, 4) || !aligned(counts, 4))
        return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws(ws, ws_bytes, n, K);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Ws w = carve(ws, n, K);
    // scale guessed from C_prev, checked on every value, exact fallback if violated
    KQ_TRY(launch_update_prepare(C_prev, K, w.acc, w.hdr, true, s));
    KQ_TRY(launch_accumulate(W, n, idx, K, w.hdr, w.acc, true, sms, s));
    KQ_TRY(launch_update_fallback(W, n, idx, K, w.hdr, w.acc, sms, s));
    KQ_TRY(launch_finalize(w.acc, K, w.hdr, C_prev, C_next, counts, s));
    return KQ_OK;
}

kq_status kq_fit_codebook(const float *W, int64_t n, int32_t K, const float *C_init, int32_t iters, int32_t flags,
                          float *C_out, int32_t *idx, int32_t *counts, double *objective, int32_t *iters_run,
                          void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !W || !C_init || !C_out || !idx || !counts) return KQ_ERR_INVALID_ARG;
    if (iters < 0 || (flags & ~(KQ_STOP_ON_STABLE | KQ_FIT_PRUNE)) != 0) return KQ_ERR_INVALID_ARG;
    if (!aligned(W, 16) || !aligned(C_init, 4) || !aligned(C_out, 4) || !aligned(idx, 4) || !aligned(counts, 4) ||
        !aligned(objective, 8))
        return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws(ws, ws_bytes, n, K);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const Ws w = carve(ws, n, K);
    const bool stop = (flags & KQ_STOP_ON_STABLE) != 0;
    if (flags & KQ_FIT_PRUNE)  // the pruned passes' work counters (kq_fit_prune_stats)
        KQ_TRY(cudaMemsetAsync(&w.hdr->yy_tiles_run, 0, 2 * sizeof(unsigned long long), s));
    if (small_fit_eligible(n, K)) {  // the whole fit in one cooperative launch
        const int nblk = (int)((n + 255) / 256) + MAX_PART_BLOCKS;
        KQ_TRY(launch_small_fit(W, n, C_init, K, iters, C_out, idx, counts, objective, w.acc, w.cbuf0, w.cbuf1,
                                w.blocksum, nblk, w.hdr, sms, s, stop));
        if (iters_run && stop) {  // the iteration count is on the device
            int32_t run = iters;
            KQ_TRY(cudaMemcpyAsync(&run, &w.hdr->fit_iters, sizeof(run), cudaMemcpyDeviceToHost, s));
            KQ_TRY(cudaStreamSynchronize(s));
            *iters_run = run;
        } else if (iters_run) {
            *iters_run = iters;
        }
        return KQ_OK;
    }
    return run_fit(W, n, K, C_init, iters, C_out, idx, counts, objective, nullptr, w, sms, s, stop, iters_run,
                   (flags & KQ_FIT_PRUNE) != 0);
}

kq_status kq_search_codebook_size(const float *W, int64_t n, const int64_t *sel, int32_t sel_len, double alpha,
                                  double r, int32_t max_steps, int32_t lloyd_iters, float *C_out, int32_t *idx,
                                  int32_t *counts, int32_t *K_out, double *err_out, int32_t *trace_K,
                                  double *trace_err, int32_t *steps_run, void *ws, size_t ws_bytes,
                                  kq_stream_t stream) {
    if (n < 1 || n >= (1LL << 31) || !W || !sel || !C_out || !idx || !counts || !K_out) return KQ_ERR_INVALID_ARG;
    if (!(alpha > 0.0) || !(alpha <= 1e9) || !(r >= 0.0) || !(r <= 1e9)) return KQ_ERR_INVALID_ARG;
    if (max_steps < 0 || max_steps > 64 || lloyd_iters < 0 || lloyd_iters > 100000) return KQ_ERR_INVALID_ARG;
    int64_t n_init = (int64_t)std::floor(alpha * (double)n);  // Algorithm 1: N_init = alpha * n
    if (n_init < 1) n_init = 1;
    if (n_init > n) n_init = n;
    if (!sizes_ok(n, (int32_t)n_init) || sel_len < n_init) return KQ_ERR_INVALID_ARG;
    if (!aligned(W, 16) || !aligned(sel, 8) || !aligned(C_out, 4) || !aligned(idx, 4) || !aligned(counts, 4))
        return KQ_ERR_ALIGNMENT;
    const int32_t N0 = (int32_t)n_init;
    kq_status st = check_ws(ws, ws_bytes, n, N0);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const Ws w = carve(ws, n, N0);  // every region sized for the largest codebook tried
    // J_0 = sum |W_i|^2: the objective against the single zero codeword
    KQ_TRY(cudaMemsetAsync(C_out, 0, D * sizeof(float), s));
    if ((st = run_fit(W, n, 1, C_out, 0, C_out, idx, counts, nullptr, &w.hdr->obj, w, sms, s)) != KQ_OK) return st;
    double J0 = 0.0;
    KQ_TRY(cudaMemcpyAsync(&J0, &w.hdr->obj, sizeof(double), cudaMemcpyDeviceToHost, s));
    KQ_TRY(cudaStreamSynchronize(s));
    int32_t last_fit = 0;
    // accuracy of a codebook of k entries: -(relative l2 reconstruction error)
    auto accuracy_of = [&](int32_t k, double *acc) -> kq_status {
        KQ_TRY(launch_init_codebook(W, n, sel, k, C_out, &w.hdr->status, s));
        kq_status e = run_fit(W, n, k, C_out, lloyd_iters, C_out, idx, counts, nullptr, &w.hdr->obj, w, sms, s);
        if (e != KQ_OK) return e;
        double J = 0.0;
        KQ_TRY(cudaMemcpyAsync(&J, &w.hdr->obj, sizeof(double), cudaMemcpyDeviceToHost, s));
        KQ_TRY(cudaStreamSynchronize(s));
        last_fit = k;
        *acc = J0 > 0.0 ? -std::sqrt(J / J0) : 0.0;
        return KQ_OK;
    };
    double a_base = 0.0;
    if ((st = accuracy_of(N0, &a_base)) != KQ_OK) return st;
    const double a_ori = 0.0;                              // the unquantised layer: no error
    const double a_target = a_base - (a_ori - a_base) * r;  // Eq. 3
    if (trace_K) trace_K[0] = N0;
    if (trace_err) trace_err[0] = -a_base;
    int32_t b_up = N0, b_lo = 0, steps = 0;
    double a_up = a_base;  // accuracy at b_up
    while (steps < max_steps && b_up - b_lo > 1) {
        ++steps;
        const int32_t k = (int32_t)(((int64_t)b_up + b_lo) / 2);
        double a = 0.0;
        if ((st = accuracy_of(k, &a)) != KQ_OK) return st;
        if (trace_K) trace_K[steps] = k;
        if (trace_err) trace_err[steps] = -a;
        if (a > a_target) {
            b_up = k;
            a_up = a;
        } else {
            b_lo = k;
        }
        if (a == a_target) break;
    }
    // leave the fit of the chosen size in C_out / idx / counts
    if (last_fit != b_up) {
        double a = 0.0;
        if ((st = accuracy_of(b_up, &a)) != KQ_OK) return st;
    }
    *K_out = b_up;
    if (err_out) *err_out = -a_up;
    if (steps_run) *steps_run = steps;
    return KQ_OK;
}

kq_status kq_quantize_codebook_6bit(const float *C, int32_t K, const int32_t *counts, int32_t max_iters,
                                    float *levels, uint8_t *codes, int32_t *iters_run, void *ws, size_t ws_bytes,
                                    kq_stream_t stream) {
    return quantize_codebook(C, K, counts, max_iters, levels, codes, iters_run, ws, ws_bytes,
                             reinterpret_cast<cudaStream_t>(stream), false);
}

kq_status kq_quantize_scalars_6bit(const float *v, int64_t m, int32_t max_iters, float *levels, uint8_t *codes,
                                   int32_t *iters_run, void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (m < 1 || m > (1LL << 40) || !v || !levels || !codes) return KQ_ERR_INVALID_ARG;
    if (max_iters < 0 || max_iters > 100000) return KQ_ERR_INVALID_ARG;
    if (!aligned(v, 4) || !aligned(levels, 4) || !aligned(iters_run, 4)) return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws_header(ws, ws_bytes);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    Header *h = static_cast<Header *>(ws);
    return cuda_status(launch_level_fit(v, m, nullptr, max_iters, levels, codes, iters_run, h, sms,
                                        reinterpret_cast<cudaStream_t>(stream)));
}

kq_status kq_codebook_grad_step(const float *G, int64_t n, const int32_t *idx, int32_t K, float lr, const float *C,
                                float *C_next, int32_t *counts, void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !G || !idx || !C || !C_next || !counts) return KQ_ERR_INVALID_ARG;
    if (!(lr == lr) || lr > 3.402823466e38f || lr < -3.402823466e38f) return KQ_ERR_INVALID_ARG;
    if (!aligned(G, 16) || !aligned(idx, 4) || !aligned(C, 4) || !aligned(C_next, 4) || !aligned(counts, 4))
        return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws(ws, ws_bytes, n, K);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Ws w = carve(ws, n, K);
    // exact mode of the update: the scale from max|G|, the sums of the gradients
    KQ_TRY(launch_update_prepare(nullptr, K, w.acc, w.hdr, false, s));
    KQ_TRY(launch_maxabs(G, n * D, &w.hdr->maxabs_bits, &w.hdr->status, sms, s));
    KQ_TRY(launch_accumulate(G, n, idx, K, w.hdr, w.acc, false, sms, s));
    KQ_TRY(launch_grad_finalize(w.acc, K, w.hdr, lr, C, C_next, counts, s));
    return KQ_OK;
}

kq_status kq_levels_grad_step(const float *G, int64_t n, const int32_t *idx, int32_t K, const uint8_t *codes,
                              float lr, const float *levels, float *levels_next, int64_t *counts, void *ws,
                              size_t ws_bytes, kq_stream_t stream) {
    if (n < 1 || n >= (1LL << 31) || K < 1 || (int64_t)K * D >= (1LL << 31)) return KQ_ERR_INVALID_ARG;
    if (!G || !idx || !codes || !levels || !levels_next) return KQ_ERR_INVALID_ARG;
    if (!(lr == lr) || lr > 3.402823466e38f || lr < -3.402823466e38f) return KQ_ERR_INVALID_ARG;
    if (!aligned(G, 16) || !aligned(idx, 4) || !aligned(levels, 4) || !aligned(levels_next, 4) ||
        !aligned(counts, 8))
        return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws_header(ws, ws_bytes);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Header *h = static_cast<Header *>(ws);
    KQ_TRY(launch_maxabs(G, n * D, &h->maxabs_bits, &h->status, sms, s));
    KQ_TRY(launch_level_grad(G, n, idx, K, codes, lr, levels, levels_next, counts, h, sms, s));
    return KQ_OK;
}

kq_status kq_reconstruct(const int32_t *idx, int64_t n, const float *C, int32_t K, const uint8_t *codes,
                         const float *levels, float *W_out, void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !idx || !W_out) return KQ_ERR_INVALID_ARG;
    if ((codes == nullptr) != (levels == nullptr)) return KQ_ERR_INVALID_ARG;
    if (!codes && !C) return KQ_ERR_INVALID_ARG;
    if (!aligned(idx, 4) || !aligned(C, 4) || !aligned(levels, 4) || !aligned(W_out, 16)) return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws(ws, ws_bytes, n, K);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Ws w = carve(ws, n, K);
    KQ_TRY(launch_decode_codebook(C, K, codes, w.cp, w.cq, &w.hdr->status, s));
    KQ_TRY(launch_gather_rows(idx, n, codes ? nullptr : w.cp, codes ? w.cq : nullptr, levels, K, W_out,
                              &w.hdr->status, sms, s));
    return KQ_OK;
}

kq_status kq_quantize_reconstruct(const int32_t *idx, int64_t n, const float *C, int32_t K, const float *levels,
                                  uint8_t *codes, float *W_out, void *ws, size_t ws_bytes, kq_stream_t stream) {
    if (!sizes_ok(n, K) || !idx || !C || !levels || !W_out) return KQ_ERR_INVALID_ARG;
    if (!aligned(idx, 4) || !aligned(C, 4) || !aligned(levels, 4) || !aligned(W_out, 16)) return KQ_ERR_ALIGNMENT;
    kq_status st = check_ws(ws, ws_bytes, n, K);
    if (st != KQ_OK) return st;
    int sms = 0;
    if ((st = num_sms(&sms)) != KQ_OK) return st;
    Ws w = carve(ws, n, K);
    return cuda_status(launch_encode_gather(C, K, levels, codes, w.cq, idx, n, W_out, w.hdr, sms,
                                            reinterpret_cast<cudaStream_t>(stream)));
}

kq_status kq_seed_indices(int64_t n, int32_t K, uint64_t seed, int64_t *out) {
    if (!out || n < 1 || n >= (1LL << 31) || K < 1 || (int64_t)K > n) return KQ_ERR_INVALID_ARG;
    const uint64_t golden = 0x9E3779B97F4A7C15ull;
    const uint64_t key = splitmix_mix(seed * 0x100000001B3ull + 4u);  // the initial-selection stream
    // positions below K live in out; the few larger positions a swap touched, in a map
    std::unordered_map<int64_t, int64_t> far;
    far.reserve((size_t)(n - K < K ? n - K : K));  // at most one entry per step, none past n
    for (int32_t j = 0; j < K; ++j) out[j] = j;
    auto get = [&](int64_t p) -> int64_t {
        if (p < K) return out[p];
        const auto it = far.find(p);
        return it == far.end() ? p : it->second;
    };
    for (int32_t j = 0; j < K; ++j) {
        const uint64_t u = splitmix_mix(key + (uint64_t)(j + 1) * golden);
        const int64_t r = j + (int64_t)(u % (uint64_t)(n - j));
        const int64_t vj = out[j], vr = get(r);
        if (r < K)
            out[r] = vj;
        else
            far[r] = vj;
        out[j] = vr;
    }
    return KQ_OK;
}

kq_status kq_compression_report(int64_t n, int32_t k, int32_t omega, int32_t b_c, kq_report *out) {
    if (n < 1 || k < 1 || omega < 1 || b_c < 1 || !out) return KQ_ERR_INVALID_ARG;
    const int64_t w2 = (int64_t)omega * omega;
    if (n > (1LL << 40) || w2 > (1LL << 20)) return KQ_ERR_INVALID_ARG;
    out->index_bits = n * ceil_log2_i64(k);
    out->codebook_bits = (int64_t)k * w2 * b_c;
    out->total_bits = out->index_bits + out->codebook_bits;
    out->beta = (double)out->total_bits / (double)(n * w2);
    out->ratio_kq = (double)(n * w2 * 32) / (double)out->total_bits;
    out->ratio_con_1bit = (double)(n * w2 * 32) / (double)(2 * 32 + n * w2);  // Eq. 5, u = 2, b_1 = 32
    return KQ_OK;
}

kq_status kq_conventional_ratio(int64_t n, int32_t omega, int32_t u, int32_t b_1, int32_t b_fp, double *out) {
    if (n < 1 || omega < 1 || u < 2 || b_1 < 1 || b_fp < 1 || !out) return KQ_ERR_INVALID_ARG;
    const int64_t w2 = (int64_t)omega * omega;
    if (n > (1LL << 40) || w2 > (1LL << 20)) return KQ_ERR_INVALID_ARG;
    *out = (double)(n * w2 * b_fp) / (double)((int64_t)u * b_1 + n * w2 * ceil_log2_i64(u));
    return KQ_OK;
}

}  // extern "C"
