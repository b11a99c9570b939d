// kq_group.cu -- kq_fit_layers: the per-layer pipeline of Sec. 3.1-3.2 (init,
// k-means fit, 6-bit codebook quantisation, K+C recovery) for all layers of a
// network in one call.
//
// The layers are independent problems. Each job runs through the same entry
// points as a single-layer caller would use (so the results are those calls'
// results, bit for bit), on one of up to GROUP_STREAMS internal streams of the
// current device: the jobs are dealt largest first to the least-loaded stream
// (longest-processing-time order, cost ~ (iters + 1) (n K + c), c standing for a
// layer's fixed per-iteration cost of launches and small grids), every used
// stream first waits for an event recorded on the caller's stream, and the
// caller's stream finally waits for an event recorded on each used stream. The
// streams and events are created once per device and kept; enqueueing holds a
// mutex, so calls from several host threads interleave whole.
#include <algorithm>
#include <mutex>
#include <vector>

#include "kq_internal.cuh"

namespace kq {
namespace {

constexpr int GROUP_STREAMS = 8;
constexpr double GROUP_FIXED_PAIRS = 1e9;  // per-iteration cost of a small layer, in kernel x codeword pairs

struct GroupPool {
    int device = -1;
    cudaStream_t s[GROUP_STREAMS] = {};
    cudaEvent_t fork = nullptr;
    cudaEvent_t join[GROUP_STREAMS] = {};
};

std::mutex g_group_mu;
std::vector<GroupPool *> g_group_pools;  // one per device, never freed (the streams outlive every call)

cudaError_t group_pool(int device, GroupPool **out) {
    for (GroupPool *p : g_group_pools)
        if (p->device == device) {
            *out = p;
            return cudaSuccess;
        }
    GroupPool *p = new GroupPool();
    p->device = device;
    cudaError_t e = cudaEventCreateWithFlags(&p->fork, cudaEventDisableTiming);
    for (int i = 0; e == cudaSuccess && i < GROUP_STREAMS; ++i) {
        e = cudaStreamCreateWithFlags(&p->s[i], cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->join[i], cudaEventDisableTiming);
    }
    if (e != cudaSuccess) {  // release what was made; the next call tries again
        for (int i = 0; i < GROUP_STREAMS; ++i) {
            if (p->s[i]) cudaStreamDestroy(p->s[i]);
            if (p->join[i]) cudaEventDestroy(p->join[i]);
        }
        if (p->fork) cudaEventDestroy(p->fork);
        delete p;
        return e;
    }
    g_group_pools.push_back(p);
    *out = p;
    return cudaSuccess;
}

// The host-side checks of one job (sizes, presence, output combinations); the
// entry points it calls check alignment and the workspace themselves.
bool job_ok(const kq_layer_job &j) {
    if (!j.W || !j.C || !j.idx || !j.counts || !j.ws || j.n < 1 || j.K < 1 || (int64_t)j.K > j.n) return false;
    if ((j.levels == nullptr) != (j.codes == nullptr)) return false;
    if (j.W_out && !j.codes) return false;
    return true;
}

}  // namespace
}  // namespace kq

using namespace kq;

extern "C" kq_status kq_fit_layers(const kq_layer_job *jobs, int32_t count, int32_t iters, int32_t level_iters,
                                   int32_t flags, kq_stream_t stream) {
    if (!jobs || count < 1 || iters < 0 || level_iters < 0 || level_iters > 100000) return KQ_ERR_INVALID_ARG;
    if ((flags & ~KQ_FIT_PRUNE) != 0) return KQ_ERR_INVALID_ARG;
    for (int32_t i = 0; i < count; ++i) {
        if (!job_ok(jobs[i])) return KQ_ERR_INVALID_ARG;
        for (int32_t j = 0; j < i; ++j)
            if (jobs[j].ws == jobs[i].ws) return KQ_ERR_INVALID_ARG;  // one workspace per concurrent call
    }

    // largest first, each to the least-loaded stream
    std::vector<int32_t> order((size_t)count);
    std::vector<double> cost((size_t)count);
    for (int32_t i = 0; i < count; ++i) {
        order[(size_t)i] = i;
        cost[(size_t)i] = (iters + 1.0) * ((double)jobs[i].n * (double)jobs[i].K + GROUP_FIXED_PAIRS);
    }
    std::stable_sort(order.begin(), order.end(), [&](int32_t a, int32_t b) { return cost[(size_t)a] > cost[(size_t)b]; });
    const int nstreams = count < GROUP_STREAMS ? (int)count : GROUP_STREAMS;
    std::vector<int> lane((size_t)count);
    double load[GROUP_STREAMS] = {};
    for (int32_t i : order) {
        int best = 0;
        for (int s = 1; s < nstreams; ++s)
            if (load[s] < load[best]) best = s;
        lane[(size_t)i] = best;
        load[best] += cost[(size_t)i];
    }

    std::lock_guard<std::mutex> lock(g_group_mu);
    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess) return KQ_ERR_CUDA;
    GroupPool *pool = nullptr;
    if (group_pool(device, &pool) != cudaSuccess) return KQ_ERR_CUDA;
    cudaStream_t caller = reinterpret_cast<cudaStream_t>(stream);
    if (cudaEventRecord(pool->fork, caller) != cudaSuccess) return KQ_ERR_CUDA;
    int forked = 0;
    kq_status st = KQ_OK;
    for (; forked < nstreams; ++forked)
        if (cudaStreamWaitEvent(pool->s[forked], pool->fork, 0) != cudaSuccess) {
            st = KQ_ERR_CUDA;
            break;
        }
    for (int32_t i : order) {
        if (st != KQ_OK) break;
        const kq_layer_job &j = jobs[i];
        const int li = lane[(size_t)i];
        if (li >= forked) {
            st = KQ_ERR_CUDA;
            break;
        }
        kq_stream_t ls = reinterpret_cast<kq_stream_t>(pool->s[li]);
        if (j.sel) st = kq_init_codebook(j.W, j.n, j.sel, j.K, j.C, j.ws, j.ws_bytes, ls);
        if (st == KQ_OK)
            st = kq_fit_codebook(j.W, j.n, j.K, j.C, iters, flags, j.C, j.idx, j.counts, j.objective, nullptr, j.ws,
                                 j.ws_bytes, ls);
        if (st == KQ_OK && j.codes)  // (the one-cluster level fit where it fits: other layers run beside it)
            st = quantize_codebook(j.C, j.K, j.counts, level_iters, j.levels, j.codes, nullptr, j.ws, j.ws_bytes,
                                   pool->s[li], true);
        if (st == KQ_OK && j.W_out)
            st = kq_reconstruct(j.idx, j.n, nullptr, j.K, j.codes, j.levels, j.W_out, j.ws, j.ws_bytes, ls);
    }
    // join every forked stream back into the caller's stream, whatever happened
    for (int s = 0; s < forked; ++s) {
        if (cudaEventRecord(pool->join[s], pool->s[s]) != cudaSuccess ||
            cudaStreamWaitEvent(caller, pool->join[s], 0) != cudaSuccess)
            if (st == KQ_OK) st = KQ_ERR_CUDA;
    }
    return st;
}
