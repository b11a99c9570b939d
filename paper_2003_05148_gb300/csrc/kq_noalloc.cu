// kq_noalloc.cu -- kq_assign_noalloc: the assignment step for callers that cannot
// allocate device memory, so cannot hand libkq a workspace.
//
// Its scratch (packed codebook, split-K partials, per-CTA sums, status word) lives
// in one file-scope __device__ array of fixed size. Every GPU that loads libkq
// holds that array until the process exits. In host code the array's name is
// only a host-side stand-in for the symbol, never a device address: the device
// address is fetched once per device with cudaGetSymbolAddress (with that device
// current) and cached; that first call on a device does this set-up.
//
// All calls on one device share the array and it keeps the last call's contents;
// two calls whose work overlaps on the GPU race on it.
#include <mutex>

#include "kq_internal.cuh"

using namespace kq;

namespace {

constexpr int64_t NOALLOC_MAX_N = 1LL << 24;  // 16,777,216 kernels
constexpr int32_t NOALLOC_MAX_K = 65536;       // codewords

// Byte offsets inside the scratch array (a workspace header comes first).
constexpr size_t SCR_HEADER = 0;
constexpr size_t SCR_CD = 4096;
constexpr size_t SCR_PART = SCR_CD + (size_t)NOALLOC_MAX_K * CD_FLOATS * sizeof(float);
constexpr size_t SCR_BLOCKSUM = SCR_PART + (size_t)MAX_PART_BLOCKS * ROW_BLOCK * sizeof(unsigned long long);
constexpr size_t SCR_BYTES =
    SCR_BLOCKSUM + (size_t)((NOALLOC_MAX_N + 255) / 256 + MAX_PART_BLOCKS) * sizeof(double);  // ~9.97 MB

constexpr int MAX_DEVICES = 64;
std::mutex g_mu;
void *g_scratch_ptr[MAX_DEVICES] = {};

}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[SCR_BYTES];

namespace {

// Device address of the scratch array on the current device (set up once per device).
kq_status scratch_for_current_device(char **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return KQ_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_ptr[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return KQ_ERR_CUDA;
        g_scratch_ptr[dev] = p;
    }
    *out = static_cast<char *>(g_scratch_ptr[dev]);
    return KQ_OK;
}

}  // namespace

extern "C" kq_status kq_assign_noalloc(const float *W, int64_t n, const float *C, int32_t K, int32_t *idx,
                                       float *dist, kq_stream_t stream) {
    if (!W || !C || !idx || n < 1 || K < 1 || (int64_t)K > n) return KQ_ERR_INVALID_ARG;
    if (n > NOALLOC_MAX_N || K > NOALLOC_MAX_K) return KQ_ERR_WORKSPACE;
    if (((uintptr_t)W % 16) || ((uintptr_t)C % 4) || ((uintptr_t)idx % 4) || ((uintptr_t)dist % 4))
        return KQ_ERR_ALIGNMENT;
    char *scr = nullptr;
    kq_status st = scratch_for_current_device(&scr);
    if (st != KQ_OK) return st;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return KQ_ERR_CUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return KQ_ERR_CUDA;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    Header *hdr = reinterpret_cast<Header *>(scr + SCR_HEADER);
    float *cd = reinterpret_cast<float *>(scr + SCR_CD);
    unsigned long long *part = reinterpret_cast<unsigned long long *>(scr + SCR_PART);
    double *blocksum = reinterpret_cast<double *>(scr + SCR_BLOCKSUM);
    // The status word and the codebook bounds (cleared by the pack launcher) must
    // start at zero; everything else is fully written before it is read.
    if (cudaMemsetAsync(&hdr->status, 0, sizeof(uint32_t), s) != cudaSuccess) return KQ_ERR_CUDA;
    if (launch_pack_codebook(C, K, cd, hdr, s) != cudaSuccess) return KQ_ERR_CUDA;
    int nb = 0;
    if (launch_assign(W, n, cd, C, K, nullptr, idx, dist, blocksum, &nb, part, hdr, sms, s) != cudaSuccess)
        return KQ_ERR_CUDA;
    return KQ_OK;
}
