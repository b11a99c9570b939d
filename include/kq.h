/*
 * kq.h -- C ABI of libkq, the sm_103a (GB300) implementation of the hot path of
 * Kernel Quantization (KQ, "Kernel Quantization for Efficient Network
 * Compression", arXiv 2003.05148).
 *
 * KQ treats each 3x3 kernel of a conv layer (a 9-float vector) as the unit of
 * quantisation: it learns a codebook of k kernels by k-means (Sec. 3.1, Eq. 1),
 * stores one ceil(log2 k)-bit index per kernel, quantises the codebook scalars to
 * 6 bits by count-weighted k-means (Sec. 3.2) and rebuilds the weights from the
 * indices at test time (Sec. 3.2, last paragraph). Eq. 4-7 count the bits.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Layouts. W is the conv weight viewed as n rows of 9 floats, row-major: the
 *   PyTorch [q][p][3][3] tensor is exactly this with n = p*q and row i = o*p + c
 *   (Sec. 3.1 reshapes W into the kernel matrix [m_0 .. m_{n-1}]). A codebook C is
 *   K rows of 9 floats. Indices are int32, counts int32, codes uint8 (one 6-bit
 *   code per byte, values 0..63), levels 64 floats.
 * - Memory. Every pointer except those documented as host pointers is device
 *   memory owned by the caller. The library allocates no device memory (the
 *   host-only kq_seed_indices uses a temporary host map).
 *   Scratch lives in a caller-allocated workspace of kq_workspace_bytes(n, K)
 *   bytes (256-byte aligned), which must be zero-filled once before its first
 *   use (e.g. torch.zeros); the library keeps it consistent afterwards. One
 *   workspace must not be used by two calls that can run at the same time.
 * - Streams. Work is enqueued on the given stream and the call returns without
 *   waiting for it, except where a call documents otherwise: kq_device_status,
 *   kq_search_codebook_size (host decisions between trial fits) and
 *   kq_fit_codebook with KQ_STOP_ON_STABLE synchronise the stream.
 * - Errors. Arguments are validated on the host before anything is enqueued; a
 *   bad argument returns a status and enqueues nothing. Problems that only the
 *   device can see (a non-finite input, an index or code out of range, a bounded
 *   device-side wait that gave up) set bits of a sticky status word in the
 *   workspace; kq_device_status() reads and clears it. Device code never traps
 *   and never spins without a bound (the one-cluster level fit also uses the
 *   cluster's hardware barrier, which every CTA of the cluster reaches by
 *   construction). A CUDA launch error returns KQ_ERR_CUDA.
 * - Determinism. For identical inputs every output is bitwise identical from
 *   run to run (no floating-point atomics anywhere).
 * - Alignment. W and W_out must be 16-byte aligned; other float / int pointers
 *   4-byte aligned; the workspace 256-byte aligned. Otherwise KQ_ERR_ALIGNMENT.
 * - Sizes. 1 <= K <= n, n < 2^31, K*9 < 2^31.
 */
#ifndef KQ_H_
#define KQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without pulling in the CUDA headers (same underlying type). */
typedef struct CUstream_st *kq_stream_t;

typedef enum {
    KQ_OK = 0,
    KQ_ERR_INVALID_ARG = 1, /* a size, pointer or flag is out of its documented range */
    KQ_ERR_ALIGNMENT = 2,   /* a pointer is not aligned as documented */
    KQ_ERR_NONFINITE = 3,   /* (device status) an input value was NaN or +-inf */
    KQ_ERR_CUDA = 4,        /* a CUDA runtime call or kernel launch failed */
    KQ_ERR_DEVICE_CHECK = 5, /* (device status) an index or code was out of range */
    KQ_ERR_WORKSPACE = 6,   /* workspace missing or smaller than kq_workspace_bytes */
    KQ_ERR_TIMEOUT = 7      /* (device status) a bounded device-side wait gave up */
} kq_status;

/* Bits of the device status word returned by kq_device_status(). */
#define KQ_FLAG_NONFINITE 0x1u
#define KQ_FLAG_INDEX_RANGE 0x2u
#define KQ_FLAG_CODE_RANGE 0x4u
#define KQ_FLAG_TIMEOUT 0x8u

/* kq_fit_codebook flags. */
#define KQ_STOP_ON_STABLE 0x1
#define KQ_FIT_PRUNE 0x2

/* Human-readable name of a status. Never NULL. */
const char *kq_status_string(kq_status s);

/* Version of this ABI; changes whenever a signature or a layout changes. */
int32_t kq_abi_version(void);

/* Number of CUDA kernels libkq has launched in this process so far (all
 * devices, all threads). A diagnostic for tracing and launch accounting. */
uint64_t kq_kernel_launches(void);

/* Kernel trace, a diagnostic for per-kernel device time. kq_trace_start makes
 * `capacity` (1 .. 2^20) pairs of CUDA events on the current device (host-side
 * objects: no device memory) and starts a trace: from then on each kernel libkq
 * launches, up to `capacity` of them, gets one event recorded on its launch
 * stream just before it and one just after it. kq_trace_stop stops recording (the
 * recorded pairs stay readable); kq_trace_count returns the launches recorded;
 * kq_trace_get waits for launch i's second event and returns the kernel's name (a
 * static string) and the time between the two events in ms. A new
 * kq_trace_start discards the previous trace. One trace per process: trace calls
 * from one host thread on one device at a time. While a trace runs, each launch
 * costs two more stream commands, and a kernel that would otherwise start while
 * its predecessor finishes (a programmatic dependent launch) starts after it.
 * Errors: KQ_ERR_INVALID_ARG for a capacity or index out of range or a NULL
 * output, KQ_ERR_CUDA when an event cannot be made or read. */
kq_status kq_trace_start(int32_t capacity);
kq_status kq_trace_stop(void);
int32_t kq_trace_count(void);
kq_status kq_trace_get(int32_t i, const char **name, float *ms);

/* Failure-detection test hook (no paper counterpart): makes the bounded device-side
 * waits of later calls on this workspace run out, so that tests can check that a
 * wait that gives up is reported (KQ_FLAG_TIMEOUT / KQ_ERR_TIMEOUT from
 * kq_device_status) and that the call still returns, without any GPU fault.
 *   faults      KQ_TEST_SKIP_ARRIVAL: in the grid barriers of the cooperative
 *               kernels (6-bit quantisation, one-launch small fits, fused recovery,
 *               update fallback) CTA 0 never arrives, so the others wait until the
 *               limit (a workspace with a fault set always takes the grid-barrier
 *               level fit, not the one-cluster one); KQ_TEST_STOP_TILE_STREAM: the tensor-core assignment streams
 *               no codeword tile beyond those it starts before its setup, so its
 *               MMA issuers wait until the limit. 0 clears both.
 *   wait_limit  polls before a bounded wait gives up (0: the normal limits, about
 *               2 s for grid barriers and 4M mbarrier polls).
 * Enqueued on `stream` (a one-thread kernel writes the workspace header); stays in
 * effect for this workspace until cleared. The outputs of a call whose wait gave
 * up are unspecified; the workspace's grid-barrier state is left inconsistent, so
 * zero-fill it (or use another) before its next use. ws_bytes >= 4096. */
#define KQ_TEST_SKIP_ARRIVAL 0x1u
#define KQ_TEST_STOP_TILE_STREAM 0x2u
kq_status kq_test_inject_wait_fault(void *ws, size_t ws_bytes, uint32_t faults, uint32_t wait_limit,
                                    kq_stream_t stream);

/* Bytes of workspace needed by any entry point for n kernels and K codewords.
 * Returns 0 when (n, K) is outside the supported range. */
size_t kq_workspace_bytes(int64_t n, int32_t K);

/* Read and clear the sticky device status word of a workspace. Synchronises
 * `stream` first (so it reports every call enqueued before it on that stream).
 * *flags_out (host pointer, may be NULL) receives the raw KQ_FLAG_* bits.
 * Returns KQ_OK, or the status of the most severe flag set:
 * KQ_ERR_TIMEOUT > KQ_ERR_DEVICE_CHECK > KQ_ERR_NONFINITE. */
kq_status kq_device_status(void *ws, size_t ws_bytes, kq_stream_t stream, uint32_t *flags_out);

/* Codeword initialisation: C0[j] = W[sel[j]] for j < K.
 * The paper does not say how k-means is initialised (Sec. 3.1); KQ here seeds
 * the codebook with K distinct kernels whose row numbers the caller draws.
 *   W    n x 9 fp32 (device);  sel  K int64 row numbers in [0, n) (device)
 *   C0   K x 9 fp32 output (device)
 * Uses only the first 4096 bytes of the workspace (ws_bytes >= 4096).
 * A row number outside [0, n) sets KQ_FLAG_INDEX_RANGE and writes zeros. */
kq_status kq_init_codebook(const float *W, int64_t n, const int64_t *sel, int32_t K, float *C0, void *ws,
                           size_t ws_bytes, kq_stream_t stream);

/* Assignment step of k-means, Sec. 3.1 Eq. 1: for every kernel m_i,
 *   idx[i]  = argmin_k || m_i - c_k ||^2,   dist[i] = that minimum,
 * with the distance evaluated in fp32 as t_j = fl(x_j - c_j), acc = fma(t_j,
 * t_j, acc) for j = 0..8 in order (acc starts at 0), and ties resolved toward
 * the lowest k (the running best starts at (+inf, 0)). The result is exactly this
 * argmin; internally most pairs are ruled out by a cheaper expanded-form test
 * with a rigorous rounding-error bound, which never changes the answer.
 *   W     n x 9 fp32 (device, 16-byte aligned)
 *   C     K x 9 fp32 (device)
 *   hint  n int32 (device) or NULL: a previous assignment (e.g. the last Lloyd
 *         iteration's). Each row's search starts from its hinted codeword; only
 *         speed depends on it, never the result. Entries outside [0, K) are
 *         ignored. May be the same array as idx (in-place update).
 *   idx   n int32 output (device)
 *   dist  n fp32 output (device) or NULL
 * A non-finite value in W or C sets KQ_FLAG_NONFINITE (the outputs are still
 * written by the rules above). */
kq_status kq_assign(const float *W, int64_t n, const float *C, int32_t K, const int32_t *hint, int32_t *idx,
                    float *dist, void *ws, size_t ws_bytes, kq_stream_t stream);

/* kq_assign (without a hint) for callers that cannot allocate device memory. The paper has no
 * counterpart: this exists for code that must not call cudaMalloc (or have
 * anyone allocate for it) -- e.g. a plugin living inside a host application
 * whose own allocator owns all of the device's memory, or a latency-critical
 * service that forbids allocation, and the synchronisation cudaMalloc/cudaFree
 * can bring, once it is running. Such a caller cannot provide the workspace.
 * Same inputs, outputs and rules as kq_assign, without the workspace: the
 * scratch is a fixed array of about 10 MB built into libkq, which every GPU that
 * loads the library holds until the process exits. Limits: n <= 16,777,216 and
 * K <= 65,536; larger sizes return KQ_ERR_WORKSPACE. It always runs the
 * CUDA-core assignment kernel (the tensor-core one needs packed codeword tiles
 * that the fixed array has no room for), so it returns the same indices and
 * distances as kq_assign, bit for bit, at lower throughput. The first call on a
 * device looks up the array's device address and keeps it (once per device, so
 * make that first call before any stream capture); a cudaDeviceReset of that
 * device invalidates the kept address, so do not call this entry point again in
 * a process after resetting a device it has used. The pointers passed must
 * belong to the current device. Every call on a device shares the array, so calls
 * whose work can overlap on the GPU race: issue them in order on one stream.
 * Device-side flags (e.g. a non-finite input) are not reported by this variant.
 * It never allocates or frees memory. */
kq_status kq_assign_noalloc(const float *W, int64_t n, const float *C, int32_t K, int32_t *idx, float *dist,
                            kq_stream_t stream);

/* Update step of k-means, Sec. 3.1 Eq. 1: for every codeword,
 *   counts[k] = z_k = |S_k| = #{ i : idx[i] == k },
 *   C_next[k] = (1 / z_k) * sum_{i in S_k} m_i   if z_k > 0, else C_prev[k],
 * the minimiser of Eq. 1 for fixed sets S_k (an empty set keeps its codeword).
 * The sums are exact int64 fixed-point sums (scale 2^S chosen from max|W| so
 * that no sum can overflow), so the result does not depend on the order in
 * which kernels are added; it differs from the exact mean by far less than
 * 1e-5 relative.
 *   W       n x 9 fp32 (device, 16-byte aligned);  idx  n int32 (device)
 *   C_prev  K x 9 fp32 (device);  C_next  K x 9 fp32 output (device, may equal C_prev)
 *   counts  K int32 output (device)
 * An index outside [0, K) is skipped and sets KQ_FLAG_INDEX_RANGE. */
kq_status kq_update_centroids(const float *W, int64_t n, const int32_t *idx, int32_t K, const float *C_prev,
                              float *C_next, int32_t *counts, void *ws, size_t ws_bytes, kq_stream_t stream);

/* k-means fit of the kernel codebook, Sec. 3.1 Eq. 1 (the k-means quantisation
 * step of Algorithm 1): from C_init, `iters` times
 * { assign against C_t; objective[t] = sum_i dist_i; C_{t+1} = update },
 * then a final assign against C_iters, objective[iters] = its sum.
 *   W          n x 9 fp32 (device, 16-byte aligned)
 *   C_init     K x 9 fp32 (device); C_out K x 9 fp32 output (device; may equal C_init)
 *   iters      >= 0
 *   flags      0 or a combination of
 *              KQ_STOP_ON_STABLE: stop iterating once an assignment equals the
 *              previous one. That is a fixed point of the iteration (the update
 *              rebuilds the same codebook from the same clusters, bit for bit, and
 *              every later assignment repeats this one), so the outputs are
 *              exactly those of all `iters` iterations; the objective entries of
 *              the skipped steps repeat the last one computed. The call then
 *              synchronises `stream` once per iteration to read the test.
 *              KQ_FIT_PRUNE: for fits of 4096 to 65536 codewords on the
 *              tensor-core path, prune as Yinyang k-means does (Sec. 4.1): the
 *              codebook is ordered by a k-d tree so that each 256-codeword tile
 *              holds nearby codewords, every kernel keeps a lower bound on its
 *              distance to each tile (lowered by the tile's codeword drift after
 *              every update), and a tile that cannot hold a codeword as close as
 *              the kernel's previous one is skipped for a whole block of kernels.
 *              The outputs are identical either way; the workspace holds the
 *              bounds, and kq_fit_prune_stats reports the tiles processed. (On
 *              the 2048 x 2048 stress layer it skips 16-46% of the tiles per
 *              update, 29.5% of a 10-update fit's tile work, but each processed
 *              tile costs more, so it is not the default.)
 *   idx        n int32 output: the final assignment (device)
 *   counts     K int32 output: cluster sizes of the final assignment (device)
 *   objective  iters + 1 fp64 outputs (device) or NULL: Eq. 1 objective per step,
 *              summed in a fixed order (bitwise reproducible)
 *   iters_run  1 int32 output (host) or NULL: codebook updates performed (iters,
 *              or fewer when KQ_STOP_ON_STABLE stopped at a fixed point)
 * Every assignment after the first is warm-started from the previous one (see
 * kq_assign's hint). Without KQ_STOP_ON_STABLE it runs entirely on `stream` with
 * no host synchronisation. */
kq_status kq_fit_codebook(const float *W, int64_t n, int32_t K, const float *C_init, int32_t iters, int32_t flags,
                          float *C_out, int32_t *idx, int32_t *counts, double *objective, int32_t *iters_run,
                          void *ws, size_t ws_bytes, kq_stream_t stream);

/* Work of a pruned fit (KQ_FIT_PRUNE; the tile skipping that stands for
 * Yinyang k-means, Sec. 4.1), for reporting executed against effective
 * distance evaluations. Call it after a kq_fit_codebook call with
 * KQ_FIT_PRUNE and before any other call on the same workspace:
 *   tiles_run  1 uint64 output (host): (256-kernel block, 256-codeword tile)
 *              pairs the tensor core processed over all the fit's assignments
 *   tiles_all  1 uint64 output (host): the pairs those assignments hold in
 *              all, i.e. what the same fit processes without pruning
 * Both are 0 when that fit did not take the pruned path (sizes outside
 * 4096..65536 codewords or off the tensor-core path). Each pair stands for
 * up to 65,536 kernel x codeword distances (fewer in a ragged last block or
 * tile). Synchronises `stream`. Errors: KQ_ERR_INVALID_ARG for a NULL output;
 * KQ_ERR_WORKSPACE / KQ_ERR_ALIGNMENT for a bad workspace. */
kq_status kq_fit_prune_stats(void *ws, size_t ws_bytes, uint64_t *tiles_run, uint64_t *tiles_all,
                             kq_stream_t stream);

/* Adaptive codebook size, Algorithm 1 with Eq. 3 (Sec. 3.1): a binary search for
 * the smallest codebook that keeps a layer's quality above a target. The paper's
 * quality test is validation accuracy; here it is the reconstruction proxy
 *   A(K) = -e(K),  e(K) = sqrt(J_K / J_0),
 * J_K the Eq. 1 objective after `lloyd_iters` updates of kq_fit_codebook from
 * C_0 = W[sel[0..K)], J_0 = sum_i |W_i|^2 (A_ori = 0: the unquantised layer has
 * no error). N_init = floor(alpha * n) (kept in [1, n]); A_base = A(N_init);
 * A_target = A_base - (A_ori - A_base) * r (Eq. 3); B_upper = N_init, B_lower = 0;
 * each step tests N_curr = floor((B_upper + B_lower) / 2) and moves B_upper there
 * when A(N_curr) > A_target, else B_lower. Stops after max_steps tests, when
 * B_upper - B_lower <= 1, or when a test equals A_target exactly. The result is
 * K = B_upper; C_out / idx / counts hold the fit of that size.
 *   W          n x 9 fp32 (device, 16-byte aligned)
 *   sel        sel_len >= N_init distinct row numbers in [0, n) (device int64): the
 *              seeded draw whose prefixes initialise every trial
 *   alpha      entry ratio, > 0;  r  threshold ratio, >= 0
 *   max_steps  0 .. 64;  lloyd_iters  0 .. 100000 (updates per trial fit)
 *   C_out      N_init x 9 fp32 (device);  idx  n int32;  counts  N_init int32 (device)
 *   K_out      host int32;  err_out  host double e(K) or NULL
 *   trace_K / trace_err  host arrays of max_steps + 1 entries or NULL: the sizes
 *              tested (N_init first) and their e
 *   steps_run  host int32 or NULL: bisection steps made
 * Needs the workspace of (n, N_init). Synchronises `stream` after every trial fit
 * (the decisions are taken on the host). */
kq_status kq_search_codebook_size(const float *W, int64_t n, const int64_t *sel, int32_t sel_len, double alpha,
                                  double r, int32_t max_steps, int32_t lloyd_iters, float *C_out, int32_t *idx,
                                  int32_t *counts, int32_t *K_out, double *err_out, int32_t *trace_K,
                                  double *trace_err, int32_t *steps_run, void *ws, size_t ws_bytes,
                                  kq_stream_t stream);

/* 6-bit kernel-codebook quantisation, Sec. 3.2: k-means with 64 levels over all
 * K*9 codebook scalars v_kj, each weighted by its entry's appearance count
 * z_k (how often the entry occurs in W), then the code of every scalar.
 *   - levels start at linspace(min, max, 64) over the scalars with z_k > 0 (all
 *     scalars if no count is positive), computed in fp64 and rounded to fp32;
 *   - a scalar's code is its nearest level by fp32 |v - level|, lower index on ties;
 *   - a level becomes the z-weighted mean of its scalars, computed from exact
 *     int64 fixed-point sums (scale 2^S, S = 62 - e with A*M = f*2^e, f in
 *     [0.5, 1), A = sum of weights, M = max |v| over weighted scalars); a level
 *     with no weighted scalar keeps its value;
 *   - stop when no code changes or after max_iters level updates; the codes
 *     returned are those of the final levels.
 *   C          K x 9 fp32 (device);  counts K int32 >= 0 (device)
 *   max_iters  0 .. 100000
 *   levels     64 fp32 output (device);  codes K x 9 uint8 output (device)
 *   iters_run  1 int32 output (device) or NULL: level updates performed
 * Uses only the first 4096 bytes of the workspace (ws_bytes >= 4096). Up to 8192
 * codewords the fit runs on one thread-block cluster of at most 16 CTAs (the
 * cluster's hardware barrier, distributed shared memory; kq_fit_layers takes it
 * up to ~23K codewords); otherwise the CTAs of the call meet at grid barriers
 * whose waits are bounded (~2 s): a wait that runs out sets KQ_FLAG_TIMEOUT and
 * the call ends without writing its outputs. Both give the same levels, codes
 * and update count. A negative count sets KQ_FLAG_INDEX_RANGE and is treated as 0. */
kq_status kq_quantize_codebook_6bit(const float *C, int32_t K, const int32_t *counts, int32_t max_iters,
                                    float *levels, uint8_t *codes, int32_t *iters_run, void *ws, size_t ws_bytes,
                                    kq_stream_t stream);

/* 6-bit quantisation of a fully-connected layer, Sec. 3.2 (last step: after the
 * codebooks, the fully-connected layers get the same layer-by-layer k-means):
 * the rules of kq_quantize_codebook_6bit over m scalars with every weight 1.
 *   v          m fp32 (device; e.g. the flattened FC weight), 1 <= m <= 2^40
 *   max_iters  0 .. 100000
 *   levels     64 fp32 output (device);  codes m uint8 output (device)
 *   iters_run  1 int32 output (device) or NULL
 * Uses only the first 4096 bytes of the workspace (ws_bytes >= 4096). Up to
 * 73,728 scalars on one thread-block cluster, beyond that bounded grid barriers,
 * as in kq_quantize_codebook_6bit. */
kq_status kq_quantize_scalars_6bit(const float *v, int64_t m, int32_t max_iters, float *levels, uint8_t *codes,
                                   int32_t *iters_run, void *ws, size_t ws_bytes, kq_stream_t stream);

/* Codebook retraining step, Sec. 3.1 Eq. 2: with G the loss gradients of the
 * (reconstructed) kernels, G_i = dL/dm_i, every entry moves against the
 * element-wise average gradient of the kernels mapped to it:
 *   counts[k] = z_k = #{ i : idx[i] == k },
 *   C_next[k] = C[k] - lr * (1 / z_k) * sum_{i in S_k} G_i   if z_k > 0, else C[k].
 * The sums are the exact int64 fixed-point sums of kq_update_centroids (scale
 * from max|G|); mean -> fp32 as there, then step = fl(lr * mean) and
 * C_next = fl(C - step).
 *   G       n x 9 fp32 (device, 16-byte aligned);  idx  n int32 (device)
 *   lr      finite learning rate (the paper's gamma)
 *   C       K x 9 fp32 (device);  C_next K x 9 fp32 output (device, may equal C)
 *   counts  K int32 output (device)
 * An index outside [0, K) is skipped and sets KQ_FLAG_INDEX_RANGE; a non-finite
 * gradient sets KQ_FLAG_NONFINITE. Needs the full workspace of (n, K). */
kq_status kq_codebook_grad_step(const float *G, int64_t n, const int32_t *idx, int32_t K, float lr, const float *C,
                                float *C_next, int32_t *counts, void *ws, size_t ws_bytes, kq_stream_t stream);

/* Retraining step of the quantised codebook, Sec. 3.2 (retrained the same way
 * as the kernel codebook, with averaged gradients): a network weight is
 * W'_ij = levels[codes[idx_i * 9 + j]], so level l moves against the average
 * gradient of every weight whose value it is:
 *   counts[l]      = #{ (i, j) : codes[idx_i * 9 + j] == l },
 *   levels_next[l] = levels[l] - lr * (1 / counts[l]) * sum of those G_ij,
 *                    or levels[l] when counts[l] == 0.
 * Exact int64 fixed-point sums (scale from max|G| and 9n values); mean, step and
 * result rounded as in kq_codebook_grad_step.
 *   G      n x 9 fp32 (device, 16-byte aligned);  idx n int32 (device)
 *   codes  K x 9 uint8 (device), values 0..63;  lr finite
 *   levels 64 fp32 (device);  levels_next 64 fp32 output (device, may equal levels)
 *   counts 64 int64 output (device, 8-byte aligned) or NULL
 * 1 <= n < 2^31, 1 <= K, K*9 < 2^31. An index outside [0, K) is skipped
 * (KQ_FLAG_INDEX_RANGE); a code above 63 is skipped (KQ_FLAG_CODE_RANGE). Uses
 * only the first 4096 bytes of the workspace (ws_bytes >= 4096). */
kq_status kq_levels_grad_step(const float *G, int64_t n, const int32_t *idx, int32_t K, const uint8_t *codes,
                              float lr, const float *levels, float *levels_next, int64_t *counts, void *ws,
                              size_t ws_bytes, kq_stream_t stream);

/* Test-time recovery, Sec. 3.2 (last paragraph): first the kernel codebook is
 * recovered (C_hat[k][j] = levels[codes[k][j]]), then the weight tensor:
 *   W_out[i] = C_hat[idx[i]]   (K+C: codes and levels given), or
 *   W_out[i] = C[idx[i]]       (kernel-level only: codes == NULL and levels == NULL).
 *   idx    n int32 (device);  C  K x 9 fp32 (device; unused when codes are given, may be NULL then)
 *   codes  K x 9 uint8 (device) or NULL;  levels 64 fp32 (device) or NULL
 *   W_out  n x 9 fp32 output (device, 16-byte aligned)
 * An index outside [0, K) writes a zero row and sets KQ_FLAG_INDEX_RANGE; a
 * code above 63 decodes to 0 and sets KQ_FLAG_CODE_RANGE. */
kq_status kq_reconstruct(const int32_t *idx, int64_t n, const float *C, int32_t K, const uint8_t *codes,
                         const float *levels, float *W_out, void *ws, size_t ws_bytes, kq_stream_t stream);

/* Fused 6-bit encode + recovery, Sec. 3.2: the codebook scalars are encoded to
 * their nearest levels (the encode rule of kq_quantize_codebook_6bit: fp32
 * |v - level|, lower index on ties) and the weights rebuilt from the encoded
 * codebook, in one launch:
 *   codes[k][j] = argmin_l |C[k][j] - levels[l]|,   W_out[i][j] = levels[codes[idx[i]][j]].
 *   idx    n int32 (device);  C  K x 9 fp32 (device);  levels 64 fp32 (device)
 *   codes  K x 9 uint8 output (device) or NULL (not stored)
 *   W_out  n x 9 fp32 output (device, 16-byte aligned)
 * An index outside [0, K) writes a zero row and sets KQ_FLAG_INDEX_RANGE; a
 * non-finite codebook value sets KQ_FLAG_NONFINITE (it encodes to level 0). The
 * CTAs meet at a bounded grid barrier (~2 s; KQ_FLAG_TIMEOUT if it runs out). */
kq_status kq_quantize_reconstruct(const int32_t *idx, int64_t n, const float *C, int32_t K, const float *levels,
                                  uint8_t *codes, float *W_out, void *ws, size_t ws_bytes, kq_stream_t stream);

/* One layer of a network for kq_fit_layers. Every pointer is device memory owned
 * by the caller, laid out as for the single-layer calls.
 *   W, n, K    the layer's kernel matrix (n x 9 fp32, 16-byte aligned) and codebook size
 *   sel        K row numbers (int64) or NULL: when given, the codebook starts as
 *              C_0 = W[sel] (kq_init_codebook); when NULL, C holds C_0 on entry
 *   C          K x 9 fp32: C_0 (read) and the fitted codebook (written)
 *   idx, counts, objective   the fit's outputs (kq_fit_codebook; objective may be NULL)
 *   levels, codes            64 fp32 / K x 9 uint8 outputs of the 6-bit codebook
 *              quantisation (kq_quantize_codebook_6bit with `level_iters`), or both NULL
 *   W_out      n x 9 fp32 output (16-byte aligned) of the K+C recovery
 *              (kq_reconstruct from idx, codes and levels), or NULL; needs codes
 *   ws, ws_bytes  this layer's own workspace of kq_workspace_bytes(n, K) bytes */
typedef struct {
    const float *W;
    int64_t n;
    int32_t K;
    const int64_t *sel;
    float *C;
    int32_t *idx;
    int32_t *counts;
    double *objective;
    float *levels;
    uint8_t *codes;
    float *W_out;
    void *ws;
    size_t ws_bytes;
} kq_layer_job;

/* Kernel quantisation of a whole network (Sec. 3.1-3.2 applied layer by layer):
 * for every job, in one call,
 *   [kq_init_codebook from sel] -> kq_fit_codebook(iters, flags)
 *   -> [kq_quantize_codebook_6bit(level_iters)] -> [kq_reconstruct, K+C],
 * a convenience over those calls with the same results, bit for bit. The layers
 * are independent problems, so the library spreads them over up to eight internal
 * streams of the current device (largest (iters + 1) n K first, each to the
 * least-loaded stream), forked from `stream` and joined back into it: the
 * latency-bound phases of one layer (small grids, grid barriers, launch gaps)
 * overlap the work of others. Work enqueued on `stream` after the call starts
 * after every layer is done; the call itself does not wait for the device.
 *   jobs       count >= 1 layers (host array); every job needs its own workspace
 *   iters      >= 0;  level_iters 0 .. 100000 (used when levels/codes are given)
 *   flags      0 or KQ_FIT_PRUNE (KQ_STOP_ON_STABLE would synchronise per layer)
 * Argument errors are reported before any work is enqueued; a failure while
 * enqueueing returns its status after the streams already forked are joined. */
kq_status kq_fit_layers(const kq_layer_job *jobs, int32_t count, int32_t iters, int32_t level_iters, int32_t flags,
                        kq_stream_t stream);

/* Storage accounting of one layer (host only, no device work), Sec. 3.2-3.3 and
 * Sec. 4.1:
 *   Eq. 4  total_bits B = k * omega^2 * b_c + n * ceil(log2 k)
 *          (index_bits = n * ceil(log2 k), codebook_bits = k * omega^2 * b_c;
 *           the 64-entry level table of the 6-bit codebook is not counted)
 *   Eq. 7  beta = B / (n * omega^2)             bits per parameter
 *   Eq. 6  ratio_kq = n * omega^2 * 32 / B      compression ratio C_KQ
 *   Eq. 5  ratio_con_1bit = n * omega^2 * 32 / (2 * 32 + n * omega^2)
 *          the same layer under conventional per-weight quantisation at its
 *          limit (a codebook of u = 2 fp32 entries, one index bit per weight;
 *          Sec. 3.3 puts that limit at 32), for comparison with ratio_kq
 * b_c = 32 for kernel-level quantisation only, 6 after codebook quantisation.
 * Requires n >= 1, 1 <= k, omega >= 1, b_c >= 1, out != NULL (host pointer). */
typedef struct {
    int64_t index_bits;
    int64_t codebook_bits;
    int64_t total_bits;
    double beta;
    double ratio_kq;
    double ratio_con_1bit;
} kq_report;

kq_status kq_compression_report(int64_t n, int32_t k, int32_t omega, int32_t b_c, kq_report *out);

/* The seeded draw of K distinct kernel rows that initialises a codebook
 * (kq_init_codebook's sel; the paper leaves the initialisation open, Sec. 3.1):
 * a partial Fisher-Yates shuffle of [0, n) whose step j = 0..K-1 swaps position j
 * with j + (u_j mod (n - j)); out[j] is position j afterwards. u_j is output j of
 * the SplitMix64 stream (Steele, Lea and Flood, OOPSLA 2014) with key
 * mix(seed * 0x100000001B3 + 4), output j = mix(key + (j + 1) * 0x9E3779B97F4A7C15),
 * mix the SplitMix64 finaliser; all arithmetic modulo 2^64.
 *   n    1 <= n < 2^31;  K  1 <= K <= n
 *   out  K int64 (host)
 * Host only (no device work); uses a temporary host map of at most K entries. */
kq_status kq_seed_indices(int64_t n, int32_t K, uint64_t seed, int64_t *out);

/* Eq. 5 (host only): compression ratio of conventional per-weight quantisation,
 * C_con = n * omega^2 * b_fp / (u * b_1 + n * omega^2 * ceil(log2 u)), with u
 * codebook entries of b_1 bits each and b_fp-bit full-precision weights. */
kq_status kq_conventional_ratio(int64_t n, int32_t omega, int32_t u, int32_t b_1, int32_t b_fp, double *out);

#ifdef __cplusplus
}
#endif

#endif /* KQ_H_ */
