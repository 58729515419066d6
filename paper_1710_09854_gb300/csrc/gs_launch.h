// gs_launch.h -- host-side launchers shared by the C ABI (gs_api.cu) and the
// kernels (gs_kernels.cu).  Internal to libgs.so.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <utility>

#include "gs.h"
#include "gs_device.cuh"

namespace gs {

// Launch with programmatic stream serialization: the grid may be scheduled
// while the previous kernel in `st` finishes; it calls grid_dep_wait() before
// touching anything that kernel wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_dep(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// launch_dep with thread-block clusters of `cluster` CTAs along x (set at launch).
template <typename... KArgs, typename... Args>
cudaError_t launch_dep_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, int cluster,
                               cudaStream_t st, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = (unsigned)cluster;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

typedef gs_info gs_info_dev;

// Largest M the sparse sum takes (its pointer tables travel as kernel
// parameters: 2 x 512 x 8 bytes).
constexpr int kMaxAggM = 512;

struct AggArgs {
    const int32_t* idx[kMaxAggM];
    const float* val[kMaxAggM];
    const int32_t* nnz;   // device, M
    int M;
    int64_t d;
    int64_t cap;          // entries beyond cap in a list are never read
};

cudaError_t launch_bound(const Layout& Lo, SegParam* sp, int n_seg, double kappa, int ns, int force_exact,
                         cudaStream_t st);
cudaError_t launch_stream(const Layout& Lo, const SegParam* sp, const Lists& Ls, int n_chunks, bool build_p,
                          cudaStream_t st);
cudaError_t launch_solve(const Layout& Lo, SegParam* sp, const Lists& Ls, int n_seg, double kappa, int iters,
                         int force_exact, int* status, gs_info_dev* info, cudaStream_t st, int64_t max_seg_len);
// Outputs of the hybrid coding (section 3.3): per worker m, rows of `cap`
// entries at m * cap.
struct HybridOut {
    int32_t* qa_idx;    // Q_A: indices of the kept coordinates with p = 1
    float* qa_val;      // Q_A: their values g_i
    uint32_t* qb_code;  // Q_B: 2 * index + (g_i < 0) of the other kept coordinates
    int32_t* n_a;       // [M] Q_A lengths
    int32_t* n_b;       // [M] Q_B lengths
    float* inv_lam;     // [M] fl32(1 / lambda), the magnitude of every Q_B value
};

// Decide, scan and compact; with sum_out also the sparse sum of the M
// compacted rows into sum_out (d fp32), fused with the compaction (with
// average, the sum divided by M; with accumulate, added in worker order to
// the sum already in sum_out); with hybrid (L == 1 only) the hybrid code
// instead of the plain lists.
cudaError_t launch_compact(const Layout& Lo, const SegParam* sp, const Lists& Ls, int n_chunks, int32_t* idx,
                           float* val, int32_t* nnz, int64_t cap, int* status, cudaStream_t st,
                           float* sum_out = nullptr, const HybridOut* hybrid = nullptr, bool average = false,
                           bool accumulate = false);
cudaError_t launch_prob(const Layout& Lo, const SegParam* sp, float* p, cudaStream_t st);
cudaError_t launch_aggregate(const AggArgs& A, int32_t* off, float* out, int* status, cudaStream_t st);
cudaError_t launch_words(uint64_t seed, uint32_t step, uint32_t worker, int64_t i0, int64_t n, uint32_t* out,
                         cudaStream_t st);
bool stream_tma_eligible(const Layout& Lo);
// One warp's bounded wait on something that never completes (kind 0: an
// mbarrier, kind 1: a device flag); records kStTimeout.
cudaError_t launch_wait_selftest(int kind, int* status, cudaStream_t st);
cudaError_t launch_stream_tma(const Layout& Lo, const SegParam* sp, const Lists& Ls, int n_chunks, int* status,
                              cudaStream_t st, bool* used);
// Algorithm 2 (variance budget eps): the histogram pass and the bracket of
// 1 / lambda (replaces launch_bound), and the Newton solve on C (replaces
// launch_solve).  hist holds eps_hist_words(n_seg) words, u_sq
// eps_units(n_chunks) doubles.
size_t eps_hist_words(int n_seg);
size_t eps_units(int n_chunks);
cudaError_t launch_eps_bracket(const Layout& Lo, SegParam* sp, uint32_t* hist, double* u_sq, int n_seg, int n_chunks,
                               double eps, int take_all, cudaStream_t st);
cudaError_t launch_solve_eps(const Layout& Lo, SegParam* sp, const Lists& Ls, int n_seg, double eps, int* status,
                             gs_info_dev* info, cudaStream_t st);
// The training loop of section 5.1 (gs_lr.cu).
constexpr int kMaxLrBatch = 64;
cudaError_t launch_lr_grad(const float* X, const float* y, int N, int d, const float* w, const int32_t* batch, int M,
                           int B, float lam2, float* G, float* gsq, int* status, cudaStream_t st);
cudaError_t launch_lr_margins(const float* X, const float* y, int N, int d, const float* w, float* out,
                              cudaStream_t st);
cudaError_t launch_row_sq(const float* val, const int32_t* nnz, int M, int64_t cap, float* out, cudaStream_t st);
cudaError_t launch_sum_rows(const float* G, int M, int64_t d, float* v, cudaStream_t st);
cudaError_t launch_sgd_step(float* w, const float* v, int64_t d, float scale, float eta0, float T0, int t,
                            const float* qsq, const float* gsq, int M, float* log, cudaStream_t st);
// The dense code of section 3.3 (gs_dense.cu): workspace bytes for M workers
// and at most max_chunks chunks in all, the encoder of the hybrid lists and
// the decoder into dense int8 rows.
size_t dense_workspace_bytes(int M, int64_t max_chunks, int64_t stride, bool encode);
cudaError_t launch_dense_encode(const int32_t* qa, const uint32_t* qb, const int32_t* n_a, const int32_t* n_b, int M,
                                int64_t d, int64_t cap, int log2_k, uint16_t* words, int64_t word_cap,
                                int64_t* n_words, void* ws, int64_t max_chunks, int* status, cudaStream_t st);
cudaError_t launch_dense_decode(const uint16_t* words, const int64_t* n_words, int M, int64_t d, int64_t word_cap,
                                int8_t* qt, void* ws, int64_t max_chunks, int* status, cudaStream_t st);
// The cluster-resident path for rows of d <= kSmallMaxD coordinates
// (gs_small.cu): Algorithm 3, the draw and the compaction of each worker in
// one cluster launch, plus a worker-order sum kernel when out is given and
// M > 1 (scratch: small_scratch_bytes(M, d) bytes of device memory, else
// unused).  With M == 1 the cluster writes out itself.
constexpr int64_t kSmallMaxD = (int64_t)1 << 21;
bool small_path_eligible(int64_t d);
size_t small_scratch_bytes(int M, int64_t d);
cudaError_t launch_small(const Layout& Lo, double kappa, int iters, int32_t* idx, float* val, int32_t* nnz,
                         int64_t cap, int* status, gs_info_dev* info, float* out, bool average, bool accumulate,
                         void* scratch, cudaStream_t st);
// The launchers record which step failed; the C ABI reports it.
void set_launch_error_site(const char* where);
const char* launch_error_site();
int agg_tiles(int64_t d);
int chunk_size();
// Segments of at most this many values get a warp of the layer-wise bound
// pass instead of a CTA.
int bound_short_max();
// Multiprocessor count of the current device (looked up once per device ordinal).
int device_sm_count();

}  // namespace gs
