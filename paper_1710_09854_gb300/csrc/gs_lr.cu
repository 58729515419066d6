// gs_lr.cu -- the training loop around the sparsifier for the convex
// experiments of section 5.1: minibatch gradients of the l2-regularised
// logistic loss of eq. (14) for M workers, the margins that give the
// objective, the squared norms that give the variance factor var, and the
// SGD step with the step size divided by var.
//
// Eq. (14): f(w) = (1/N) sum_n log2(1 + exp(-b_n a_n^T w)) + lam2 ||w||^2, so
// one sample's gradient is -b_n a_n sigma(-b_n a_n^T w) / ln 2 + 2 lam2 w,
// sigma(z) = 1 / (1 + exp(-z)).  Minibatch indices are inputs (drawn by the
// caller), so the loop is a pure function of its inputs.
#include <cuda_runtime.h>

#include <cstdint>

#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {

namespace {

constexpr int kLrThreads = 256;
constexpr int kLrWarps = kLrThreads / 32;
constexpr float kInvLn2 = 1.4426950408889634f;

// Block sum with a fixed tree; every thread gets it.
__device__ __forceinline__ float lr_block_sum(float v, float* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) sh[warp] = v;
    __syncthreads();
    if (warp == 0) {
        float t = lane < kLrWarps ? sh[lane] : 0.0f;
        t = warp_sum(t);
        if (lane == 0) sh[32] = t;
    }
    __syncthreads();
    return sh[32];
}

// One CTA per worker: the B margins (one warp per row, fixed shuffle tree),
// then g_i = sum_j c_j X[n_j, i] + 2 lam2 w_i with c_j = -b sigma(-b a^T w) / (B ln 2),
// added in minibatch order, and ||g||^2.
// A batch index outside [0, N) is reported (kStInvalid) and its row skipped.
__global__ void __launch_bounds__(kLrThreads) k_lr_grad(const float* __restrict__ X, const float* __restrict__ y,
                                                        int N, int d, const float* __restrict__ w,
                                                        const int32_t* __restrict__ batch, int B, float lam2,
                                                        float* __restrict__ G, float* __restrict__ gsq,
                                                        int* status) {
    grid_dep_wait();
    __shared__ float coef[kMaxLrBatch];
    __shared__ int32_t rows[kMaxLrBatch];
    __shared__ float sh[33];
    const int m = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = warp; j < B; j += kLrWarps) {
        const int32_t n = batch[(int64_t)m * B + j];
        if ((unsigned)n >= (unsigned)N) {
            if (lane == 0) {
                coef[j] = 0.0f;
                rows[j] = 0;
                atomicOr(status, kStInvalid);
            }
            continue;
        }
        const float* a = X + (int64_t)n * d;
        float s = 0.0f;
        for (int i = lane; i < d; i += 32) s = fmaf(a[i], w[i], s);
        s = warp_sum(s);
        if (lane == 0) {
            const float b = y[n];
            const float sig = 1.0f / (1.0f + expf(b * s));   // sigma(-b a^T w)
            coef[j] = -b * sig * kInvLn2 / (float)B;
            rows[j] = n;
        }
    }
    __syncthreads();
    float sq = 0.0f;
    float* g = G + (int64_t)m * d;
    for (int i = threadIdx.x; i < d; i += kLrThreads) {
        float acc = 0.0f;
        for (int j = 0; j < B; ++j) acc = fmaf(coef[j], X[(int64_t)rows[j] * d + i], acc);
        const float gi = fmaf(2.0f * lam2, w[i], acc);
        g[i] = gi;
        sq = fmaf(gi, gi, sq);
    }
    sq = lr_block_sum(sq, sh);
    if (threadIdx.x == 0) gsq[m] = sq;
}

// margins[n] = b_n a_n^T w: one warp per row.
__global__ void __launch_bounds__(kLrThreads) k_lr_margins(const float* __restrict__ X, const float* __restrict__ y,
                                                           int N, int d, const float* __restrict__ w,
                                                           float* __restrict__ out) {
    grid_dep_wait();
    const int lane = threadIdx.x & 31;
    const int n = blockIdx.x * kLrWarps + (threadIdx.x >> 5);
    if (n >= N) return;
    const float* a = X + (int64_t)n * d;
    float s = 0.0f;
    for (int i = lane; i < d; i += 32) s = fmaf(a[i], w[i], s);
    s = warp_sum(s);
    if (lane == 0) out[n] = y[n] * s;
}

// out[m] = sum of val[m][0..nnz[m])^2 (one CTA per row).
__global__ void __launch_bounds__(kLrThreads) k_row_sq(const float* __restrict__ val, const int32_t* __restrict__ nnz,
                                                       int64_t cap, float* __restrict__ out) {
    grid_dep_wait();
    __shared__ float sh[33];
    const int m = blockIdx.x;
    const int64_t n = min((int64_t)nnz[m], cap);
    const float* v = val + (int64_t)m * cap;
    float s = 0.0f;
    for (int64_t e = threadIdx.x; e < n; e += kLrThreads) s = fmaf(v[e], v[e], s);
    s = lr_block_sum(s, sh);
    if (threadIdx.x == 0) out[m] = s;
}

// v = sum of the M rows of G, in row order.
__global__ void k_sum_rows(const float* __restrict__ G, int M, int64_t d, float* __restrict__ v) {
    grid_dep_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d; i += (int64_t)gridDim.x * blockDim.x) {
        float s = 0.0f;
        for (int m = 0; m < M; ++m) s += G[(int64_t)m * d + i];
        v[i] = s;
    }
}

// w -= eta_t * scale * v with eta_t = eta0 / ((1 + t / T0) var_t) and
// var_t = sum_m qsq[m] / sum_m gsq[m] (section 5.1); log[0..1] = (eta_t, var_t).
__global__ void k_sgd_step(float* __restrict__ w, const float* __restrict__ v, int64_t d, float scale, float eta0,
                           float T0, int t, const float* __restrict__ qsq, const float* __restrict__ gsq, int M,
                           float* __restrict__ log) {
    grid_dep_wait();
    float q = 0.0f, g = 0.0f;
    for (int m = 0; m < M; ++m) {
        q += qsq[m];
        g += gsq[m];
    }
    const float var = g > 0.0f ? q / g : 1.0f;
    const float eta = eta0 / ((1.0f + (float)t / T0) * var);
    const float c = eta * scale;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d; i += (int64_t)gridDim.x * blockDim.x)
        w[i] = fmaf(-c, v[i], w[i]);
    if (log && blockIdx.x == 0 && threadIdx.x == 0) {
        log[0] = eta;
        log[1] = var;
    }
}

int small_grid(int64_t n, int threads) {
    const int64_t b = (n + threads - 1) / threads;
    return (int)(b < 1024 ? (b < 1 ? 1 : b) : 1024);
}

}  // namespace

cudaError_t launch_lr_grad(const float* X, const float* y, int N, int d, const float* w, const int32_t* batch, int M,
                           int B, float lam2, float* G, float* gsq, int* status, cudaStream_t st) {
    set_launch_error_site("k_lr_grad launch");
    TraceScope ts(kKLrGrad, st);
    k_lr_grad<<<M, kLrThreads, 0, st>>>(X, y, N, d, w, batch, B, lam2, G, gsq, status);
    return cudaGetLastError();
}

cudaError_t launch_lr_margins(const float* X, const float* y, int N, int d, const float* w, float* out,
                              cudaStream_t st) {
    set_launch_error_site("k_lr_margins launch");
    TraceScope ts(kKLrMargins, st);
    k_lr_margins<<<(N + kLrWarps - 1) / kLrWarps, kLrThreads, 0, st>>>(X, y, N, d, w, out);
    return cudaGetLastError();
}

cudaError_t launch_row_sq(const float* val, const int32_t* nnz, int M, int64_t cap, float* out, cudaStream_t st) {
    set_launch_error_site("k_row_sq launch");
    TraceScope ts(kKRowSq, st);
    k_row_sq<<<M, kLrThreads, 0, st>>>(val, nnz, cap, out);
    return cudaGetLastError();
}

cudaError_t launch_sum_rows(const float* G, int M, int64_t d, float* v, cudaStream_t st) {
    set_launch_error_site("k_sum_rows launch");
    TraceScope ts(kKSumRows, st);
    k_sum_rows<<<small_grid(d, 256), 256, 0, st>>>(G, M, d, v);
    return cudaGetLastError();
}

cudaError_t launch_sgd_step(float* w, const float* v, int64_t d, float scale, float eta0, float T0, int t,
                            const float* qsq, const float* gsq, int M, float* log, cudaStream_t st) {
    set_launch_error_site("k_sgd_step launch");
    TraceScope ts(kKSgdStep, st);
    k_sgd_step<<<small_grid(d, 256), 256, 0, st>>>(w, v, d, scale, eta0, T0, t, qsq, gsq, M, log);
    return cudaGetLastError();
}

}  // namespace gs
