// gs_api.cu -- the C ABI of libgs.so (declared in include/gs.h): argument
// validation, the library's stream-ordered memory pool, the per-device
// status word, and the order of the kernel launches of each call.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <vector>

#include "gs.h"
#include "gs_launch.h"
#include "gs_trace.h"

using namespace gs;

namespace {

constexpr int kMaxDevices = 64;
constexpr int64_t kMaxD = (int64_t)1 << 31;

struct SegMeta {
    int64_t* off = nullptr;     // device [L+1]
    int32_t* chunk0 = nullptr;  // device [L+1]
    int32_t* bnd = nullptr;     // device [L]: long segments (> bound_short_max()), then short ones
    int bnd_long = 0;
    int cpw = 0;
};

constexpr int kPipeGroups = 8;   // worker groups of gs_pipeline_host (copies overlapped with compute)

struct DevState {
    bool ready = false;
    cudaMemPool_t pool = nullptr;
    int* status = nullptr;  // device word, OR of kSt* bits
    std::map<std::vector<int64_t>, SegMeta> segs;
    // gs_pipeline_host: two copy streams and the events that order them
    bool pipe_ready = false;
    cudaStream_t copy[2] = {nullptr, nullptr};
    cudaEvent_t ev_start = nullptr;
    cudaEvent_t ev_done = nullptr;       // the last group's sum is written
    cudaEvent_t ev_back[2] = {};         // each half of the read-back has landed
    cudaEvent_t ev_group[kPipeGroups] = {};
    std::mutex pipe_mu;     // one pipeline call at a time per device (they share the events)
};

std::mutex g_mu;
DevState g_dev[kMaxDevices];
thread_local char g_last_error[256] = "";

// Returns GS_ERR_CUDA and remembers which call failed and why.
gs_status cuda_fail(const char* where, cudaError_t e) {
    snprintf(g_last_error, sizeof(g_last_error), "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
    return GS_ERR_CUDA;
}

#define GS_TRY(expr)                                  \
    do {                                              \
        const cudaError_t e_ = (expr);                \
        if (e_ != cudaSuccess) return cuda_fail(#expr, e_); \
    } while (0)
int g_force_exact = 0;
int g_sample = 0;   // 0: automatic (sample_size)

// Coordinates the bound pass samples from each segment: the option when set,
// else 8192 for calls whose longest segment has at most 2^25 coordinates and
// 16384 above.  The bound's cost is per segment, the candidates a looser
// bound adds are per coordinate: measured on GB300, the smaller sample was
// faster on 16 x 2^24 and on the 161 ResNet-50 layers, slower on 8 x 2^27.
int sample_size(int opt, int64_t max_seg_len) {
    return opt > 0 ? opt : (max_seg_len <= ((int64_t)1 << 25) ? 8192 : 16384);
}
int g_stream_path = 0;  // 0 auto, 1 generic loads, 2 TMA (when eligible)
int g_small_path = 0;   // 0 auto, 1 never, 2 whenever the row is short enough

// Rows of at most kSmallMaxD coordinates take the cluster-resident path
// (gs_small.cu) when the whole call is small too (M d <= 2^24): there one
// cluster per worker beats the chunked path's six launches over a few
// busy warps.  Larger calls fill the GPU through the chunked path, whose
// single read of g wins once the cluster path's extra passes do not fit in L2.
bool choose_small(int M, int64_t d) {
    int opt;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        opt = g_small_path;
    }
    if (opt == 1 || !small_path_eligible(d)) return false;
    return opt == 2 || (int64_t)M * d <= ((int64_t)1 << 24);
}

gs_status device_state(DevState** out) {
    int dev = 0;
    GS_TRY(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDevices) return cuda_fail("device ordinal", cudaErrorInvalidDevice);
    std::lock_guard<std::mutex> lk(g_mu);
    DevState& s = g_dev[dev];
    if (!s.ready) {
        cudaMemPoolProps props;
        std::memset(&props, 0, sizeof(props));
        props.allocType = cudaMemAllocationTypePinned;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        GS_TRY(cudaMemPoolCreate(&s.pool, &props));
        uint64_t keep = UINT64_MAX;  // keep freed blocks for the next call
        cudaMemPoolSetAttribute(s.pool, cudaMemPoolAttrReleaseThreshold, &keep);
        GS_TRY(cudaMalloc(&s.status, sizeof(int)));
        GS_TRY(cudaMemset(s.status, 0, sizeof(int)));
        GS_TRY(cudaDeviceSynchronize());
        s.ready = true;
    }
    *out = &s;
    return GS_OK;
}

// Segment tables for layer-wise calls, uploaded once per distinct layout.
gs_status segment_meta(DevState* s, const int64_t* off, int L, SegMeta* out) {
    std::vector<int64_t> key(off, off + L + 1);
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = s->segs.find(key);
    if (it != s->segs.end()) {
        *out = it->second;
        return GS_OK;
    }
    std::vector<int32_t> c0(L + 1);
    int64_t acc = 0;
    for (int l = 0; l < L; ++l) {
        c0[l] = (int32_t)acc;
        acc += (off[l + 1] - off[l] + chunk_size() - 1) / chunk_size();
    }
    c0[L] = (int32_t)acc;
    if (acc > INT32_MAX) return GS_ERR_INVALID_ARG;
    // The bound pass's order: one CTA for each long segment, then warps for
    // the short ones (each in index order).
    std::vector<int32_t> bnd;
    for (int l = 0; l < L; ++l)
        if (off[l + 1] - off[l] > bound_short_max()) bnd.push_back(l);
    const int n_long = (int)bnd.size();
    for (int l = 0; l < L; ++l)
        if (off[l + 1] - off[l] <= bound_short_max()) bnd.push_back(l);
    SegMeta m;
    m.cpw = (int)acc;
    m.bnd_long = n_long;
    GS_TRY(cudaMalloc(&m.off, sizeof(int64_t) * (L + 1)));
    GS_TRY(cudaMalloc(&m.chunk0, sizeof(int32_t) * (L + 1)));
    GS_TRY(cudaMalloc(&m.bnd, sizeof(int32_t) * L));
    GS_TRY(cudaMemcpy(m.off, off, sizeof(int64_t) * (L + 1), cudaMemcpyHostToDevice));
    GS_TRY(cudaMemcpy(m.chunk0, c0.data(), sizeof(int32_t) * (L + 1), cudaMemcpyHostToDevice));
    GS_TRY(cudaMemcpy(m.bnd, bnd.data(), sizeof(int32_t) * L, cudaMemcpyHostToDevice));
    if (s->segs.size() >= 32) s->segs.clear();  // bounded cache (device tables are tiny; kept until exit)
    s->segs[key] = m;
    *out = m;
    return GS_OK;
}

// Bump allocator over one pool allocation; a null base only measures.
struct Arena {
    char* base = nullptr;
    size_t off = 0;
    template <typename T>
    T* take(size_t n) {
        off = (off + 255) & ~(size_t)255;
        T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
        off += n * sizeof(T);
        return p;
    }
};

bool bad_kappa(double kappa) { return !(kappa > 0.0) || kappa > 1.0 || !std::isfinite(kappa); }

struct Workspace {
    SegParam* sp;
    Lists ls;
    int32_t* nnz;       // hybrid calls: the per-worker kept counts (plain calls write the caller's)
    uint32_t* hist;     // Algorithm 2: per-segment magnitude histograms
    double* u_sq;       // Algorithm 2: sum g^2 partials
};

void carve(Arena& a, Workspace& w, int n_seg, int n_chunks, int64_t n, bool build_p, bool hybrid = false,
           int M = 0, bool alg2 = false) {
    std::memset(&w, 0, sizeof(w));
    w.sp = a.take<SegParam>(n_seg);
    if (alg2) {
        w.hist = a.take<uint32_t>(eps_hist_words(n_seg));
        w.u_sq = a.take<double>(eps_units(n_chunks));
        w.ls.b_low = a.take<double>(n_chunks);
    }
    w.ls.c_val = a.take<float>(n);
    w.ls.c_cnt = a.take<int32_t>(n_chunks);
    w.ls.s_low = a.take<double>(n_chunks);
    w.ls.c_pre = a.take<int32_t>((size_t)n_chunks + n_seg);
    if (build_p) {
        w.ls.p_ent = a.take<int2>(n);
        w.ls.p_cnt = a.take<int32_t>(n_chunks);
        w.ls.k_sub = a.take<int32_t>((size_t)n_chunks * kSubStride);
        w.ls.k_off = a.take<int32_t>(n_chunks);
        if (hybrid) {
            w.ls.e_bits = a.take<uint32_t>((size_t)n_chunks * (kChunk / 32));   // the hybrid emit's decision bits
            w.ls.k_offa = a.take<int32_t>(n_chunks);
            w.nnz = a.take<int32_t>(M);
        }
    }
}

// Shared driver of every sparsify / probabilities call.  eps >= 0 selects
// Algorithm 2 (variance budget eps; kappa and iters unused), else Algorithm 3.
gs_status run(const void* g, int dtype, int M, int64_t d, const int64_t* seg_off, int L, double kappa, int iters,
              uint64_t seed, uint32_t step, uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
              gs_info* info, float* p, cudaStream_t st, float* agg_out = nullptr, const HybridOut* hy = nullptr,
              double eps = -1.0, bool average = false, bool accumulate = false, int path_hint = -1) {
    const bool prob = p != nullptr;
    const bool alg2 = eps >= 0.0;
    if (!g || M < 1 || d < 1 || d >= kMaxD) return GS_ERR_INVALID_ARG;
    if (alg2 ? !std::isfinite(eps) : (bad_kappa(kappa) || iters < 0)) return GS_ERR_INVALID_ARG;
    if (dtype != GS_DTYPE_F32 && dtype != GS_DTYPE_BF16) return GS_ERR_INVALID_ARG;
    const size_t esz = dtype == GS_DTYPE_F32 ? 4 : 2;
    if ((reinterpret_cast<uintptr_t>(g) % esz) != 0) return GS_ERR_INVALID_ARG;
    if (hy) {
        if (!hy->qa_idx || !hy->qa_val || !hy->qb_code || !hy->n_a || !hy->n_b || !hy->inv_lam || cap < 1 || L != 1)
            return GS_ERR_INVALID_ARG;
    } else if (!prob && (!idx || !val || !nnz || cap < 1)) {
        return GS_ERR_INVALID_ARG;
    }
    if ((int64_t)M > ((int64_t)1 << 40) / d) return GS_ERR_INVALID_ARG;
    if (L < 1) return GS_ERR_INVALID_ARG;
    if (L > 1) {
        if (!seg_off || seg_off[0] != 0 || seg_off[L] != d) return GS_ERR_INVALID_ARG;
        for (int l = 0; l < L; ++l)
            if (seg_off[l + 1] <= seg_off[l]) return GS_ERR_INVALID_ARG;
    }

    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;

    Layout Lo;
    std::memset(&Lo, 0, sizeof(Lo));
    Lo.g = g;
    Lo.dtype = dtype;
    Lo.M = M;
    Lo.L = L;
    Lo.d = d;
    Lo.seed = seed;
    Lo.step = step;
    Lo.worker0 = worker0;
    for (int r = 0; r < 10; ++r) {
        Lo.rk0[r] = (uint32_t)(seed & 0xFFFFFFFFu) + (uint32_t)r * 0x9E3779B9u;
        Lo.rk1[r] = (uint32_t)(seed >> 32) + (uint32_t)r * 0xBB67AE85u;
    }
    int force_opt;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        force_opt = g_force_exact;
    }
    // Short rows: the cluster-resident path (always exact, so a forced exact
    // solve, which exercises the chunked path's fallback, keeps the chunked path).
    const bool small_ok = !prob && !hy && !alg2 && L == 1 && force_opt == 0 && small_path_eligible(d);
    if (small_ok && (path_hint == 1 || (path_hint < 0 && choose_small(M, d)))) {
        const bool sum_kernel = agg_out != nullptr && M > 1;
        void* mem = nullptr;
        if (sum_kernel) {
            const cudaError_t ea = cudaMallocFromPoolAsync(&mem, small_scratch_bytes(M, d), s->pool, st);
            if (ea != cudaSuccess) return cuda_fail("cudaMallocFromPoolAsync", ea);
        }
        const cudaError_t e = launch_small(Lo, kappa, iters, idx, val, nnz, cap, s->status, info, agg_out, average,
                                           accumulate, mem, st);
        const cudaError_t ef = mem ? cudaFreeAsync(mem, st) : cudaSuccess;
        if (e != cudaSuccess) return cuda_fail(launch_error_site(), e);
        if (ef != cudaSuccess) return cuda_fail("cudaFreeAsync", ef);
        return GS_OK;
    }
    if (L == 1) {
        const int64_t cpw = (d + chunk_size() - 1) / chunk_size();
        Lo.cpw = (int)cpw;
    } else {
        SegMeta meta;
        rc = segment_meta(s, seg_off, L, &meta);
        if (rc != GS_OK) return rc;
        Lo.seg_off = meta.off;
        Lo.seg_chunk0 = meta.chunk0;
        Lo.bnd_seg = meta.bnd;
        Lo.bnd_long = meta.bnd_long;
        Lo.cpw = meta.cpw;
    }
    int64_t max_seg_len = d;   // the longest segment (sizes the solve's shared memory)
    if (L > 1) {
        max_seg_len = 0;
        for (int l = 0; l < L; ++l) max_seg_len = std::max<int64_t>(max_seg_len, seg_off[l + 1] - seg_off[l]);
    }
    const int64_t n_chunks64 = (int64_t)M * Lo.cpw;
    const int64_t n_seg64 = (int64_t)M * L;
    if (n_chunks64 > INT32_MAX || n_seg64 > INT32_MAX) return GS_ERR_INVALID_ARG;
    const int n_chunks = (int)n_chunks64, n_seg = (int)n_seg64;

    Arena a;
    Workspace w;
    carve(a, w, n_seg, n_chunks, (int64_t)M * d, !prob, hy != nullptr, M, alg2);
    void* mem = nullptr;
    {
        const cudaError_t ea = cudaMallocFromPoolAsync(&mem, a.off, s->pool, st);
        if (ea != cudaSuccess) return cuda_fail("cudaMallocFromPoolAsync", ea);
    }
    a.base = static_cast<char*>(mem);
    a.off = 0;
    carve(a, w, n_seg, n_chunks, (int64_t)M * d, !prob, hy != nullptr, M, alg2);

    int force, ns, path;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        force = g_force_exact;
        ns = sample_size(g_sample, max_seg_len);
        path = g_stream_path;
    }
    bool tma_ok = path != 1 && stream_tma_eligible(Lo);
    for (int l = 0; tma_ok && L > 1 && l <= L; ++l)
        if (seg_off[l] % 4 != 0) tma_ok = false;
    cudaError_t e = alg2 ? launch_eps_bracket(Lo, w.sp, w.hist, w.u_sq, n_seg, n_chunks, eps, force, st)
                         : launch_bound(Lo, w.sp, n_seg, kappa, ns, force, st);
    if (e == cudaSuccess) {
        bool used = false;
        if (tma_ok) e = launch_stream_tma(Lo, w.sp, w.ls, n_chunks, s->status, st, &used);
        if (e == cudaSuccess && !used) e = launch_stream(Lo, w.sp, w.ls, n_chunks, !prob, st);
    }
    if (e == cudaSuccess) {
        e = alg2 ? launch_solve_eps(Lo, w.sp, w.ls, n_seg, eps, s->status, info, st)
                 : launch_solve(Lo, w.sp, w.ls, n_seg, kappa, iters, force, s->status, info, st, max_seg_len);
    }
    if (e == cudaSuccess) {
        if (prob) e = launch_prob(Lo, w.sp, p, st);
        else e = launch_compact(Lo, w.sp, w.ls, n_chunks, idx, val, hy ? w.nnz : nnz, cap, s->status, st, agg_out,
                                hy, average, accumulate);
    }
    cudaError_t ef = cudaFreeAsync(mem, st);
    if (e != cudaSuccess) return cuda_fail(launch_error_site(), e);
    if (ef != cudaSuccess) return cuda_fail("cudaFreeAsync", ef);
    return GS_OK;
}

gs_status run_aggregate(const int32_t* const* idx, const float* const* val, const int32_t* nnz, int M, int64_t d,
                        float* out, int64_t cap, cudaStream_t st) {
    if (!idx || !val || !nnz || !out || M < 1 || M > kMaxAggM || d < 1 || d >= kMaxD) return GS_ERR_INVALID_ARG;
    for (int m = 0; m < M; ++m)
        if (!idx[m] || !val[m]) return GS_ERR_INVALID_ARG;
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    AggArgs A;
    std::memset(&A, 0, sizeof(A));
    for (int m = 0; m < M; ++m) {
        A.idx[m] = idx[m];
        A.val[m] = val[m];
    }
    A.nnz = nnz;
    A.M = M;
    A.d = d;
    A.cap = cap;
    const int nt = agg_tiles(d);
    void* mem = nullptr;
    const size_t bytes = sizeof(int32_t) * (size_t)M * (size_t)(nt + 1);
    GS_TRY(cudaMallocFromPoolAsync(&mem, bytes, s->pool, st));
    cudaError_t e = launch_aggregate(A, static_cast<int32_t*>(mem), out, s->status, st);
    cudaError_t ef = cudaFreeAsync(mem, st);
    if (e != cudaSuccess) return cuda_fail(launch_error_site(), e);
    if (ef != cudaSuccess) return cuda_fail("cudaFreeAsync", ef);
    return GS_OK;
}

// ---------------------------------------------------------------------------
// Single-worker sparsify with no allocation (gs_sparsify_noalloc).  Its
// scratch is one file-scope device array sized for d <= kNoAllocMaxD; a
// device that loads this library holds the array until the process exits.

constexpr int64_t kNoAllocMaxD = (int64_t)1 << 22;

constexpr size_t up256(size_t b) { return (b + 255) & ~(size_t)255; }

// Upper bound of what carve() takes for one worker and one segment.
constexpr size_t noalloc_bytes(int64_t n) {
    const size_t nc = (size_t)((n + kChunk - 1) / kChunk);
    return up256(sizeof(SegParam)) + up256(sizeof(float) * n) + up256(sizeof(int32_t) * nc) +
           up256(sizeof(double) * nc) + up256(sizeof(int32_t) * (nc + 1)) + up256(sizeof(int2) * n) +
           up256(sizeof(int32_t) * nc) + up256(sizeof(int32_t) * nc * kSubStride) + up256(sizeof(int32_t) * nc) + up256(sizeof(uint32_t) * nc * (kChunk / 32));
}

constexpr size_t kNoAllocBytes = noalloc_bytes(kNoAllocMaxD);

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];
static __device__ int g_noalloc_status;  // OR of kSt* bits of the current call

struct NoAllocDev {
    bool ready = false;
    char* scratch = nullptr;
    int* status = nullptr;
};
NoAllocDev g_noalloc[kMaxDevices];

// Device addresses of the array and the status word, looked up once per
// device (the lookup may load this library's code onto the device).
gs_status noalloc_device(NoAllocDev** out) {
    int dev = 0;
    GS_TRY(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDevices) return cuda_fail("device ordinal", cudaErrorInvalidDevice);
    std::lock_guard<std::mutex> lk(g_mu);
    NoAllocDev& s = g_noalloc[dev];
    if (!s.ready) {
        void* a = nullptr;
        void* b = nullptr;
        GS_TRY(cudaGetSymbolAddress(&a, g_noalloc_scratch));
        GS_TRY(cudaGetSymbolAddress(&b, g_noalloc_status));
        s.scratch = static_cast<char*>(a);
        s.status = static_cast<int*>(b);
        s.ready = true;
    }
    *out = &s;
    return GS_OK;
}

// Turns the call's status bits into one gs_status code (same precedence as
// gs_sync_status) for the caller's word.
__global__ void k_noalloc_status(const int* bits, int32_t* code) {
    grid_dep_wait();
    const int h = *bits;
    int32_t c = GS_OK;
    if (h & kStAborted) c = GS_ERR_ABORTED;
    else if (h & kStNonfinite) c = GS_ERR_NONFINITE;
    else if (h & kStCapacity) c = GS_ERR_CAPACITY;
    else if (h & kStInvalid) c = GS_ERR_INVALID_ARG;
    else if (h & kStTimeout) c = GS_ERR_TIMEOUT;
    else if (h & kStInternal) c = GS_ERR_INTERNAL;
    *code = c;
}

gs_status run_noalloc(const float* g, int64_t d, double kappa, int iters, uint64_t seed, uint32_t step,
                      uint32_t worker, int32_t* idx, float* val, int32_t* nnz, gs_info* info, int32_t* status,
                      cudaStream_t st) {
    g_last_error[0] = '\0';
    if (!g || !idx || !val || !nnz || d < 1 || bad_kappa(kappa) || iters < 0) return GS_ERR_INVALID_ARG;
    if (!status) {
        // The caller's word is the one place this call's device-side errors go.
        snprintf(g_last_error, sizeof(g_last_error), "gs_sparsify_noalloc: the status word is required");
        return GS_ERR_INVALID_ARG;
    }
    if ((reinterpret_cast<uintptr_t>(g) % sizeof(float)) != 0) return GS_ERR_INVALID_ARG;
    if (d > kNoAllocMaxD) {
        snprintf(g_last_error, sizeof(g_last_error),
                 "gs_sparsify_noalloc: d = %lld is above the limit %lld of its static scratch", (long long)d,
                 (long long)kNoAllocMaxD);
        return GS_ERR_INVALID_ARG;
    }
    NoAllocDev* s = nullptr;
    gs_status rc = noalloc_device(&s);
    if (rc != GS_OK) return rc;

    Layout Lo;
    std::memset(&Lo, 0, sizeof(Lo));
    Lo.g = g;
    Lo.dtype = GS_DTYPE_F32;
    Lo.M = 1;
    Lo.L = 1;
    Lo.d = d;
    Lo.seed = seed;
    Lo.step = step;
    Lo.worker0 = worker;
    for (int r = 0; r < 10; ++r) {
        Lo.rk0[r] = (uint32_t)(seed & 0xFFFFFFFFu) + (uint32_t)r * 0x9E3779B9u;
        Lo.rk1[r] = (uint32_t)(seed >> 32) + (uint32_t)r * 0xBB67AE85u;
    }
    Lo.cpw = (int)((d + chunk_size() - 1) / chunk_size());
    const int n_chunks = Lo.cpw;

    Arena a;
    Workspace w;
    carve(a, w, 1, n_chunks, d, true);
    if (a.off > kNoAllocBytes) return GS_ERR_INTERNAL;
    a.base = s->scratch;
    a.off = 0;
    carve(a, w, 1, n_chunks, d, true);

    int force, ns, path;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        force = g_force_exact;
        ns = sample_size(g_sample, d);
        path = g_stream_path;
    }
    // Every scratch word a kernel reads was written earlier in the same call;
    // the status word is the one thing left from the previous call.
    GS_TRY(cudaMemsetAsync(s->status, 0, sizeof(int), st));
    cudaError_t e = cudaSuccess;
    if (force == 0 && small_path_eligible(d) && choose_small(1, d)) {
        // The path gs_sparsify takes for this d (it needs no scratch at all).
        e = launch_small(Lo, kappa, iters, idx, val, nnz, d, s->status, info, nullptr, false, false, nullptr, st);
    } else {
        const bool tma_ok = path != 1 && stream_tma_eligible(Lo);
        e = launch_bound(Lo, w.sp, 1, kappa, ns, force, st);
        if (e == cudaSuccess) {
            bool used = false;
            if (tma_ok) e = launch_stream_tma(Lo, w.sp, w.ls, n_chunks, s->status, st, &used);
            if (e == cudaSuccess && !used) e = launch_stream(Lo, w.sp, w.ls, n_chunks, true, st);
        }
        if (e == cudaSuccess) e = launch_solve(Lo, w.sp, w.ls, 1, kappa, iters, force, s->status, info, st, d);
        if (e == cudaSuccess) e = launch_compact(Lo, w.sp, w.ls, n_chunks, idx, val, nnz, d, s->status, st);
    }
    if (e == cudaSuccess) {
        k_noalloc_status<<<1, 1, 0, st>>>(s->status, status);
        e = cudaGetLastError();
        if (e != cudaSuccess) set_launch_error_site("k_noalloc_status");
    }
    if (e != cudaSuccess) return cuda_fail(launch_error_site(), e);
    return GS_OK;
}

}  // namespace

extern "C" {

const char* gs_status_string(int status) {
    switch (status) {
        case GS_OK: return "GS_OK";
        case GS_ERR_INVALID_ARG: return "GS_ERR_INVALID_ARG";
        case GS_ERR_CUDA: return "GS_ERR_CUDA";
        case GS_ERR_CAPACITY: return "GS_ERR_CAPACITY";
        case GS_ERR_NONFINITE: return "GS_ERR_NONFINITE";
        case GS_ERR_TIMEOUT: return "GS_ERR_TIMEOUT";
        case GS_ERR_INTERNAL: return "GS_ERR_INTERNAL";
        case GS_ERR_ABORTED: return "GS_ERR_ABORTED";
        default: return "GS_UNKNOWN_STATUS";
    }
}

int gs_version(void) { return 100; }

const char* gs_last_error(void) { return g_last_error; }

gs_status gs_sync_status(void* stream) {
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    int h = 0;
    GS_TRY(cudaMemcpyAsync(&h, s->status, sizeof(int), cudaMemcpyDeviceToHost, st));
    GS_TRY(cudaMemsetAsync(s->status, 0, sizeof(int), st));
    GS_TRY(cudaStreamSynchronize(st));
    if (h & kStAborted) return GS_ERR_ABORTED;
    if (h & kStNonfinite) return GS_ERR_NONFINITE;
    if (h & kStCapacity) return GS_ERR_CAPACITY;
    if (h & kStInvalid) return GS_ERR_INVALID_ARG;
    if (h & kStTimeout) return GS_ERR_TIMEOUT;
    if (h & kStInternal) return GS_ERR_INTERNAL;
    return GS_OK;
}

gs_status gs_probabilities(const float* g, int64_t d, double kappa, int iters, float* p, void* stream) {
    return gs_probabilities_ex(g, d, kappa, iters, p, nullptr, stream);
}

gs_status gs_probabilities_ex(const float* g, int64_t d, double kappa, int iters, float* p, gs_info* info,
                              void* stream) {
    if (!p) return GS_ERR_INVALID_ARG;
    return run(g, GS_DTYPE_F32, 1, d, nullptr, 1, kappa, iters, 0, 0, 0, nullptr, nullptr, nullptr, 0, info, p,
               static_cast<cudaStream_t>(stream));
}

gs_status gs_sparsify(const float* g, int64_t d, double kappa, int iters, uint64_t seed, uint32_t step,
                      uint32_t worker, int32_t* idx, float* val, int32_t* nnz, void* stream) {
    return run(g, GS_DTYPE_F32, 1, d, nullptr, 1, kappa, iters, seed, step, worker, idx, val, nnz, d, nullptr,
               nullptr, static_cast<cudaStream_t>(stream));
}

gs_status gs_batched_sparsify(const void* g, int dtype, int M, int64_t d, double kappa, int iters, uint64_t seed,
                              uint32_t step, uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
                              gs_info* info, void* stream) {
    return run(g, dtype, M, d, nullptr, 1, kappa, iters, seed, step, worker0, idx, val, nnz, cap, info, nullptr,
               static_cast<cudaStream_t>(stream));
}

gs_status gs_segmented_sparsify(const void* g, int dtype, int M, int64_t d, const int64_t* seg_offsets, int L,
                                double kappa, int iters, uint64_t seed, uint32_t step, uint32_t worker0, int32_t* idx,
                                float* val, int32_t* nnz, int64_t cap, gs_info* info, void* stream) {
    if (L < 1 || !seg_offsets) return GS_ERR_INVALID_ARG;
    if (L == 1 && (seg_offsets[0] != 0 || seg_offsets[1] != d)) return GS_ERR_INVALID_ARG;
    return run(g, dtype, M, d, seg_offsets, L, kappa, iters, seed, step, worker0, idx, val, nnz, cap, info, nullptr,
               static_cast<cudaStream_t>(stream));
}

gs_status gs_sparse_aggregate(const int32_t* const* idx, const float* const* val, const int32_t* nnz, int M, int64_t d,
                              float* out, void* stream) {
    return run_aggregate(idx, val, nnz, M, d, out, INT64_MAX, static_cast<cudaStream_t>(stream));
}

gs_status gs_sparsify_aggregate(const void* g, int dtype, int M, int64_t d, double kappa, int iters, uint64_t seed,
                                uint32_t step, uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
                                gs_info* info, float* out, void* stream) {
    if (!out || M < 1 || M > kMaxAggM) return GS_ERR_INVALID_ARG;
    return run(g, dtype, M, d, nullptr, 1, kappa, iters, seed, step, worker0, idx, val, nnz, cap, info, nullptr,
               static_cast<cudaStream_t>(stream), out);
}

gs_status gs_segmented_sparsify_aggregate(const void* g, int dtype, int M, int64_t d, const int64_t* seg_offsets,
                                          int L, double kappa, int iters, uint64_t seed, uint32_t step,
                                          uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
                                          gs_info* info, float* out, void* stream) {
    if (!out || M < 1 || M > kMaxAggM || L < 1 || !seg_offsets) return GS_ERR_INVALID_ARG;
    if (L == 1 && (seg_offsets[0] != 0 || seg_offsets[1] != d)) return GS_ERR_INVALID_ARG;
    return run(g, dtype, M, d, seg_offsets, L, kappa, iters, seed, step, worker0, idx, val, nnz, cap, info, nullptr,
               static_cast<cudaStream_t>(stream), out);
}

gs_status gs_sparsify_average_sparsify(const void* g, int dtype, int M, int64_t d, double kappa, int iters,
                                       uint64_t seed, uint32_t step, uint32_t worker0, int32_t* idx, float* val,
                                       int32_t* nnz, int64_t cap, float* v, double kappa_v, int iters_v,
                                       uint32_t worker_v, int32_t* idx_v, float* val_v, int32_t* nnz_v,
                                       gs_info* info, void* stream) {
    if (!v || !idx_v || !val_v || !nnz_v || M < 1 || M > kMaxAggM) return GS_ERR_INVALID_ARG;
    if (bad_kappa(kappa_v) || iters_v < 0) return GS_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(v) % sizeof(float)) != 0) return GS_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // Steps 4-6: the workers' Q(g^m) and their average v.
    gs_status rc = run(g, dtype, M, d, nullptr, 1, kappa, iters, seed, step, worker0, idx, val, nnz, cap, info,
                       nullptr, st, v, nullptr, -1.0, true);
    if (rc != GS_OK) return rc;
    // Step 7: v = Q(v), drawn from the stream of worker id worker_v.
    return run(v, GS_DTYPE_F32, 1, d, nullptr, 1, kappa_v, iters_v, seed, step, worker_v, idx_v, val_v, nnz_v, d,
               info ? info + M : nullptr, nullptr, st);
}

gs_status gs_batched_sparsify_hybrid(const void* g, int dtype, int M, int64_t d, double kappa, int iters,
                                     uint64_t seed, uint32_t step, uint32_t worker0, int32_t* qa_idx, float* qa_val,
                                     uint32_t* qb_code, int32_t* n_a, int32_t* n_b, float* inv_lam, int64_t cap,
                                     gs_info* info, void* stream) {
    HybridOut h;
    h.qa_idx = qa_idx;
    h.qa_val = qa_val;
    h.qb_code = qb_code;
    h.n_a = n_a;
    h.n_b = n_b;
    h.inv_lam = inv_lam;
    return run(g, dtype, M, d, nullptr, 1, kappa, iters, seed, step, worker0, nullptr, nullptr, nullptr, cap, info,
               nullptr, static_cast<cudaStream_t>(stream), nullptr, &h);
}

gs_status gs_probabilities_eps(const float* g, int64_t d, double eps, float* p, gs_info* info, void* stream) {
    if (!p || !(eps >= 0.0) || !std::isfinite(eps)) return GS_ERR_INVALID_ARG;
    return run(g, GS_DTYPE_F32, 1, d, nullptr, 1, 0.0, 0, 0, 0, 0, nullptr, nullptr, nullptr, 0, info, p,
               static_cast<cudaStream_t>(stream), nullptr, nullptr, eps);
}

gs_status gs_batched_sparsify_eps(const void* g, int dtype, int M, int64_t d, double eps, uint64_t seed, uint32_t step,
                                  uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap, gs_info* info,
                                  void* stream) {
    if (!(eps >= 0.0) || !std::isfinite(eps)) return GS_ERR_INVALID_ARG;
    return run(g, dtype, M, d, nullptr, 1, 0.0, 0, seed, step, worker0, idx, val, nnz, cap, info, nullptr,
               static_cast<cudaStream_t>(stream), nullptr, nullptr, eps);
}

gs_status gs_sparsify_noalloc(const float* g, int64_t d, double kappa, int iters, uint64_t seed, uint32_t step,
                              uint32_t worker, int32_t* idx, float* val, int32_t* nnz, gs_info* info, int32_t* status,
                              void* stream) {
    return run_noalloc(g, d, kappa, iters, seed, step, worker, idx, val, nnz, info, status,
                       static_cast<cudaStream_t>(stream));
}

gs_status gs_dense_encode(const int32_t* qa_idx, const uint32_t* qb_code, const int32_t* n_a, const int32_t* n_b,
                          int M, int64_t d, int64_t cap, int log2_k, uint16_t* words, int64_t word_cap,
                          int64_t* n_words, void* stream) {
    if (!qa_idx || !qb_code || !n_a || !n_b || !words || !n_words || M < 1 || d < 1 || d >= kMaxD || cap < 1 ||
        log2_k < 4 || log2_k > 10 || word_cap < 1)
        return GS_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    // Chunks: at most ceil(min(d, 2 cap) / K) per worker (the lists hold at most 2 cap entries).
    const int64_t per = (std::min<int64_t>(d, 2 * cap) + (1 << log2_k) - 1) >> log2_k;
    const int64_t max_chunks = (int64_t)M * per;
    void* mem = nullptr;
    GS_TRY(cudaMallocFromPoolAsync(&mem, dense_workspace_bytes(M, max_chunks, std::min<int64_t>(d, 2 * cap), true), s->pool, st));
    const cudaError_t e = launch_dense_encode(qa_idx, qb_code, n_a, n_b, M, d, cap, log2_k, words, word_cap, n_words,
                                              mem, max_chunks, s->status, st);
    const cudaError_t ef = cudaFreeAsync(mem, st);
    if (e != cudaSuccess) return cuda_fail(launch_error_site(), e);
    if (ef != cudaSuccess) return cuda_fail("cudaFreeAsync", ef);
    return GS_OK;
}

gs_status gs_dense_decode(const uint16_t* words, const int64_t* n_words, int M, int64_t d, int64_t word_cap,
                          int8_t* qt, void* stream) {
    if (!words || !n_words || !qt || M < 1 || d < 1 || d >= kMaxD || word_cap < 9) return GS_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    // Chunks: at most (word_cap - 9) / 3 directory entries per worker, and at
    // most ceil(d / 16) (K >= 16, one non-zero symbol per coordinate at most).
    const int64_t per = std::min<int64_t>((d + 15) / 16, (word_cap - 9) / 3);
    const int64_t max_chunks = std::max<int64_t>(1, (int64_t)M * per);
    void* mem = nullptr;
    GS_TRY(cudaMallocFromPoolAsync(&mem, dense_workspace_bytes(M, max_chunks, 0, false), s->pool, st));
    const cudaError_t e = launch_dense_decode(words, n_words, M, d, word_cap, qt, mem, max_chunks, s->status, st);
    const cudaError_t ef = cudaFreeAsync(mem, st);
    if (e != cudaSuccess) return cuda_fail(launch_error_site(), e);
    if (ef != cudaSuccess) return cuda_fail("cudaFreeAsync", ef);
    return GS_OK;
}

gs_status gs_logreg_grad(const float* X, const float* y, int N, int d, const float* w, const int32_t* batch, int M,
                         int B, float lam2, float* G, float* gsq, void* stream) {
    if (!X || !y || !w || !batch || !G || !gsq || N < 1 || d < 1 || M < 1 || B < 1 || B > kMaxLrBatch)
        return GS_ERR_INVALID_ARG;
    if (!std::isfinite(lam2) || lam2 < 0.0f) return GS_ERR_INVALID_ARG;
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    GS_TRY(launch_lr_grad(X, y, N, d, w, batch, M, B, lam2, G, gsq, s->status, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_logreg_margins(const float* X, const float* y, int N, int d, const float* w, float* margins,
                            void* stream) {
    if (!X || !y || !w || !margins || N < 1 || d < 1) return GS_ERR_INVALID_ARG;
    GS_TRY(launch_lr_margins(X, y, N, d, w, margins, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_row_sq_norms(const float* val, const int32_t* nnz, int M, int64_t cap, float* out, void* stream) {
    if (!val || !nnz || !out || M < 1 || cap < 1) return GS_ERR_INVALID_ARG;
    GS_TRY(launch_row_sq(val, nnz, M, cap, out, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_sum_rows(const float* G, int M, int64_t d, float* v, void* stream) {
    if (!G || !v || M < 1 || d < 1) return GS_ERR_INVALID_ARG;
    GS_TRY(launch_sum_rows(G, M, d, v, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_sgd_step(float* w, const float* v, int64_t d, float scale, float eta0, float T0, int t, const float* qsq,
                      const float* gsq, int M, float* log, void* stream) {
    if (!w || !v || !qsq || !gsq || d < 1 || M < 1 || t < 0 || !(T0 > 0.0f) || !std::isfinite(eta0) ||
        !std::isfinite(scale))
        return GS_ERR_INVALID_ARG;
    GS_TRY(launch_sgd_step(w, v, d, scale, eta0, T0, t, qsq, gsq, M, log, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_pipeline_host(const void* g_host, int dtype, int M, int64_t d, double kappa, int iters, uint64_t seed,
                           uint32_t step, uint32_t worker0, void* g_dev, int32_t* idx, float* val, int32_t* nnz,
                           int64_t cap, float* out, float* out_host, int32_t* nnz_host, void* stream) {
    if (!g_host || !g_dev || !out || !out_host || !nnz_host) return GS_ERR_INVALID_ARG;
    if (M < 1 || M > kMaxAggM || d < 1 || d >= kMaxD || cap < 1) return GS_ERR_INVALID_ARG;
    if (dtype != GS_DTYPE_F32 && dtype != GS_DTYPE_BF16) return GS_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    std::lock_guard<std::mutex> lk(s->pipe_mu);
    if (!s->pipe_ready) {
        for (int i = 0; i < 2; ++i) GS_TRY(cudaStreamCreateWithFlags(&s->copy[i], cudaStreamNonBlocking));
        GS_TRY(cudaEventCreateWithFlags(&s->ev_start, cudaEventDisableTiming));
        GS_TRY(cudaEventCreateWithFlags(&s->ev_done, cudaEventDisableTiming));
        for (int i = 0; i < 2; ++i) GS_TRY(cudaEventCreateWithFlags(&s->ev_back[i], cudaEventDisableTiming));
        for (int k = 0; k < kPipeGroups; ++k) GS_TRY(cudaEventCreateWithFlags(&s->ev_group[k], cudaEventDisableTiming));
        s->pipe_ready = true;
    }
    const size_t esz = dtype == GS_DTYPE_F32 ? 4 : 2;
    // Worker groups: group k's copy (alternating between the two copy
    // streams, which run side by side) is ordered after everything already on
    // `stream` (an earlier call may still read g_dev) and before group k's
    // sparsify + sum on `stream`; the sum continues across groups in worker
    // order, so out is what one call over all M workers would give.
    const int G = std::min(M, kPipeGroups);
    // One path for every group, the one a single call over all M workers takes.
    const int hint = choose_small(M, d) ? 1 : 0;
    GS_TRY(cudaEventRecord(s->ev_start, st));
    for (int i = 0; i < 2; ++i) GS_TRY(cudaStreamWaitEvent(s->copy[i], s->ev_start, 0));
    int m0 = 0;
    for (int k = 0; k < G; ++k) {
        const int m1 = (int)((int64_t)M * (k + 1) / G);
        const size_t off = esz * (size_t)m0 * (size_t)d, bytes = esz * (size_t)(m1 - m0) * (size_t)d;
        cudaStream_t cs = s->copy[k & 1];
        GS_TRY(cudaMemcpyAsync(static_cast<char*>(g_dev) + off, static_cast<const char*>(g_host) + off, bytes,
                               cudaMemcpyHostToDevice, cs));
        GS_TRY(cudaEventRecord(s->ev_group[k], cs));
        m0 = m1;
    }
    m0 = 0;
    for (int k = 0; k < G; ++k) {
        const int m1 = (int)((int64_t)M * (k + 1) / G);
        GS_TRY(cudaStreamWaitEvent(st, s->ev_group[k], 0));
        rc = run(static_cast<const char*>(g_dev) + esz * (size_t)m0 * (size_t)d, dtype, m1 - m0, d, nullptr, 1,
                 kappa, iters, seed, step, worker0 + (uint32_t)m0, idx + (int64_t)m0 * cap, val + (int64_t)m0 * cap,
                 nnz + m0, cap, nullptr, nullptr, st, out, nullptr, -1.0, false, k > 0, hint);
        if (rc != GS_OK) return rc;
        m0 = m1;
    }
    // The sum and counts back to the host in two halves, one per copy stream
    // (one stream reaches about half of the link); `stream` waits for both,
    // so its completion still means out_host and nnz_host are written.
    GS_TRY(cudaEventRecord(s->ev_done, st));
    const size_t half = (size_t)d / 2;
    for (int i = 0; i < 2; ++i) {
        cudaStream_t cs = s->copy[i];
        GS_TRY(cudaStreamWaitEvent(cs, s->ev_done, 0));
        const size_t b = i == 0 ? 0 : half, e = i == 0 ? half : (size_t)d;
        if (e > b)
            GS_TRY(cudaMemcpyAsync(out_host + b, out + b, sizeof(float) * (e - b), cudaMemcpyDeviceToHost, cs));
        if (i == 1)
            GS_TRY(cudaMemcpyAsync(nnz_host, nnz, sizeof(int32_t) * (size_t)M, cudaMemcpyDeviceToHost, cs));
        GS_TRY(cudaEventRecord(s->ev_back[i], cs));
        GS_TRY(cudaStreamWaitEvent(st, s->ev_back[i], 0));
    }
    return GS_OK;
}

gs_status gs_selftest_timeout(int kind, void* stream) {
    if (kind != 0 && kind != 1) return GS_ERR_INVALID_ARG;
    DevState* s = nullptr;
    gs_status rc = device_state(&s);
    if (rc != GS_OK) return rc;
    GS_TRY(launch_wait_selftest(kind, s->status, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_random_words(uint64_t seed, uint32_t step, uint32_t worker, int64_t i0, int64_t n, uint32_t* out,
                          void* stream) {
    if (!out || i0 < 0 || n < 0 || i0 > INT64_MAX - n) return GS_ERR_INVALID_ARG;
    if (n == 0) return GS_OK;
    GS_TRY(launch_words(seed, step, worker, i0, n, out, static_cast<cudaStream_t>(stream)));
    return GS_OK;
}

gs_status gs_set_option(int option, int64_t value) {
    std::lock_guard<std::mutex> lk(g_mu);
    switch (option) {
        case GS_OPT_FORCE_EXACT_SOLVE:
            if (value != 0 && value != 1) return GS_ERR_INVALID_ARG;
            g_force_exact = (int)value;
            return GS_OK;
        case GS_OPT_SAMPLE_SIZE:
            if (value != 0 && (value < 256 || value > 32768 || value % 8 != 0)) return GS_ERR_INVALID_ARG;
            g_sample = (int)value;
            return GS_OK;
        case GS_OPT_STREAM_PATH:
            if (value < 0 || value > 2) return GS_ERR_INVALID_ARG;
            g_stream_path = (int)value;
            return GS_OK;
        case GS_OPT_SMALL_PATH:
            if (value < 0 || value > 2) return GS_ERR_INVALID_ARG;
            g_small_path = (int)value;
            return GS_OK;
        case GS_OPT_KERNEL_TIMING:
            if (value < 0 || value > 2) return GS_ERR_INVALID_ARG;
            trace_set_timing((int)value);
            return GS_OK;
        default:
            return GS_ERR_INVALID_ARG;
    }
}

}  // extern "C"
