// gs_trace.cu -- launch counting and optional per-kernel CUDA-event timing.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>
#include <vector>

#include "gs.h"
#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {
namespace {

const char* kNames[kNumKernels] = {"k_bound", "k_stream", "k_solve", "k_emit",
                                   "k_prob",  "k_words",  "k_bucket", "k_tiles",
                                   "k_stream_tma", "k_decide",
                                   "k_eps_hist", "k_eps_bracket", "k_solve_eps",
                                   "k_lr_grad", "k_lr_margins", "k_row_sq", "k_sum_rows", "k_sgd_step",
                                   "k_dense_count", "k_dense_merge", "k_dense_setup", "k_dense_encode", "k_dense_scan",
                                   "k_dense_decode", "k_small", "k_small_sum", "k_emit_sum"};

struct Pending {
    int k;
    cudaEvent_t a, b;
};

std::mutex mu;
std::atomic<long long> launches[kNumKernels];
std::atomic<int> timing_on{0};
std::vector<Pending> pending;
std::vector<cudaEvent_t> spare;
double acc_ms[kNumKernels];

cudaEvent_t take_event() {
    if (!spare.empty()) {
        cudaEvent_t e = spare.back();
        spare.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

}  // namespace

void trace_set_timing(int mode) { timing_on.store(mode); }

namespace {
thread_local const char* g_site = "kernel launch";
}
void set_launch_error_site(const char* where) { g_site = where; }
const char* launch_error_site() { return g_site; }

TraceScope::TraceScope(int k, cudaStream_t st) : k_(k), st_(st), a_(nullptr) {
    launches[k].fetch_add(1);
    // 1: every kernel; 2: the streaming pass only (on the cluster path, its one kernel)
    const int mode = timing_on.load();
    if (mode == 1 || (mode == 2 && (k == kKStream || k == kKStreamTma || k == kKSmall))) {
        std::lock_guard<std::mutex> lk(mu);
        a_ = take_event();
        if (a_) cudaEventRecord(a_, st_);
    }
}

TraceScope::~TraceScope() {
    if (!a_) return;
    std::lock_guard<std::mutex> lk(mu);
    cudaEvent_t b = take_event();
    if (!b) return;
    cudaEventRecord(b, st_);
    pending.push_back({k_, a_, b});
}

}  // namespace gs

extern "C" {

int gs_kernel_count(void) { return gs::kNumKernels; }

const char* gs_kernel_name(int k) {
    if (k < 0 || k >= gs::kNumKernels) return "unknown";
    return gs::kNames[k];
}

gs_status gs_kernel_times(double* ms, int64_t* nlaunch, int n) {
    using namespace gs;
    std::lock_guard<std::mutex> lk(mu);
    gs_status rc = GS_OK;
    for (auto& p : pending) {
        float t = 0.0f;
        if (cudaEventSynchronize(p.b) != cudaSuccess || cudaEventElapsedTime(&t, p.a, p.b) != cudaSuccess) rc = GS_ERR_CUDA;
        acc_ms[p.k] += (double)t;
        spare.push_back(p.a);
        spare.push_back(p.b);
    }
    pending.clear();
    for (int k = 0; k < kNumKernels; ++k) {
        if (k < n) {
            if (ms) ms[k] = acc_ms[k];
            if (nlaunch) nlaunch[k] = launches[k].load();
        }
        acc_ms[k] = 0.0;
        launches[k].store(0);
    }
    return rc;
}

}  // extern "C"
