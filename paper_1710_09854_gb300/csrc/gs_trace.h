// gs_trace.h -- launch counting / timing scopes (internal to libgs.so).
#pragma once

#include <cuda_runtime.h>

namespace gs {

enum KernelId : int {
    kKBound = 0,
    kKStream,
    kKSolve,
    kKEmit,
    kKProb,
    kKWords,
    kKBucket,
    kKTiles,
    kKStreamTma,
    kKDecide,
    kKEpsHist,
    kKEpsBracket,
    kKSolveEps,
    kKLrGrad,
    kKLrMargins,
    kKRowSq,
    kKSumRows,
    kKSgdStep,
    kKDenseCount,
    kKDenseMerge,
    kKDenseSetup,
    kKDenseEncode,
    kKDenseScan,
    kKDenseDecode,
    kKSmall,
    kKSmallSum,
    kKEmitSum,
    kNumKernels
};

void trace_set_timing(int on);

// Counts one launch of kernel k and, when timing is on, brackets everything
// enqueued on `st` during the scope's lifetime with two CUDA events.
class TraceScope {
public:
    TraceScope(int k, cudaStream_t st);
    ~TraceScope();

private:
    int k_;
    cudaStream_t st_;
    cudaEvent_t a_;
};

}  // namespace gs
