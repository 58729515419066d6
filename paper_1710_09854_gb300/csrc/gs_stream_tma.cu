// gs_stream_tma.cu -- the single streaming pass over g (steps 1-3 of the
// path: l1 sums of Algorithm 3, the capped candidates, the ordered keep
// candidates) as a persistent sm_103a kernel fed by the Tensor Memory
// Accelerator.
//
// Every warp owns whole chunks and a private ring of shared-memory buffers,
// each guarded by one "full" mbarrier.  A warp's first chunk is fixed by its
// index; whenever its prefetcher passes the end of a chunk it takes the next
// one from a counter shared by the grid (so the last round of chunks spreads
// over the warps that are free, instead of a fixed 6 or 7 chunks per warp),
// and a small per-warp queue hands the same sequence to the consumer.  One
// lane of the warp keeps the ring kRing buffers ahead with
// cp.async.bulk.tensor loads, refilling a buffer as soon as the warp is done
// with it, so warps never wait for one another and a chunk's lists are
// ordered by warp shuffles alone.  A warp takes its chunk 1024 coordinates
// (one buffer) at a time: every lane owns 32 consecutive coordinates, reads
// them from shared memory (the 128-byte swizzle of the tensor map makes those
// reads bank-conflict free), draws the 4 Philox words of each 4-coordinate
// group, and tests every coordinate against the bound lam_up.  Lists come out
// in ascending coordinate order, exactly as k_stream writes them.
//
// The global tensor is g viewed as rows of 128 bytes (32 fp32 or 64 bf16);
// one buffer is one box of 32 x 128 B (fp32) or 16 x 128 B (bf16).  Rows
// past the end of the tensor read as zero and coordinates outside the chunk
// are masked.  Every wait is bounded: on a timeout the warp records
// GS_ERR_TIMEOUT, stops issuing, waits (again bounded) for its outstanding
// copies and leaves.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstddef>
#include <cstdint>
#include <mutex>

#include "gs_device.cuh"
#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {
namespace {

// Occupancy and ring depth.  The kernel is bound by instruction latency (its
// integer work per coordinate is mostly Philox), so resident warps matter
// more than deep rings: kCtas CTAs of kCW warps per SM, each CTA's rings in
// 64 KiB (three CTAs, at most 85 registers a thread: two fp32 buffers a
// warp) or 96 KiB (two CTAs) of shared memory.  Three are faster for whole
// fp32 rows under Algorithm 3; bf16 rows, layer-wise rows (whose segment
// edges take the per-lane path) and the instantiation that also sums
// squares run faster with two.
template <int kCtas>
__host__ __device__ constexpr int ring_budget() { return (kCtas == 3 ? 64 : 96) * 1024; }
constexpr int kCW = 8;                         // warps per CTA
constexpr int kTmaThreads = 32 * kCW;
constexpr int kLaneCoords = 32;                // coordinates per lane per buffer
constexpr int kBufCoords = 32 * kLaneCoords;   // 1024 coordinates per buffer
constexpr int kRowBytes = 128;
constexpr long long kWaitLimit = 1ll << 22;    // try_wait polls before giving up
constexpr int kQueue = 8;                      // per-warp queue of taken chunks (> kRing + 1)

struct StreamArgs {
    Layout Lo;
    const SegParam* sp;
    Lists Ls;
    int n_chunks;
    int* status;
    int* next_chunk;   // chunks handed out past each warp's first (zero at launch)
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(b)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t* b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(b)), "r"(bytes) : "memory");
}
// Orders this thread's earlier shared-memory reads (generic proxy) before a
// later TMA write (async proxy) to the same buffer.
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait until the phase with the given parity has completed; false after
// `limit` polls (each try_wait returns by itself within a hardware time limit).
__device__ __forceinline__ bool mbar_wait_n(uint64_t* b, uint32_t parity, long long limit) {
    for (long long i = 0; i < limit; ++i)
        if (mbar_test(b, parity)) return true;
    return false;
}
__device__ __forceinline__ bool mbar_wait(uint64_t* b, uint32_t parity) { return mbar_wait_n(b, parity, kWaitLimit); }

// A device word nothing ever writes (the self-test's flag).
__device__ int g_never_set = 0;

// Self-test of the bounded waits: one warp waits, with a short limit, on an
// mbarrier that nothing arrives at (kind 0: the streaming kernel's primitive)
// or on a flag that nothing sets (kind 1); on expiry it records kStTimeout in
// the status word and returns, leaving the context usable.
__global__ void k_wait_selftest(int kind, long long limit, int* status) {
    grid_dep_wait();
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    bool ok = false;
    if (kind == 0) {
        ok = mbar_wait_n(&bar, 0u, limit);   // phase 0 never completes
    } else {
        const volatile int* f = &g_never_set;
        for (long long i = 0; i < limit && !ok; ++i) ok = *f != 0;
    }
    if (!__all_sync(0xFFFFFFFFu, ok) && threadIdx.x == 0) atomicOr(status, kStTimeout);
}
__device__ __forceinline__ void tma_load_rows(void* dst, const CUtensorMap* map, int row, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_addr(dst)),
        "l"(map), "r"(0), "r"(row), "r"(smem_addr(bar))
        : "memory");
}

// (m << 1) | sign bit of r: appends one candidate flag to a mask in one funnel shift.
__device__ __forceinline__ uint32_t shl_in(uint32_t m, float r) {
    uint32_t o;
    asm("shf.l.wrap.b32 %0, %1, %2, 1;" : "=r"(o) : "r"(__float_as_uint(r)), "r"(m));
    return o;
}

// Keep-candidate test of one coordinate as a sign bit: negative iff
// 1 + (x >> 9) 2^-23 < fl32(lam_up |g| + 1 + 2^-20), compared as the bit
// patterns of two positive floats (integer subtraction, no fp32 rounding of
// the difference).  (x >> 9) 2^-23 <= u = x 2^-32 and the rounding of the
// right-hand side is below its 2^-20 slack, so every coordinate kept under a
// lambda <= lam_up passes (NaN and Inf |g| pass too).
// (A shift, a three-input add and, at the caller, a funnel shift on the
// integer ALU: measured faster than forming the difference by integer
// multiply-adds, which share the pipe with Philox's wide multiplies.)
__device__ __forceinline__ float cand_sign(uint32_t x, float lam_up, float a, float pbias) {
    const uint32_t pf = __float_as_uint(fmaf(lam_up, fabsf(a), pbias));
    return __uint_as_float((x >> 9) + 0x3F800000u - pf);
}

// Coordinate k (0..31) of a lane's 32, read back from its row of the buffer
// (first_chunk: the lane's first 16-byte chunk; sw: the row's swizzle).
template <int kDtype>
__device__ __forceinline__ float stage_value(const unsigned char* rp, int first_chunk, int sw, int k) {
    if (kDtype == 0) {
        const int chunk = (first_chunk + (k >> 2)) ^ sw;
        return *reinterpret_cast<const float*>(rp + (chunk << 4) + ((k & 3) << 2));
    } else {
        const int chunk = (first_chunk + (k >> 3)) ^ sw;
        const uint16_t b = *reinterpret_cast<const uint16_t*>(rp + (chunk << 4) + ((k & 7) << 1));
        return __uint_as_float((uint32_t)b << 16);
    }
}

// Group j (0..7, four coordinates) of a lane's 32 as g values (signed; the
// callers take |g| where they use it, which folds into their float operands).
// fp32: from a 32-bit shared address, bsa = the lane's row in the buffer with
// the 128-byte swizzle folded in (row | sw << 4): chunk j sits at j ^ sw, so
// one XOR finds it.  bf16 (half a row per lane): from the generic row
// pointer rp, the lane's first chunk and the swizzle (measured faster there).
template <int kDtype>
__device__ __forceinline__ float4 group_at(uint32_t bsa, const unsigned char* rp, int first_chunk, int sw, int j) {
    if (kDtype == 0) {
        return *reinterpret_cast<const float4*>(__cvta_shared_to_generic(bsa ^ (uint32_t)(j << 4)));
    } else {
        const uint2 t = *reinterpret_cast<const uint2*>(rp + (((first_chunk + (j >> 1)) ^ sw) << 4) + ((j & 1) << 3));
        return make_float4(__uint_as_float(t.x << 16), __uint_as_float(t.x & 0xFFFF0000u),
                           __uint_as_float(t.y << 16), __uint_as_float(t.y & 0xFFFF0000u));
    }
}

__device__ __forceinline__ float abs_sum4(const float4& a) {
    return (fabsf(a.x) + fabsf(a.y)) + (fabsf(a.z) + fabsf(a.w));
}
__device__ __forceinline__ float abs_sq4(const float4& a) {
    return (a.x * a.x + a.y * a.y) + (a.z * a.z + a.w * a.w);
}

// A chunk index with its worker and its chunk within the worker.
struct ChunkWalk {
    int c, m, k;
    __device__ __forceinline__ ChunkWalk(const Layout& Lo, int first) { jump(Lo, first); }
    __device__ __forceinline__ void jump(const Layout& Lo, int cc) {
        c = cc;
        m = cc / Lo.cpw;
        k = cc - m * Lo.cpw;
    }
    // The chunk's segment and worker-local range [lo, hi).
    __device__ __forceinline__ void range(const Layout& Lo, int& seg, int64_t& lo, int64_t& hi) const {
        int l = 0;
        if (Lo.L == 1) {
            lo = (int64_t)k * kChunk;
            hi = min(Lo.d, lo + kChunk);
        } else {
            int a = 0, b = Lo.L - 1;
            while (a < b) {
                const int mid = (a + b + 1) >> 1;
                if (Lo.seg_chunk0[mid] <= k) a = mid; else b = mid - 1;
            }
            l = a;
            lo = Lo.seg_off[a] + (int64_t)(k - Lo.seg_chunk0[a]) * kChunk;
            hi = min(Lo.seg_off[a + 1], lo + kChunk);
        }
        seg = m * Lo.L + l;
    }
    // First row and end row (rows of kInner elements) of the chunk.
    __device__ __forceinline__ void rows(const Layout& Lo, int inner, int64_t& flat_lo, int64_t& r_first,
                                         int64_t& r_end, int& seg, int64_t& lo, int64_t& hi) const {
        range(Lo, seg, lo, hi);
        flat_lo = (int64_t)m * Lo.d + lo;
        const int64_t flat_hi = (int64_t)m * Lo.d + hi;
        r_first = flat_lo / inner;
        r_end = (flat_hi + inner - 1) / inner;
    }
};

// kDtype 0: fp32 rows of 32; 1: bf16 rows of 64.  kSq: also the sum of g^2
// outside C (Algorithm 2's solve), the same way as s_low.
template <int kDtype, bool kSq, int kCtas>
__global__ void __launch_bounds__(kTmaThreads, kCtas)
    k_stream_tma(const __grid_constant__ CUtensorMap map, const __grid_constant__ StreamArgs A) {
    constexpr int kInner = kDtype == 0 ? 32 : 64;          // elements per 128-byte row
    constexpr int kBufRows = kBufCoords / kInner;          // 32 or 16
    constexpr int kBufBytes = kBufRows * kRowBytes;        // 4 KiB or 2 KiB
    constexpr int kRing = ring_budget<kCtas>() / (kCW * kBufBytes);   // buffers per warp
    extern __shared__ unsigned char dsm_raw[];
    unsigned char* base = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(base + kCW * kRing * kBufBytes);   // [kCW][kRing]
    volatile int* abort_flag = reinterpret_cast<volatile int*>(full + kCW * kRing);
    // Per-warp queue of the chunks the prefetcher took, in order, for the
    // consumer (at most kRing + 1 <= 7 outstanding).
    volatile int* my_q = reinterpret_cast<volatile int*>(full + kCW * kRing) + 4 + (threadIdx.x >> 5) * kQueue;
    int qt = 0, qh = 0;   // queue tail (prefetcher) and head (consumer)

    const Layout& Lo = A.Lo;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_first = gridDim.x * kCW;                   // chunks 0 .. n_first - 1 are the warps' first
    if (threadIdx.x == 0) {
        for (int i = 0; i < kCW * kRing; ++i) mbar_init(&full[i], 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    uint64_t* my_full = full + warp * kRing;
    unsigned char* my_buf = base + warp * kRing * kBufBytes;
    const int first = blockIdx.x * kCW + warp;

    // Prefetch cursor: the next buffer's row and its chunk's end row.
    // (Rows of 128 bytes number fewer than 2^31: the launcher checks.)
    ChunkWalk pc(Lo, first);
    int prow = 0, prow_end = 0;
    auto cursor = [&]() {
        if (pc.c < A.n_chunks) {
            int64_t fl, lo, hi, r0, r1;
            int seg;
            pc.rows(Lo, kInner, fl, r0, r1, seg, lo, hi);
            prow = (int)r0;
            prow_end = (int)r1;
        }
    };
    cursor();
    int issued = 0, pslot = 0;
    auto prefetch = [&]() {
        if (pc.c >= A.n_chunks) return;
        const int b = pslot;
        pslot = pslot == kRing - 1 ? 0 : pslot + 1;
        if (lane == 0) {
            mbar_arrive_tx(&my_full[b], kBufBytes);
            tma_load_rows(my_buf + b * kBufBytes, &map, prow, &my_full[b]);
        }
        ++issued;
        prow += kBufRows;
        if (prow >= prow_end) {
            int nc = 0;
            if (lane == 0) {
                nc = n_first + atomicAdd(A.next_chunk, 1);
                my_q[qt % kQueue] = nc;
            }
            nc = __shfl_sync(0xFFFFFFFFu, nc, 0);
            ++qt;
            pc.jump(Lo, nc);
            cursor();
        }
    };
    // Until the predecessor grid has completed, only loads of g (an input of
    // the call) are issued: the buffers of the warp's first chunk that need
    // no chunk from the counter (the predecessor zeroes it).  Segment
    // layouts read their tables from device memory, so they wait first.
    int pre = 0;
    if (Lo.L == 1) {
#pragma unroll 1
        while (pre < kRing && pc.c < A.n_chunks && prow + kBufRows < prow_end) {
            prefetch();
            ++pre;
        }
    }
    grid_dep_wait();
#pragma unroll 1
    for (; pre < kRing; ++pre) prefetch();

    // candidate iff 1 + (x >> 9) 2^-23 < fl32(lam_up |g| + 1 + 2^-20) (cand_sign)
    const float pbias = 1.0f + 0x1p-20f;
    // Probability-only calls keep no keep-candidate lists (their pointer is NULL).
    const bool build_p = A.Ls.p_ent != nullptr;
    // This lane's 32 coordinates of every buffer: one 128-byte row (fp32) or half of one (bf16).
    const int brow = kDtype == 0 ? lane : (lane >> 1);
    const int first_chunk = kDtype == 0 ? 0 : (lane & 1) * 4;
    const int lane_off = lane * kLaneCoords;                 // within the buffer
    const int sw = brow & 7;
    int slot = 0, consumed = 0;
    uint32_t full_parity = 0;
    // This lane's row in buffer 0 as a 32-bit shared address, its first
    // chunk and the 128-byte swizzle folded in (group_at, fp32).
    const uint32_t lane_sa =
        smem_addr(my_buf) + (uint32_t)(brow * kRowBytes) + ((uint32_t)(first_chunk ^ sw) << 4);
    bool live = true;
    // The consumer's next chunk: the one the prefetcher took after the
    // current one; once the prefetcher has stopped (a timeout) the consumer
    // takes chunks itself, so every chunk still gets its counts written.
    auto take_next = [&](ChunkWalk& cw) {
        __syncwarp();
        int nc = 0;
        if (qh != qt) {
            nc = my_q[qh % kQueue];
            ++qh;
        } else {
            if (lane == 0) nc = n_first + atomicAdd(A.next_chunk, 1);
            nc = __shfl_sync(0xFFFFFFFFu, nc, 0);
        }
        cw.jump(Lo, nc);
    };
    for (ChunkWalk cw(Lo, first); cw.c < A.n_chunks; take_next(cw)) {
        int seg;
        int64_t lo, hi, flat_lo, r_first, r_end;
        cw.rows(Lo, kInner, flat_lo, r_first, r_end, seg, lo, hi);
        const int c = cw.c;
        const float lup = A.sp[seg].lam_up32, t_c = A.sp[seg].t_c;
        const int len = (int)(hi - lo);
        const int lead = (int)(flat_lo - r_first * kInner);   // coordinates of the first row before the chunk
        const int span = (int)((r_end - r_first) * kInner);   // coordinates the chunk's buffers cover
        const PhiloxStream ph(Lo, Lo.worker0 + (uint32_t)cw.m);
        float acc_hi = 0.0f, acc_lo = 0.0f;
        float sq_hi = 0.0f, sq_lo = 0.0f;
        int runP = 0, runC = 0;
        // live stays warp-uniform: the refill below is a warp-wide step.  Another
        // warp's abort is seen at the next chunk (a warp whose own wait runs
        // out stops at once).
        live = __all_sync(0xFFFFFFFFu, live && !*abort_flag);
        // A whole chunk: every lane's 32 coordinates lie inside it in every
        // buffer, i.e. its first row starts at the chunk and its length is a
        // whole number of buffers (then lo is a multiple of 4 and the lane's
        // first group is lo / 4 + buf_off / 4 + 8 lane).
        const bool whole = lead == 0 && span == len && len % kBufCoords == 0;
        uint32_t qw = (uint32_t)(lo >> 2) + (uint32_t)(lane_off >> 2);
        for (int buf_off = 0; buf_off < span; buf_off += kBufCoords, qw += kBufCoords / 4) {
            if (live) {
                live = __all_sync(0xFFFFFFFFu, mbar_wait(&my_full[slot], full_parity));
                if (live) {
                    ++consumed;
                } else if (lane == 0) {
                    *abort_flag = 1;
                    atomicOr(A.status, kStTimeout);
                }
            }
            const unsigned char* rp = my_buf + slot * kBufBytes + brow * kRowBytes;
            const int rel = buf_off + lane_off - lead;      // chunk-relative index of coordinate 0
            uint32_t pm = 0, cm = 0;
            float s32 = 0.0f, q32 = 0.0f;
            if (live && (whole || (rel < len && rel + kLaneCoords > 0))) {
                const uint32_t q0 = whole ? qw : (uint32_t)((lo + rel) >> 2);   // worker-local group of coordinate 0
                if (whole || (rel >= 0 && rel + kLaneCoords <= len)) {
                    // All 32 coordinates belong to the chunk: groups of 4 in order,
                    // the l1 (and square) sums accumulated group by group.
                    if constexpr (!kSq) {
                        // Round 1's product 0xD2511F53 q of consecutive groups is
                        // carried by a 64-bit add (integer ALU) instead of a wide
                        // multiply per group.
                        uint64_t m0 = (uint64_t)0xD2511F53u * (uint64_t)q0;
                        const uint32_t bsa = lane_sa + (uint32_t)(slot * kBufBytes);   // this buffer's row, swizzle folded in
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const float4 a = group_at<kDtype>(bsa, rp, first_chunk, sw, j);
                            s32 += abs_sum4(a);
                            if (build_p) {
                                const uint4 w = ph.words_after(m0);
                                m0 += 0xD2511F53u;
                                pm = shl_in(pm, cand_sign(w.x, lup, a.x, pbias));
                                pm = shl_in(pm, cand_sign(w.y, lup, a.y, pbias));
                                pm = shl_in(pm, cand_sign(w.z, lup, a.z, pbias));
                                pm = shl_in(pm, cand_sign(w.w, lup, a.w, pbias));
                            }
                        }
                    } else {
                        // Two groups per step (independent Philox chains) pays in the
                        // instantiation that also sums squares (not in the one above).
                        const uint32_t bsa = lane_sa + (uint32_t)(slot * kBufBytes);
#pragma unroll
                        for (int j = 0; j < 8; j += 2) {
                            const float4 a = group_at<kDtype>(bsa, rp, first_chunk, sw, j);
                            const float4 b = group_at<kDtype>(bsa, rp, first_chunk, sw, j + 1);
                            s32 += abs_sum4(a) + abs_sum4(b);
                            if (kSq) q32 += abs_sq4(a) + abs_sq4(b);
                            if (build_p) {
                                const uint4 w = ph.words(q0 + j);
                                const uint4 v = ph.words(q0 + j + 1);
                                pm = shl_in(pm, cand_sign(w.x, lup, a.x, pbias));
                                pm = shl_in(pm, cand_sign(w.y, lup, a.y, pbias));
                                pm = shl_in(pm, cand_sign(w.z, lup, a.z, pbias));
                                pm = shl_in(pm, cand_sign(w.w, lup, a.w, pbias));
                                pm = shl_in(pm, cand_sign(v.x, lup, b.x, pbias));
                                pm = shl_in(pm, cand_sign(v.y, lup, b.y, pbias));
                                pm = shl_in(pm, cand_sign(v.z, lup, b.z, pbias));
                                pm = shl_in(pm, cand_sign(v.w, lup, b.w, pbias));
                            }
                        }
                    }
                    pm = __brev(pm);   // coordinate k at bit k
                    if (!(s32 < t_c)) {
                        // Some |g| may reach t_c (or be non-finite): split exactly.
                        // (A sum of non-negative floats is at least its largest term.)
                        s32 = 0.0f;
                        q32 = 0.0f;
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            float m4[4];
#pragma unroll
                            for (int k = 0; k < 4; ++k) {
                                const float a = fabsf(stage_value<kDtype>(rp, first_chunk, sw, 4 * j + k));
                                const bool in_c = !(a < t_c);
                                cm |= in_c ? (1u << (4 * j + k)) : 0u;
                                m4[k] = in_c ? 0.0f : a;
                            }
                            s32 += (m4[0] + m4[1]) + (m4[2] + m4[3]);
                            if (kSq) q32 += (m4[0] * m4[0] + m4[1] * m4[1]) + (m4[2] * m4[2] + m4[3] * m4[3]);
                        }
                    }
                } else {
                    // The lane straddles an edge of the chunk: test each coordinate.
                    float s4[8], q4[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint4 w = build_p ? ph.words(q0 + j) : make_uint4(0, 0, 0, 0);
                        float m4[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int e = 4 * j + k;
                            const bool valid = rel + e >= 0 && rel + e < len;
                            const float a = valid ? fabsf(stage_value<kDtype>(rp, first_chunk, sw, e)) : 0.0f;
                            const bool in_c = valid && !(a < t_c);
                            m4[k] = (valid && !in_c) ? a : 0.0f;
                            cm |= in_c ? (1u << e) : 0u;
                            if (build_p && valid &&
                                shl_in(0u, cand_sign(word_of(w, k), lup, a, pbias)) != 0u)
                                pm |= 1u << e;
                        }
                        s4[j] = (m4[0] + m4[1]) + (m4[2] + m4[3]);
                        if (kSq) q4[j] = (m4[0] * m4[0] + m4[1] * m4[1]) + (m4[2] * m4[2] + m4[3] * m4[3]);
                    }
                    s32 = ((s4[0] + s4[1]) + (s4[2] + s4[3])) + ((s4[4] + s4[5]) + (s4[6] + s4[7]));
                    if (kSq) q32 = ((q4[0] + q4[1]) + (q4[2] + q4[3])) + ((q4[4] + q4[5]) + (q4[6] + q4[7]));
                }
            }
            two_sum_add(acc_hi, acc_lo, s32);
            if (kSq) two_sum_add(sq_hi, sq_lo, q32);

            // Order the buffer's candidates by a lane scan.
            const uint32_t packed = (uint32_t)__popc(pm) | ((uint32_t)__popc(cm) << 16);
            uint32_t inc = packed;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                if (lane >= o) inc += t;
            }
            const uint32_t wall = __shfl_sync(0xFFFFFFFFu, inc, 31);
            const uint32_t excl = inc - packed;
            if (pm) {
                int2* e = A.Ls.p_ent + flat_lo + runP + (int)(excl & 0xFFFFu);
                const int32_t i0 = (int32_t)(lo + rel);
                while (pm) {
                    const int k = __ffs(pm) - 1;
                    pm &= pm - 1u;
                    *e++ = make_int2(i0 + k, __float_as_int(stage_value<kDtype>(rp, first_chunk, sw, k)));
                }
            }
            if (cm) {
                float* e = A.Ls.c_val + flat_lo + runC + (int)(excl >> 16);
                while (cm) {
                    const int k = __ffs(cm) - 1;
                    cm &= cm - 1u;
                    *e++ = fabsf(stage_value<kDtype>(rp, first_chunk, sw, k));
                }
            }
            // The warp is done with the buffer: refill it with the buffer kRing ahead.
            if (live) {
                fence_proxy_async();
                __syncwarp();
                prefetch();
            }
            runP += (int)(wall & 0xFFFFu);
            runC += (int)(wall >> 16);
            if (++slot == kRing) {
                slot = 0;
                full_parity ^= 1u;
            }
        }
        // Chunk total: the lanes' (hi, lo) pairs reduced error-free across the warp.
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float oh = __shfl_xor_sync(0xFFFFFFFFu, acc_hi, o);
            const float ol = __shfl_xor_sync(0xFFFFFFFFu, acc_lo, o);
            df_add(acc_hi, acc_lo, oh, ol);
            if (kSq) {
                const float qh = __shfl_xor_sync(0xFFFFFFFFu, sq_hi, o);
                const float ql = __shfl_xor_sync(0xFFFFFFFFu, sq_lo, o);
                df_add(sq_hi, sq_lo, qh, ql);
            }
        }
        if (lane == 0) {
            A.Ls.s_low[c] = (double)acc_hi + (double)acc_lo;
            if (kSq) A.Ls.b_low[c] = (double)sq_hi + (double)sq_lo;
            A.Ls.c_cnt[c] = runC;
            if (A.Ls.p_cnt) A.Ls.p_cnt[c] = runP;
        }
    }
    // After a timeout, wait (bounded) for the copies still in flight into this
    // warp's ring (consumed counts the buffers whose wait succeeded).  The wait
    // is bounded too: a copy that has not landed after another 2^22 polls
    // means the memory system no longer answers, and waiting forever would
    // hang the GPU for every later user of it.  Leaving instead records
    // kStAborted, which the host reports as GS_ERR_ABORTED: a copy may still
    // land in shared memory the CTA has given up, so every result since the
    // last status check is suspect.
    bool landed = true;
    for (int n = consumed; n < issued; ++n) landed = mbar_wait(&my_full[n % kRing], (uint32_t)((n / kRing) & 1)) && landed;
    if (!__all_sync(0xFFFFFFFFu, landed) && lane == 0) atomicOr(A.status, kStAborted);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, looked up once per process (host threads
// making their first call at the same time wait for one lookup).
EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

bool make_map(CUtensorMap* map, const void* g, int dtype, int64_t rows, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const int inner = dtype == 0 ? 32 : 64;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)kRowBytes};
    cuuint32_t box[2] = {(cuuint32_t)inner, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(map, dtype == 0 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                          const_cast<void*>(g), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int kDtype, int kCtas>
size_t tma_smem_bytes() {
    constexpr int kInner = kDtype == 0 ? 32 : 64;
    constexpr int kBufBytes = (kBufCoords / kInner) * kRowBytes;
    constexpr int kRing = ring_budget<kCtas>() / (kCW * kBufBytes);
    static_assert(kQueue > kRing + 1, "the chunk queue must hold every chunk the prefetcher can be ahead");
    // alignment slack + buffers + full barriers + abort flag + chunk queues
    return 1024 + (size_t)kCW * kRing * kBufBytes + (size_t)kCW * kRing * 8 + 16 + (size_t)kCW * kQueue * 4;
}

int sm_count_tma() { return device_sm_count(); }

}  // namespace

cudaError_t launch_wait_selftest(int kind, int* status, cudaStream_t st) {
    set_launch_error_site("k_wait_selftest launch");
    // Short limits: the mbarrier wait gives up after 256 polls, the flag spin
    // after 2^20 loads.
    k_wait_selftest<<<1, 32, 0, st>>>(kind, kind == 0 ? 256 : (1ll << 20), status);
    return cudaGetLastError();
}

bool stream_tma_eligible(const Layout& Lo) {
    if ((reinterpret_cast<uintptr_t>(Lo.g) & 15u) != 0) return false;
    if (Lo.d % 4 != 0) return false;
    const int64_t inner = Lo.dtype == 0 ? 32 : 64;
    const int64_t total = (int64_t)Lo.M * Lo.d;
    if (total % inner != 0) return false;
    if (total / inner >= ((int64_t)1 << 31)) return false;
    return encode_fn() != nullptr;
}

// Segment offsets must be multiples of 4 for the group alignment (checked by the caller).
cudaError_t launch_stream_tma(const Layout& Lo, const SegParam* sp, const Lists& Ls, int n_chunks, int* status,
                              cudaStream_t st, bool* used) {
    set_launch_error_site("k_stream_tma launch");
    *used = false;
    const int64_t inner = Lo.dtype == 0 ? 32 : 64;
    const int64_t rows = (int64_t)Lo.M * Lo.d / inner;
    CUtensorMap map;
    if (!make_map(&map, Lo.g, Lo.dtype, rows, kBufCoords / (int)inner))
        return cudaSuccess;  // caller falls back to the generic pass
    StreamArgs A;
    A.Lo = Lo;
    A.sp = sp;
    A.Ls = Ls;
    A.n_chunks = n_chunks;
    A.status = status;
    // The chunk counter lives in segment 0's parameters (zeroed by the kernel
    // that wrote the bounds, which this launch waits for).
    A.next_chunk = reinterpret_cast<int*>(reinterpret_cast<char*>(const_cast<SegParam*>(sp)) +
                                          offsetof(SegParam, next_chunk));
    // One chunk per warp at a time; as many CTAs as fit on the SMs at once.
    const bool sq = Ls.b_low != nullptr;
    const int ctas = (Lo.dtype == 0 && !sq && Lo.L == 1) ? 3 : 2;
    const int grid = std::min((n_chunks + kCW - 1) / kCW, ctas * sm_count_tma());
    cudaError_t e;
    TraceScope ts(kKStreamTma, st);
    void (*kern)(const CUtensorMap, const StreamArgs);
    size_t smem;
    if (Lo.dtype == 0) {
        kern = sq ? k_stream_tma<0, true, 2> : (ctas == 3 ? k_stream_tma<0, false, 3> : k_stream_tma<0, false, 2>);
        smem = ctas == 3 ? tma_smem_bytes<0, 3>() : tma_smem_bytes<0, 2>();
    } else {
        kern = sq ? k_stream_tma<1, true, 2> : k_stream_tma<1, false, 2>;
        smem = tma_smem_bytes<1, 2>();
    }
    set_launch_error_site("k_stream_tma shared-memory attribute");
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    set_launch_error_site(Lo.dtype == 0 ? "k_stream_tma<fp32> launch" : "k_stream_tma<bf16> launch");
    e = launch_dep(kern, dim3(grid), dim3(kTmaThreads), smem, st, map, A);
    if (e != cudaSuccess) return e;
    *used = true;
    return cudaGetLastError();
}

}  // namespace gs
