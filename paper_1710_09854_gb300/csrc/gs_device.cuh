// gs_device.cuh -- device-side building blocks of the GB300 gradient
// sparsifier: Philox4x32-10, the chunk layout of M worker gradients, the
// per-segment solve record, and deterministic block reductions.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace gs {

// Coordinates per chunk: the unit of work of the streaming pass and the
// capacity of each chunk's candidate lists.  A multiple of 4 so that chunk
// starts inside a worker row keep the 4-coordinate Philox groups aligned.
constexpr int kChunk = 16384;
// Slices of 1024 coordinates per chunk: the unit of work of the sparse sum.
constexpr int kSliceLog = 10;
constexpr int kSlice = 1 << kSliceLog;
constexpr int kSlices = kChunk / kSlice;
constexpr int kSubStride = kSlices + 1;   // k_sub entries per chunk (slice starts 0..16)
// Coordinates per output tile of the sparse sum.
constexpr int kAggTile = 8192;
// Threads per CTA of the streaming / solve / decide kernels.
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
// 4-coordinate groups each thread handles per step of the streaming pass.
constexpr int kGroupsPerThread = 4;

// Device status bits (the host maps them to gs_status codes).
enum : int {
    kStInvalid = 1 << 1,
    kStCapacity = 1 << 3,
    kStNonfinite = 1 << 4,
    kStTimeout = 1 << 5,
    kStInternal = 1 << 6,
    kStAborted = 1 << 7,   // a kernel left with copies into its shared memory still in flight
};

// Segment flags.
enum : int {
    kSegExact = 1,       // the exact fallback solve ran for this segment
    kSegNonfinite = 2,   // the segment holds NaN / Inf
    kSegTakeAll = 4,     // the bound pass kept every candidate (short segment)
};

// Where the M gradients live and how they are cut into segments / chunks.
struct Layout {
    const void* g;            // M x d, row-major
    int dtype;                // 0 fp32, 1 bf16
    int M;
    int L;                    // segments per worker (1: whole row)
    int cpw;                  // chunks per worker
    int64_t d;
    const int64_t* seg_off;   // [L+1] local offsets; NULL when L == 1
    const int32_t* seg_chunk0;// [L+1] first chunk (within a worker) of each segment; NULL when L == 1
    const int32_t* bnd_seg;   // [L] the bound's segment order: those longer than kBoundWarpMax values
                              // first, then the short ones; NULL when L == 1
    int bnd_long;             // how many of bnd_seg are long
    uint64_t seed;
    uint32_t step;
    uint32_t worker0;
    uint32_t rk0[10], rk1[10];  // Philox round keys: seed lo / hi plus r times the Weyl increments
};

// Per-segment state: the bound of the sampling pass and the final solve.
struct SegParam {
    double lam_up;     // upper bound used to build the candidate lists
    double lam;        // final lambda (Algorithm 3)
    double sum_p;      // sum p at the final lambda
    double l1;         // sum |g|
    long long capped;  // #{p = 1}
    float lam_up32;    // fl32(lam_up), rounded up
    float t_c;         // |g| >= t_c goes to the capped-candidate list C
    float lam32;       // fl32(lam)
    float a_cap;       // smallest fp32 a with fl64(lam * a) >= 1 (capped iff |g| >= a_cap)
    float inv_lam32;   // fl32(1 / lam): the amplified value of uncapped entries
    int iters_run;
    int flags;
    int done;          // chunks of the segment whose streaming outputs are written (zeroed by k_bound)
    int w_done;        // segment l == 0 only: chunks of the worker that k_decide has finished (zeroed by k_bound)
    int next_chunk;    // segment 0 only: chunks the streaming pass has handed out past each warp's first
                       // (zeroed by k_bound and k_eps_bracket)
    double sq;         // Algorithm 2 only: sum g_i^2 of the segment
    float t_up;        // Algorithm 2 only: an upper bound of 1 / lambda (+inf if none)
};

// Candidate lists written by the streaming pass, one region per chunk at the
// chunk's flat offset (capacity = chunk length).
struct Lists {
    int2* p_ent;        // keep candidates: (worker-local index, bits of g_i)
    int32_t* p_cnt;     // [n_chunks]
    int32_t* k_sub;     // [n_chunks][kSubStride] kept entries of the chunk before each 1024-coordinate slice
    float* c_val;       // |g| of each capped candidate
    int32_t* c_cnt;     // [n_chunks]
    double* s_low;      // [n_chunks] sum of |g| outside C
    int32_t* k_off;     // [n_chunks] kept count of the chunk, then (after k_scan) the offset
                        // of its first kept entry in its worker's output
    uint32_t* e_bits;   // [n_chunks][kChunk / 32] decision bit of every keep candidate (hybrid code only)
    int32_t* k_offa;    // [n_chunks] hybrid code only (else NULL): kept entries with p = 1, then their offsets
    int32_t* c_pre;     // [n_chunks + n_seg] prefix scratch for segments with many chunks
    double* b_low;      // [n_chunks] Algorithm 2 only (else NULL): sum of g^2 outside C
};

struct Chunk {
    int m;         // worker row
    int l;         // segment within the row
    int seg;       // m * L + l
    int64_t lo;    // worker-local coordinate range [lo, hi)
    int64_t hi;
};

__device__ __forceinline__ Chunk decode_chunk(const Layout& Lo, int c) {
    Chunk ch;
    ch.m = c / Lo.cpw;
    int k = c - ch.m * Lo.cpw;
    if (Lo.L == 1) {
        ch.l = 0;
        ch.lo = (int64_t)k * kChunk;
        ch.hi = min(Lo.d, ch.lo + kChunk);
    } else {
        // last segment whose first chunk is <= k
        int a = 0, b = Lo.L - 1;
        while (a < b) {
            int mid = (a + b + 1) >> 1;
            if (Lo.seg_chunk0[mid] <= k) a = mid; else b = mid - 1;
        }
        ch.l = a;
        ch.lo = Lo.seg_off[a] + (int64_t)(k - Lo.seg_chunk0[a]) * kChunk;
        ch.hi = min(Lo.seg_off[a + 1], ch.lo + kChunk);
    }
    ch.seg = ch.m * Lo.L + ch.l;
    return ch;
}

__device__ __forceinline__ void seg_range(const Layout& Lo, int seg, int& m, int& l, int64_t& lo, int64_t& hi,
                                          int& c0, int& c1) {
    m = seg / Lo.L;
    l = seg - m * Lo.L;
    if (Lo.L == 1) {
        lo = 0;
        hi = Lo.d;
        c0 = m * Lo.cpw;
        c1 = c0 + Lo.cpw;
    } else {
        lo = Lo.seg_off[l];
        hi = Lo.seg_off[l + 1];
        c0 = m * Lo.cpw + Lo.seg_chunk0[l];
        c1 = m * Lo.cpw + Lo.seg_chunk0[l + 1];
    }
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11).  Each round multiplies
// words 0 and 2 by the published constants, swaps the high halves into the
// odd positions crossed with the key, and bumps the key by the Weyl
// increments.  The 32x32->64 products map to one wide integer multiply each.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                               uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint64_t m0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
        const uint64_t m1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
        const uint32_t n0 = (uint32_t)(m1 >> 32) ^ c1 ^ k0;
        const uint32_t n2 = (uint32_t)(m0 >> 32) ^ c3 ^ k1;
        c1 = (uint32_t)m1;
        c3 = (uint32_t)m0;
        c0 = n0;
        c2 = n2;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return make_uint4(c0, c1, c2, c3);
}

// The 4 words of the 4-coordinate group q of worker `worker` at `step`.
__device__ __forceinline__ uint4 group_words(uint64_t seed, uint32_t step, uint32_t worker, int64_t q) {
    return philox4x32_10((uint32_t)((uint64_t)q & 0xFFFFFFFFu), (uint32_t)((uint64_t)q >> 32), worker, step,
                         (uint32_t)(seed & 0xFFFFFFFFu), (uint32_t)(seed >> 32));
}

// Philox4x32-10 for the groups q < 2^32 of one (worker, step): the first
// round's terms that do not depend on q are computed once per chunk.
// The round keys come from the kernel's parameter space (Layout::rk0/rk1),
// so every key XOR reads its key straight from the constant bank.
struct PhiloxStream {
    const uint32_t* rk0;
    const uint32_t* rk1;
    uint32_t x0, x1;     // words 0 and 1 after round 1 (independent of q)
    uint32_t c3k1;       // step ^ key1, the constant half of word 2 after round 1
    __device__ __forceinline__ PhiloxStream(const Layout& Lo, uint32_t worker) : rk0(Lo.rk0), rk1(Lo.rk1) {
        const uint64_t m1 = (uint64_t)0xCD9E8D57u * (uint64_t)worker;
        x0 = (uint32_t)(m1 >> 32) ^ 0u ^ rk0[0];   // counter word 1 (q >> 32) is 0
        x1 = (uint32_t)m1;
        c3k1 = Lo.step ^ rk1[0];
    }
    __device__ __forceinline__ uint4 words(uint32_t q) const {
        return words_after((uint64_t)0xD2511F53u * (uint64_t)q);
    }
    // The same words given round 1's product m0 = 0xD2511F53 * q (which a
    // caller walking consecutive q can carry forward by adding the constant).
    __device__ __forceinline__ uint4 words_after(uint64_t m0) const {
        uint32_t c0 = x0, c1 = x1, c2 = (uint32_t)(m0 >> 32) ^ c3k1, c3 = (uint32_t)m0;
#pragma unroll
        for (int r = 1; r < 10; ++r) {
            const uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
            const uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
            const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ rk0[r];
            const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ rk1[r];
            c1 = (uint32_t)p1;
            c3 = (uint32_t)p0;
            c0 = n0;
            c2 = n2;
        }
        return make_uint4(c0, c1, c2, c3);
    }
};

__device__ __forceinline__ uint32_t word_of(const uint4& w, int s) {
    return s == 0 ? w.x : (s == 1 ? w.y : (s == 2 ? w.z : w.w));
}

// Programmatic dependent launch: a kernel launched with programmatic stream
// serialization may start while its predecessor in the stream still runs;
// this waits until the predecessor grid has completed and its writes are
// visible.  Every kernel of the library calls it, unconditionally, before it
// reads anything a predecessor may have written (all but the streaming pass
// call it first; a plain launch returns at once), so completion stays
// transitive down the stream.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the next kernel in the stream launch before this grid completes (it
// still waits for this grid in its own grid_dep_wait before it reads
// anything this grid writes).
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// 1 + (x >> 9) * 2^-23: a float in [1, 2) that never exceeds 1 + x * 2^-32.
// hi(x * 2^23) = x >> 9, so one multiply-add forms it on the integer-multiply pipe.
__device__ __forceinline__ float unit_plus_one(uint32_t x) {
    uint32_t r;
    asm("mad.hi.u32 %0, %1, 8388608, 1065353216;" : "=r"(r) : "r"(x));
    return __uint_as_float(r);
}

// m | (t & bit) in one three-input logic op.
__device__ __forceinline__ uint32_t or_and(uint32_t m, uint32_t t, uint32_t bit) {
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xF8;" : "=r"(r) : "r"(m), "r"(t), "r"(bit));
    return r;
}

// All ones when a < b (floats), else 0: one compare, no predicate round trip.
__device__ __forceinline__ uint32_t lt_mask(float a, float b) {
    uint32_t r;
    asm("set.lt.u32.f32 %0, %1, %2;" : "=r"(r) : "f"(a), "f"(b));
    return r;
}

// ---------------------------------------------------------------------------
// Loads
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_bits_to_float(uint32_t b) { return __uint_as_float(b << 16); }

// Load the coordinates 4q..4q+3 of worker row `m` that fall in [lo, hi).
// Returns a 4-bit mask of the valid ones; invalid slots read as 0.
__device__ __forceinline__ int load_group(const Layout& Lo, int m, int64_t q, int64_t lo, int64_t hi, float v[4]) {
    const int64_t i0 = q * 4;
    const int64_t flat = (int64_t)m * Lo.d + i0;
    const bool full = (i0 >= lo) && (i0 + 4 <= hi);
    if (Lo.dtype == 0) {
        const float* g = static_cast<const float*>(Lo.g);
        if (full && ((reinterpret_cast<uintptr_t>(g + flat) & 15u) == 0)) {
            float4 t = __ldcs(reinterpret_cast<const float4*>(g + flat));
            v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
            return 0xF;
        }
        int mask = 0;
#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const int64_t i = i0 + s;
            if (i >= lo && i < hi) { v[s] = __ldcs(g + flat + s); mask |= 1 << s; }
            else v[s] = 0.0f;
        }
        return mask;
    } else {
        const uint16_t* g = static_cast<const uint16_t*>(Lo.g);
        if (full && ((reinterpret_cast<uintptr_t>(g + flat) & 7u) == 0)) {
            uint2 t = __ldcs(reinterpret_cast<const uint2*>(g + flat));
            v[0] = bf16_bits_to_float(t.x & 0xFFFFu); v[1] = bf16_bits_to_float(t.x >> 16);
            v[2] = bf16_bits_to_float(t.y & 0xFFFFu); v[3] = bf16_bits_to_float(t.y >> 16);
            return 0xF;
        }
        int mask = 0;
#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const int64_t i = i0 + s;
            if (i >= lo && i < hi) { v[s] = bf16_bits_to_float(g[flat + s]); mask |= 1 << s; }
            else v[s] = 0.0f;
        }
        return mask;
    }
}

__device__ __forceinline__ float load_one(const Layout& Lo, int m, int64_t i) {
    const int64_t flat = (int64_t)m * Lo.d + i;
    if (Lo.dtype == 0) return static_cast<const float*>(Lo.g)[flat];
    return bf16_bits_to_float(static_cast<const uint16_t*>(Lo.g)[flat]);
}

// ---------------------------------------------------------------------------
// Deterministic block reductions (fixed shuffle tree, fixed warp order).
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

// Sum over the block; every thread receives the result.  `sh` holds >= 33 T.
template <typename T>
__device__ __forceinline__ T block_sum(T v, T* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) sh[warp] = v;
    __syncthreads();
    if (warp == 0) {
        T t = lane < nw ? sh[lane] : T(0);
        t = warp_sum(t);
        if (lane == 0) sh[32] = t;
    }
    __syncthreads();
    return sh[32];
}

// Error-free fp32 accumulation (Knuth's TwoSum): hi + lo carries the exact
// running sum to ~2^-48 without touching the fp64 pipe.
__device__ __forceinline__ void two_sum_add(float& hi, float& lo, float x) {
    const float s = hi + x;
    const float bb = s - hi;
    lo += (hi - (s - bb)) + (x - bb);
    hi = s;
}

// (hi, lo) += (bh, bl) for two double-float values, renormalised.
__device__ __forceinline__ void df_add(float& hi, float& lo, float bh, float bl) {
    const float s = hi + bh;
    const float bb = s - hi;
    const float err = (hi - (s - bb)) + (bh - bb);
    const float l = (lo + bl) + err;
    const float t = s + l;
    lo = l - (t - s);
    hi = t;
}

// Sum of double-float values and of ints over the block (butterfly inside
// warps, warps in order); every thread gets the result.
__device__ __forceinline__ void block_sum_df(float& hi, float& lo, int& k, float4* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xFFFFFFFFu, hi, o);
        const float ol = __shfl_xor_sync(0xFFFFFFFFu, lo, o);
        df_add(hi, lo, oh, ol);
        k += __shfl_xor_sync(0xFFFFFFFFu, k, o);
    }
    __syncthreads();
    if (lane == 0) sh[warp] = make_float4(hi, lo, __int_as_float(k), 0.0f);
    __syncthreads();
    if (warp == 0) {
        float4 t = lane < nw ? sh[lane] : make_float4(0.0f, 0.0f, __int_as_float(0), 0.0f);
        float h = t.x, l = t.y;
        int kk = __float_as_int(t.z);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float oh = __shfl_xor_sync(0xFFFFFFFFu, h, o);
            const float ol = __shfl_xor_sync(0xFFFFFFFFu, l, o);
            df_add(h, l, oh, ol);
            kk += __shfl_xor_sync(0xFFFFFFFFu, kk, o);
        }
        if (lane == 0) sh[32] = make_float4(h, l, __int_as_float(kk), 0.0f);
    }
    __syncthreads();
    hi = sh[32].x;
    lo = sh[32].y;
    k = __float_as_int(sh[32].z);
}

// Smallest positive fp32 a with fl64(lam * a) >= 1; +inf when no finite
// float qualifies (lam = 0 or lam * FLT_MAX < 1).  fl64(lam * a) is
// monotone in a, so "fl64(lam*|g|) >= 1" is exactly "|g| >= a_cap".
__device__ __forceinline__ float cap_threshold(double lam) {
    if (!(lam > 0.0)) return __int_as_float(0x7F800000);
    if (lam * 3.4028234663852886e38 < 1.0) return __int_as_float(0x7F800000);
    // Start from an fp32 reciprocal and step one ulp at a time (a few fp64
    // products); fall back to a bisection over the float bit patterns.
    const float f = (float)lam;
    if (f > 0.0f && f < 3.0e38f) {
        uint32_t b = __float_as_uint(__frcp_rn(f));
        if (b > 0u && b < 0x7F7FFFFFu) {
            int guard = 0;
            while (lam * (double)__uint_as_float(b) < 1.0 && b < 0x7F7FFFFFu && ++guard < 16) ++b;
            while (b > 1u && lam * (double)__uint_as_float(b - 1u) >= 1.0 && ++guard < 32) --b;
            if (lam * (double)__uint_as_float(b) >= 1.0 &&
                (b == 1u || lam * (double)__uint_as_float(b - 1u) < 1.0))
                return __uint_as_float(b);
        }
    }
    uint32_t lo = 0, hi = 0x7F7FFFFFu;   // search the bit patterns of finite positive floats
    while (lo < hi) {
        uint32_t mid = lo + ((hi - lo) >> 1);
        if (lam * (double)__uint_as_float(mid) >= 1.0) hi = mid; else lo = mid + 1;
    }
    return __uint_as_float(lo);
}

}  // namespace gs
