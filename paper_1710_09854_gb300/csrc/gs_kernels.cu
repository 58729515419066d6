// gs_kernels.cu -- CUDA kernels (sm_103a) of the gradient-sparsification
// path, Wangni et al., arXiv:1710.09854.
//
// One call over M worker gradients runs:
//   k_bound    per segment: a stratified sample of |g| and Algorithm 3 run to
//              its fixed point on the sample give an upper bound lam_up on
//              the final lambda (a search bound only; correctness never
//              depends on it, see k_solve).
//   k_stream   ONE pass over g (section 3.2, Algorithm 3 step 3 needs
//              sum |g|): per chunk, the sum of |g| outside the capped-candidate
//              set C = {|g| >= t_c}, the values in C, and the ordered list P of
//              coordinates whose Philox word could fall below p_i for any
//              lambda <= lam_up (index, value, word).
//   k_solve    per segment: Algorithm 3 (steps 3-10) run exactly on
//              (S_low, C): every coordinate that any lambda_j <= lam_up caps
//              is in C, so K_j and the uncapped l1 mass are exact.  If the
//              final lambda exceeds lam_up the segment falls back to an exact
//              multi-pass solve over g and rebuilds its P lists.
//   k_decide   per (worker, chunk): the Bernoulli draw Z_i = [u_i < p_i]
//              (section 3) on the P lists; the kept entries, amplified to
//              g_i / p_i, compacted in place over the chunk's P list (for
//              the hybrid code: decision bits instead), and the kept counts;
//              the last warp of each worker scans its counts into offsets.
//   k_emit     per (worker, chunk): each chunk's compacted run copied to
//              its place in the worker's ascending (idx, val) list
//              (k_emit_hybrid: the hybrid code of section 3.3 instead);
//   k_emit_sum for the fused calls, k_emit's work and, in the same launch,
//              per 1024-coordinate slice the worker-order fp32 sum of
//              Algorithm 1 step 6 over the compacted runs.
//   k_bucket / k_tiles
//              the worker-order fp32 sum of M arbitrary sparse vectors
//              (Algorithm 1, step 6; gs_sparse_aggregate).
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <cfloat>
#include <cmath>
#include <algorithm>
#include <atomic>
#include <cstddef>
#include <cstdint>

#include "gs_decide.cuh"
#include "gs_device.cuh"
#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {

namespace {

#define kInf __int_as_float(0x7F800000)

__device__ __forceinline__ uint32_t mix32(uint32_t h) {
    h ^= h >> 16;
    h *= 0x85EBCA6Bu;
    h ^= h >> 13;
    h *= 0xC2B2AE35u;
    h ^= h >> 16;
    return h;
}

// ---------------------------------------------------------------------------
// Block-ordered append helper: per-thread counts for the kGroupsPerThread
// sub-steps of one step (byte j of `packed` = count of sub-step j), returns
// the offset of each sub-step's first entry of this thread relative to
// `run`, and advances `run` by the block's total.  Order: sub-step, thread.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void ordered_offsets(uint32_t packed, uint32_t (*sh)[32], int& buf, int& run,
                                                int off[kGroupsPerThread]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    uint32_t inc = packed;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += t;
    }
    const uint32_t excl = inc - packed;
    if (lane == 31) sh[buf][warp] = inc;
    __syncthreads();
    int total = 0;
#pragma unroll
    for (int j = 0; j < kGroupsPerThread; ++j) {
        int before = 0, cta = 0;
        for (int w = 0; w < nw; ++w) {
            const int b = (int)((sh[buf][w] >> (8 * j)) & 0xFFu);
            cta += b;
            before += (w < warp) ? b : 0;
        }
        off[j] = run + total + before + (int)((excl >> (8 * j)) & 0xFFu);
        total += cta;
    }
    run += total;
    buf ^= 1;
}

// ---------------------------------------------------------------------------
// Candidate lists of one chunk, built by the whole CTA (any multiple of 32 threads).
//   P: 1 + (x >> 9) 2^-23 < fl32(lam_up32 |g| + 1 + 2^-20).  Since
//      (x >> 9) 2^-23 <= u = x 2^-32, every coordinate kept under a lambda
//      <= lam_up (u < min(lambda |g|, 1)) passes; the 2^-20 slack covers the
//      fp32 rounding of the right-hand side.
//   C: !(|g| < t_c) (NaN and Inf land here, so the l1 sum flags them).
//   s_low: sum of |g| outside C; fp32 pairwise over 16 values, fp64 above.
//   b_low (Algorithm 2 only): the same for g^2.
// Lists are written in ascending coordinate order.
// ---------------------------------------------------------------------------
template <bool kWithC>
__device__ void chunk_candidates(const Layout& Lo, int c, const Chunk& ch, float lam_up32, float t_c, const Lists& Ls,
                                 bool build_p) {
    __shared__ uint32_t shP[2][32];
    __shared__ uint32_t shC[2][32];
    __shared__ double shd[33];
    const int tid = threadIdx.x;
    const int64_t q0 = ch.lo >> 2, q1 = (ch.hi + 3) >> 2;
    const int64_t region = (int64_t)ch.m * Lo.d + ch.lo;
    const uint32_t worker = Lo.worker0 + (uint32_t)ch.m;
    const float pbias = 1.0f + 0x1p-20f;
    double acc = 0.0, acc2 = 0.0;
    const bool sq = kWithC && Ls.b_low != nullptr;
    int runP = 0, runC = 0, bufP = 0, bufC = 0;

    const int nthr = blockDim.x;
    for (int64_t qb = q0; qb < q1; qb += (int64_t)nthr * kGroupsPerThread) {
        float v[kGroupsPerThread][4];
        uint4 w[kGroupsPerThread];
        uint32_t pm = 0, cm = 0;
        float s4[kGroupsPerThread], q4[kGroupsPerThread];
#pragma unroll
        for (int j = 0; j < kGroupsPerThread; ++j) {
            const int64_t q = qb + (int64_t)j * nthr + tid;
            int valid = 0;
            if (q < q1) {
                valid = load_group(Lo, ch.m, q, ch.lo, ch.hi, v[j]);
            } else {
                v[j][0] = v[j][1] = v[j][2] = v[j][3] = 0.0f;
            }
            float m4[4];
            bool need = false;
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                const float a = fabsf(v[j][s]);
                const bool vs = (valid >> s) & 1;
                const bool in_c = vs && !(a < t_c);
                m4[s] = (vs && !in_c) ? a : 0.0f;
                if (in_c) cm |= 1u << (4 * j + s);
                need = need || (vs && a > 0.0f);
            }
            s4[j] = (m4[0] + m4[1]) + (m4[2] + m4[3]);
            q4[j] = (m4[0] * m4[0] + m4[1] * m4[1]) + (m4[2] * m4[2] + m4[3] * m4[3]);
            w[j] = make_uint4(0, 0, 0, 0);
            if (build_p && need) {
                w[j] = group_words(Lo.seed, Lo.step, worker, q);
#pragma unroll
                for (int s = 0; s < 4; ++s) {
                    const float a = fabsf(v[j][s]);
                    const bool vs = (valid >> s) & 1;
                    if (vs && unit_plus_one(word_of(w[j], s)) < fmaf(lam_up32, a, pbias)) pm |= 1u << (4 * j + s);
                }
            }
        }
        acc += (double)((s4[0] + s4[1]) + (s4[2] + s4[3]));
        if (sq) acc2 += (double)((q4[0] + q4[1]) + (q4[2] + q4[3]));

        if (build_p) {
            uint32_t packed = 0;
#pragma unroll
            for (int j = 0; j < kGroupsPerThread; ++j) packed |= (uint32_t)__popc((pm >> (4 * j)) & 0xFu) << (8 * j);
            int off[kGroupsPerThread];
            ordered_offsets(packed, shP, bufP, runP, off);
#pragma unroll
            for (int j = 0; j < kGroupsPerThread; ++j) {
                uint32_t bits = (pm >> (4 * j)) & 0xFu;
                int k = 0;
                const int64_t q = qb + (int64_t)j * nthr + tid;
                while (bits) {
                    const int s = __ffs(bits) - 1;
                    bits &= bits - 1;
                    Ls.p_ent[region + off[j] + k] = make_int2((int32_t)(q * 4 + s), __float_as_int(v[j][s]));
                    ++k;
                }
            }
        }
        if (kWithC) {
            uint32_t packed = 0;
#pragma unroll
            for (int j = 0; j < kGroupsPerThread; ++j) packed |= (uint32_t)__popc((cm >> (4 * j)) & 0xFu) << (8 * j);
            int off[kGroupsPerThread];
            ordered_offsets(packed, shC, bufC, runC, off);
#pragma unroll
            for (int j = 0; j < kGroupsPerThread; ++j) {
                uint32_t bits = (cm >> (4 * j)) & 0xFu;
                int k = 0;
                while (bits) {
                    const int s = __ffs(bits) - 1;
                    bits &= bits - 1;
                    Ls.c_val[region + off[j] + k] = fabsf(v[j][s]);
                    ++k;
                }
            }
        }
    }
    const double tot = block_sum(acc, shd);
    const double tot2 = sq ? block_sum(acc2, shd) : 0.0;
    if (tid == 0) {
        if (sq) Ls.b_low[c] = tot2;
        if (build_p) Ls.p_cnt[c] = runP;
        if (kWithC) {
            Ls.c_cnt[c] = runC;
            Ls.s_low[c] = tot;
        }
    }
    __syncthreads();
}

// Sums over one segment of one worker row, by one CTA: K = #{|g| >= acap},
// su = sum of the other |g| (NaN / Inf propagate into su when acap is NaN).
__device__ void segment_stats(const Layout& Lo, int m, int64_t lo, int64_t hi, float acap, double& K, double& su,
                              double* shd) {
    const int64_t q0 = lo >> 2, q1 = (hi + 3) >> 2;
    double acc = 0.0, cnt = 0.0;
    const int nthr = blockDim.x;
    for (int64_t qb = q0; qb < q1; qb += (int64_t)nthr * kGroupsPerThread) {
        float s4[kGroupsPerThread];
        int k = 0;
#pragma unroll
        for (int j = 0; j < kGroupsPerThread; ++j) {
            const int64_t q = qb + (int64_t)j * nthr + threadIdx.x;
            float v[4] = {0.f, 0.f, 0.f, 0.f};
            int valid = 0;
            if (q < q1) valid = load_group(Lo, m, q, lo, hi, v);
            float m4[4];
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                const float a = fabsf(v[s]);
                const bool vs = (valid >> s) & 1;
                const bool capped = vs && (a >= acap);
                k += capped ? 1 : 0;
                m4[s] = (vs && !capped) ? a : 0.0f;
            }
            s4[j] = (m4[0] + m4[1]) + (m4[2] + m4[3]);
        }
        acc += (double)((s4[0] + s4[1]) + (s4[2] + s4[3]));
        cnt += (double)k;
    }
    su = block_sum(acc, shd);
    K = block_sum(cnt, shd);
}

// ---------------------------------------------------------------------------
// Block-wide helpers over kThreads threads.
// ---------------------------------------------------------------------------
// Sum of two doubles over the block (one reduction); every thread gets both.

// Exclusive scan of cnt[0..n) into pre[0..n]; pre[n] = total.  `pre` may live
// in shared or global memory (written and read back by this block only).
__device__ void block_exclusive_scan(const int32_t* __restrict__ cnt, int n, int32_t* pre, int* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int run = 0;
    for (int b = 0; b < n; b += blockDim.x) {
        const int i = b + threadIdx.x;
        const int v = i < n ? cnt[i] : 0;
        int inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xFFFFFFFFu, inc, o);
            if (lane >= o) inc += t;
        }
        if (lane == 31) sh[warp] = inc;
        __syncthreads();
        if (warp == 0) {
            int t = lane < nw ? sh[lane] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(0xFFFFFFFFu, t, o);
                if (lane >= o) t += u;
            }
            sh[lane] = t;
        }
        __syncthreads();
        const int before = warp > 0 ? sh[warp - 1] : 0;
        if (i < n) pre[i] = run + before + inc - v;
        run += sh[nw - 1];
        __syncthreads();
    }
    if (threadIdx.x == 0) pre[n] = run;
    __syncthreads();
}

// Largest k in [0, n) with pre[k] <= e (pre ascending, pre[0] = 0).
__device__ __forceinline__ int upper_slot(const int32_t* pre, int n, int e) {
    int a = 0, b = n - 1;
    while (a < b) {
        const int mid = (a + b + 1) >> 1;
        if (pre[mid] <= e) a = mid; else b = mid - 1;
    }
    return a;
}

// ---------------------------------------------------------------------------
// k_bound: one CTA per segment.
// ---------------------------------------------------------------------------
constexpr double kBoundZ = 5.0;
constexpr double kBoundZs = 8.0;         // standard errors of the spread-based margin
constexpr double kBoundFloor = 0.04;     // smallest relative margin

// Sum of two floats over the block; every thread gets both.
__device__ __forceinline__ float2 block_sum2f(float a, float b, float2* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
        b += __shfl_xor_sync(0xFFFFFFFFu, b, o);
    }
    __syncthreads();
    if (lane == 0) sh[warp] = make_float2(a, b);
    __syncthreads();
    if (warp == 0) {
        float2 t = lane < nw ? sh[lane] : make_float2(0.0f, 0.0f);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            t.x += __shfl_xor_sync(0xFFFFFFFFu, t.x, o);
            t.y += __shfl_xor_sync(0xFFFFFFFFu, t.y, o);
        }
        if (lane == 0) sh[32] = t;
    }
    __syncthreads();
    return sh[32];
}

// Three float sums over the block at once; every thread receives them (x, y, z).
__device__ __forceinline__ float4 block_sum3f(float a, float b, float c, float4* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
        b += __shfl_xor_sync(0xFFFFFFFFu, b, o);
        c += __shfl_xor_sync(0xFFFFFFFFu, c, o);
    }
    __syncthreads();
    if (lane == 0) sh[warp] = make_float4(a, b, c, 0.0f);
    __syncthreads();
    if (warp == 0) {
        float4 t = lane < nw ? sh[lane] : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            t.x += __shfl_xor_sync(0xFFFFFFFFu, t.x, o);
            t.y += __shfl_xor_sync(0xFFFFFFFFu, t.y, o);
            t.z += __shfl_xor_sync(0xFFFFFFFFu, t.z, o);
        }
        if (lane == 0) sh[32] = t;
    }
    __syncthreads();
    return sh[32];
}

// The bound only steers how many candidates the streaming pass keeps, so it
// is estimated in fp32: a stratified sample of |g| (a run of kBoundRun
// consecutive coordinates, at a hashed position, from each of ns / kBoundRun
// equal strata) and Algorithm 3 run on the sample until its scaling factor
// is within 1e-5 of 1.
constexpr int kBoundCTAs = 8;
constexpr int kBoundCtaThreads = 1024;
constexpr int kBoundRun = 8;             // consecutive coordinates read per stratum
constexpr int kBoundWarpMax = 1024;      // samples up to which warp 0 alone runs the fixed point

// Algorithm 3 run to its fixed point (in fp32) on a sample of |g| in shared
// memory, and the upper bound on lambda it gives, written to the segment's
// parameters by thread t == 0.  kWarp: one warp alone (t = lane, shuffle
// sums); else the whole CTA (t = tid, block sums).  whole: the sample is the
// whole segment (the fixed point is then Algorithm 3 itself, whose iterates
// never pass it, so a 1% margin covers the fp32 rounding).
template <bool kWarp>
__device__ __forceinline__ void bound_from_sample(SegParam& P, const float* sa, int ns, double kappa, bool whole,
                                                  int t, float2* sh2, float4* sh4) {
    const int nthr = kWarp ? 32 : (int)blockDim.x;
    float ls = 0.0f;
    for (int k = t; k < ns; k += nthr) ls += sa[k];
    const float S = kWarp ? warp_sum(ls) : block_sum2f(ls, 0.0f, sh2).x;
    const float budget = (float)(kappa * (double)ns);
    float lam = S > 0.0f ? budget / S : 0.0f;
    float K = 0.0f, Su = S;
    bool take_all = !(S > 0.0f) || !(lam < kInf);
    float Sq = 0.0f;   // sum of squares of the uncapped sample values (for the margin)
    for (int it = 0; it < 32 && !take_all; ++it) {
        const float acap = 1.0f / lam;
        float su = 0.0f, kc = 0.0f, sq = 0.0f;
        for (int k = t; k < ns; k += nthr) {
            const float x = sa[k];
            if (x >= acap) kc += 1.0f; else { su += x; sq += x * x; }
        }
        const float4 r = kWarp ? make_float4(warp_sum(kc), warp_sum(su), warp_sum(sq), 0.0f)
                               : block_sum3f(kc, su, sq, sh4);
        K = r.x;
        Su = r.y;
        Sq = r.z;
        if (!(Su > 0.0f)) { take_all = true; break; }
        const float c = (budget - K) / (lam * Su);
        if (!(c > 1.0f + 1e-5f)) break;
        lam *= c;
    }
    if (t == 0) {
        P.done = 0;
        P.w_done = 0;
        P.next_chunk = 0;
        const float e = take_all ? 0.0f : lam * Su / budget;  // uncapped share of the budget
        if (take_all || K >= budget || !(lam > 0.0f)) {
            P.lam_up = (double)kInf;
            P.lam_up32 = kInf;
            P.t_c = 0.0f;
            P.flags = kSegTakeAll;
        } else {
            // A count-based bound on the sample's error, tightened by the sample's
            // own spread: lambda = (kappa d - K) / S_u at the fixed point, so its
            // relative error is about that of S_u (std of a sum of the
            // uncapped values) and of kappa d - K (binomial K).  A sample that
            // caught large values also has a large spread, which keeps the bound
            // safe for heavy tails; a violated bound only costs the exact fallback.
            // (fp32 throughout: a heuristic, and fp64 is slow on this part)
            const float kns = (float)kappa * (float)ns;
            float margin = 1.0f + (float)kBoundZ * rsqrtf(kns) / fmaxf(e, 1.0f / 16.0f);
            const float nu = (float)ns - K;
            if (nu > 1.0f && Su > 0.0f && isfinite(Sq)) {
                const float mean = Su / nu;
                const float var = fmaxf(Sq / nu - mean * mean, 0.0f);
                const float rel_s = sqrtf(var * nu) / Su;
                const float room = kns - K;
                const float rel_k = room > 0.0f ? sqrtf(K) / room : 1.0f;
                margin = fminf(margin, 1.0f + fmaxf((float)kBoundFloor,
                                                    (float)kBoundZs * sqrtf(rel_s * rel_s + rel_k * rel_k)));
            }
            margin = fminf(margin, 64.0f);
            if (whole) margin = 1.01f;
            // lam_up32 rounded up and t_c rounded down keep both lists supersets;
            // the fp64 bound is lam_up32 itself.
            const float up32 = __fmul_ru(lam, margin);
            P.lam_up32 = up32;
            P.lam_up = (double)up32;
            P.t_c = __fmul_rd(__frcp_rd(up32), 1.0f - 0x1p-20f);
            P.flags = 0;
        }
    }
}

// One thread-block cluster of kCTAs CTAs per segment (kBoundCTAs, or one for
// layer-wise calls): the CTAs share the sample's random loads and store the
// |g| values straight into rank 0's shared memory (DSMEM); rank 0 then runs
// Algorithm 3 to its fixed point on the sample alone, with block-wide sums.
template <int kCTAs>
__global__ void __cluster_dims__(kCTAs, 1, 1) __launch_bounds__(kBoundCtaThreads, 2)
    k_bound(Layout Lo, SegParam* sp, double kappa, int ns, int force_exact, int short_per_cta) {
    grid_dep_wait();
    // The streaming pass may launch now: it only loads g (an input of the
    // call) until its own wait for this grid.
    grid_dep_launch();
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    extern __shared__ __align__(16) float sa[];   // rank 0: all ns samples
    __shared__ float2 sh2[33];
    __shared__ float4 sh4[33];
    const int rank = (int)cluster.block_rank();
    const int tid = threadIdx.x;
    int s = blockIdx.x / kCTAs;
    if (kCTAs == 1 && short_per_cta > 0) {
        // Layer-wise calls: a CTA for each worker's copy of each long segment
        // (bnd_seg's first bnd_long), then short_per_cta short segments (at
        // most kBoundWarpMax values) to a CTA, one per warp, each taken whole
        // into the warp's own slice of shared memory.
        const int n_long = Lo.M * Lo.bnd_long;
        if (s < n_long) {
            s = (s % Lo.M) * Lo.L + Lo.bnd_seg[s / Lo.M];
        } else {
            const int w = tid >> 5, lane = tid & 31;
            const int t = (s - n_long) * short_per_cta + w;
            if (w >= short_per_cta || t >= Lo.M * (Lo.L - Lo.bnd_long)) return;
            const int ss = (t % Lo.M) * Lo.L + Lo.bnd_seg[Lo.bnd_long + t / Lo.M];
            int m, l, c0, c1;
            int64_t lo, hi;
            seg_range(Lo, ss, m, l, lo, hi, c0, c1);
            const int len = (int)(hi - lo);
            SegParam& Q = sp[ss];
            float* ws = sa + w * kBoundWarpMax;
            if (!force_exact) {
                for (int e = lane; e < len; e += 32) {
                    float x = fabsf(load_one(Lo, m, lo + e));
                    if (!(x < kInf)) x = 0.0f;  // non-finite values are reported by the solve
                    ws[e] = x;
                }
                __syncwarp();
                bound_from_sample<true>(Q, ws, len, kappa, true, lane, sh2, sh4);
            } else if (lane == 0) {
                Q.done = 0;
                Q.w_done = 0;
                Q.next_chunk = 0;
                Q.lam_up = (double)kInf;
                Q.lam_up32 = kInf;
                Q.t_c = 0.0f;
                Q.flags = kSegTakeAll;
            }
            return;
        }
    }
    int m, l, c0, c1;
    int64_t lo, hi;
    seg_range(Lo, s, m, l, lo, hi, c0, c1);
    const int64_t len = hi - lo;
    SegParam& P = sp[s];
    if (force_exact) {
        // Exact mode: every coordinate is a candidate.
        if (rank == 0 && tid == 0) {
            P.done = 0;
            P.w_done = 0;
            P.next_chunk = 0;
            P.lam_up = (double)kInf;
            P.lam_up32 = kInf;
            P.t_c = 0.0f;
            P.flags = kSegTakeAll;
        }
        return;   // uniform over the cluster: no CTA reaches a cluster barrier
    }
    float* dst = cluster.map_shared_rank(sa, 0);
    // A segment no longer than the sample is taken whole: the fixed point below
    // is then Algorithm 3 itself (in fp32), whose iterates never pass the fixed
    // point, so a 1% margin covers the fp32 rounding.
    const bool whole = len <= ns;
    if (whole) {
        for (int e = rank * kBoundCtaThreads + tid; e < (int)len; e += kCTAs * kBoundCtaThreads) {
            float x = fabsf(load_one(Lo, m, lo + e));
            if (!(x < kInf)) x = 0.0f;  // non-finite values are reported by the solve
            dst[e] = x;
        }
        ns = (int)len;
    }
    // ns / 8 strata; from each, 8 consecutive coordinates starting at a
    // random multiple of 8 (one 32-byte sector of fp32 g).
    const int per = whole ? 0 : ns / (kBoundRun * kCTAs);      // strata of this CTA
    const int nst = per * kCTAs;
    if (!whole) ns = nst * kBoundRun;                               // samples actually drawn
    const int64_t q = whole ? 1 : len / nst;                        // stratum width (the last one takes the rest)
    const int64_t q_last = whole ? 1 : len - (int64_t)(nst - 1) * q;
    const uint32_t hs = mix32((uint32_t)s + 0x68E31DA4u);
    // One thread per stratum: its run's start is found once, and a run that
    // lies inside the segment on a 16-byte grid is read with vector loads
    // (its flat start is a multiple of kBoundRun = 8 elements).
    const bool vec = (reinterpret_cast<uintptr_t>(Lo.g) & 15u) == 0;
    for (int kk = tid; kk < per; kk += kBoundCtaThreads) {
        const int k = rank * per + kk;                              // stratum
        const uint32_t h = mix32((uint32_t)k * 0x9E3779B9u ^ hs);
        const int64_t width = k == nst - 1 ? q_last : q;            // >= kBoundRun since len > ns
        const int64_t runs = width / kBoundRun;
        int64_t start = lo + (int64_t)k * q + (int64_t)(h % (uint32_t)runs) * kBoundRun;
        start -= (start + (int64_t)m * Lo.d) % kBoundRun;           // align the run to the flat index
        if (start < lo + (int64_t)k * q) start += kBoundRun;
        float x[kBoundRun];
        if (vec && start + kBoundRun <= hi) {
            const int64_t flat = (int64_t)m * Lo.d + start;
            if (Lo.dtype == 0) {
                const float4* p4 = reinterpret_cast<const float4*>(static_cast<const float*>(Lo.g) + flat);
                const float4 a = p4[0], b = p4[1];
                x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
                x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
            } else {
                const uint4 t = *reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(Lo.g) + flat);
                const uint32_t w4[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    x[2 * r] = bf16_bits_to_float(w4[r] & 0xFFFFu);
                    x[2 * r + 1] = bf16_bits_to_float(w4[r] >> 16);
                }
            }
        } else {
#pragma unroll
            for (int r = 0; r < kBoundRun; ++r) x[r] = load_one(Lo, m, min(start + r, hi - 1));
        }
#pragma unroll
        for (int r = 0; r < kBoundRun; ++r) {
            float a = fabsf(x[r]);
            if (!(a < kInf)) a = 0.0f;  // non-finite values are reported by the solve
            x[r] = a;
        }
        float4* d4 = reinterpret_cast<float4*>(dst + (size_t)k * kBoundRun);
        d4[0] = make_float4(x[0], x[1], x[2], x[3]);
        d4[1] = make_float4(x[4], x[5], x[6], x[7]);
    }
    cluster.sync();   // the sample is complete in rank 0; nobody touches another CTA's memory after this
    if (rank != 0) return;

    // A sample of at most kBoundWarpMax values (a short segment taken whole)
    // is iterated by warp 0 alone with shuffle sums: no block barrier per
    // iteration.  The other warps leave; nothing below waits for them.
    if (ns <= kBoundWarpMax) {
        if (tid < 32) bound_from_sample<true>(P, sa, ns, kappa, whole, tid, sh2, sh4);
        return;
    }
    bound_from_sample<false>(P, sa, ns, kappa, whole, tid, sh2, sh4);
}

// ---------------------------------------------------------------------------
// k_stream (generic loads; any alignment): the single pass over g.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_stream(Layout Lo, const SegParam* __restrict__ sp, Lists Ls,
                                                     int n_chunks, int build_p) {
    grid_dep_wait();
    for (int c = blockIdx.x; c < n_chunks; c += gridDim.x) {
        const Chunk ch = decode_chunk(Lo, c);
        chunk_candidates<true>(Lo, c, ch, sp[ch.seg].lam_up32, sp[ch.seg].t_c, Ls, build_p != 0);
    }
}

// ---------------------------------------------------------------------------
// k_solve: one CTA per segment.  Algorithm 3 in the lambda form of
// Proposition 1: lambda_0 = kappa d / S (step 3); K = #{fl64(lambda |g|) >= 1}
// (capped, outside the active set of step 5); A = lambda * (uncapped l1 mass)
// = sum_{i in I} p_i; c = (kappa d - K) / A (step 6); stop if c <= 1 (step 7);
// lambda <- c lambda (step 8).  K and the uncapped mass come from (S_low, C):
// every coordinate any lambda_j <= lam_up caps is in C.
// ---------------------------------------------------------------------------
constexpr int kSolveSmemChunks = 8192;   // chunk-prefix entries kept in shared memory
constexpr int kSolveSmemC = 12288;       // candidate values kept in shared memory
constexpr int kSolvePer = 4;             // chunks per thread of the one-round start (segments <= 1024 chunks)
// Long segments (budgets above 2^20) are solved by a cluster of kSolveCTAs
// CTAs of kSolveClusterThreads threads: their walks over a C of millions of
// values wait on L2, and 32 warps per SM hide that where 8 did not; twelve
// 1024-thread CTAs is the largest cluster of which eight are resident at once.
constexpr int kSolveCTAs = 12;
constexpr int kSolveClusterThreads = 1024;
constexpr int kSolveMaxThreads = 1024;   // k_solve runs on kThreads threads alone, or kSolveClusterThreads in a cluster

// Exclusive prefix of v over the block (any blockDim <= 1024) and the total.
__device__ __forceinline__ int block_scan_total(int v, int* sh, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += t;
    }
    if (lane == 31) sh[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int t = lane < nw ? sh[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xFFFFFFFFu, t, o);
            if (lane >= o) t += u;
        }
        sh[lane] = t;
    }
    __syncthreads();
    const int before = warp > 0 ? sh[warp - 1] : 0;
    total = sh[nw - 1];
    __syncthreads();
    return before + inc - v;
}

struct CView {
    const float* smem;       // compacted candidates (when they fit in shared memory), else NULL
    const float* gbase;      // c_val + region of the segment's first chunk
    const int32_t* pre;      // chunk prefix over the segment's chunks
    int nch;
    int nC;
    __device__ __forceinline__ float at(int e) const {
        if (smem) return smem[e];
        const int k = upper_slot(pre, nch + 1, e);
        return gbase[(int64_t)k * kChunk + (e - pre[k])];
    }
};

// c_stats for one warp: every lane receives (hi, lo, count).
__device__ __forceinline__ void warp_c_stats(const CView& C, float acap, float& hi, float& lo, int& k) {
    hi = 0.0f;
    lo = 0.0f;
    k = 0;
    for (int e = threadIdx.x & 31; e < C.nC; e += 32) {
        const float a = C.at(e);
        if (a >= acap) ++k; else two_sum_add(hi, lo, a);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xFFFFFFFFu, hi, o);
        const float ol = __shfl_xor_sync(0xFFFFFFFFu, lo, o);
        df_add(hi, lo, oh, ol);
        k += __shfl_xor_sync(0xFFFFFFFFu, k, o);
    }
}

// Sum of one double per thread, added by warp 0 alone (fixed order); every
// thread receives it.  `sh` holds blockDim.x + 1 doubles.
__device__ __forceinline__ double warp0_sum_double(double v, double* sh) {
    sh[threadIdx.x] = v;
    __syncthreads();
    if (threadIdx.x < 32) {
        double t = 0.0;
        for (int i = threadIdx.x; i < blockDim.x; i += 32) t += sh[i];
        t = warp_sum(t);
        if (threadIdx.x == 0) sh[blockDim.x] = t;
    }
    __syncthreads();
    return sh[blockDim.x];
}

// Exact fallback of k_solve for one segment, by the whole CTA: every sum of
// Algorithm 3 straight from g, then the segment's P lists rebuilt for the
// final lambda (sparsify calls only).  Out of line: it almost never runs, and
// its code (the candidate builder included) would otherwise crowd the
// instruction cache of the common path.
__device__ __noinline__ void solve_exact(const Layout& Lo, const Lists& Ls, int m, int64_t lo, int64_t hi, int c0,
                                         int c1, double budget, int iters, double* shd, double& S, double& lam,
                                         double& K, double& Su, int& j) {
    __shared__ float s_acap;
    double k0;
    segment_stats(Lo, m, lo, hi, __int_as_float(0x7FC00000), k0, S, shd);
    lam = S > 0.0 ? budget / S : 0.0;
    j = 0;
    K = 0.0;
    Su = S;
    if (lam > 0.0) {
        while (j < iters) {
            if (threadIdx.x == 0) s_acap = cap_threshold_call(lam);
            __syncthreads();
            segment_stats(Lo, m, lo, hi, s_acap, K, Su, shd);
            const double A = lam * Su;
            if (A == 0.0) break;
            const double cc = (budget - K) / A;
            if (!(cc > 1.0)) break;
            lam = cc * lam;
            ++j;
        }
        if (threadIdx.x == 0) s_acap = cap_threshold_call(lam);
        __syncthreads();
        segment_stats(Lo, m, lo, hi, s_acap, K, Su, shd);
    }
    const float up32 = lam > 0.0 ? __double2float_ru(lam) : 0.0f;
    for (int c = c0; Ls.p_ent != nullptr && c < c1; ++c) {
        const Chunk ch = decode_chunk(Lo, c);
        chunk_candidates<false>(Lo, c, ch, up32, 0.0f, Ls, true);
    }
}

// Launched with clusters of 1 or kSolveCTAs CTAs per segment (block x / cluster
// size = segment).  Small C: the cluster's rank 0 solves alone.  Large C: every
// CTA of the cluster walks a share of the segment's chunks in each pass and the
// CTA partials are combined through distributed shared memory in rank order.
__global__ void __launch_bounds__(kSolveMaxThreads) k_solve(Layout Lo, SegParam* sp, Lists Ls, double kappa, int iters,
                                                    int force_exact, int* status, gs_info_dev* info,
                                                    int cap_chunks, int cap_c) {
    grid_dep_wait();
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int ncta = (int)cluster.num_blocks(), rank = (int)cluster.block_rank();
    // Dynamic shared memory, sized by the launcher for the largest segment:
    // cap_chunks chunk-prefix entries (+4), then cap_c candidate values.
    extern __shared__ unsigned char dsm[];
    int32_t* spre = reinterpret_cast<int32_t*>(dsm);
    float* sc = reinterpret_cast<float*>(dsm + sizeof(int32_t) * (cap_chunks + 4));
    __shared__ double shd[33];
    __shared__ int shi[33];
    __shared__ float s_acap;
    __shared__ double shdd[kSolveMaxThreads + 1];
    __shared__ double s_S, s_lam, s_K, s_Su;
    __shared__ int s_go, s_j, s_fresh;
    __shared__ float4 sh4[33];
    __shared__ float4 xch[2];           // this CTA's partial (hi, lo, count) of a pass, double-buffered
    const int s = blockIdx.x / ncta, tid = threadIdx.x;
    const int lane = tid & 31, warp = tid >> 5;
    int m, l, c0, c1;
    int64_t lo, hi;
    seg_range(Lo, s, m, l, lo, hi, c0, c1);
    const int64_t len = hi - lo;
    const double budget = kappa * (double)len;
    const double lam_up = sp[s].lam_up;
    int flags = sp[s].flags & kSegTakeAll;

    // Candidate view: chunk prefix (shared or global scratch), values gathered to shared memory when they fit.
    const int nch = c1 - c0;
    int32_t* pre = nch <= cap_chunks ? spre : Ls.c_pre + c0 + s;
    CView C;
    C.pre = pre;
    C.nch = nch;
    C.gbase = Ls.c_val + (int64_t)m * Lo.d + lo;
    C.smem = nullptr;
    double sl = 0.0;
    const int nthr = blockDim.x, nwarp = nthr >> 5;
    if (nch <= kSolvePer * nthr) {
        // Every chunk count and l1 partial in one round of loads (kSolvePer
        // consecutive chunks per thread), one block scan, and each thread
        // copies its own chunks' values of C.
        int cnt[kSolvePer];
        int tot = 0;
#pragma unroll
        for (int j = 0; j < kSolvePer; ++j) {
            const int c = c0 + kSolvePer * tid + j;
            cnt[j] = c < c1 ? Ls.c_cnt[c] : 0;
            sl += c < c1 ? Ls.s_low[c] : 0.0;
            tot += cnt[j];
        }
        int total;
        int run = block_scan_total(tot, shi, total);
#pragma unroll
        for (int j = 0; j < kSolvePer; ++j) {
            if (kSolvePer * tid + j < nch) pre[kSolvePer * tid + j] = run;
            run += cnt[j];
        }
        if (tid == 0) pre[nch] = total;
        C.nC = total;
        if (total <= cap_c) {
            // The values of C copied to shared memory.  Many sparse chunks (at
            // least two per thread, 32 values or fewer on average): each thread
            // copies its own, their loads being independent.  Otherwise (few or
            // dense chunks; a short segment takes every coordinate): a warp per
            // chunk, or the whole CTA per chunk when there are few.
            if (nch >= 2 * nthr && total <= 32 * nch) {
                int at = run - tot;
#pragma unroll
                for (int j = 0; j < kSolvePer; ++j) {
                    const int64_t base = (int64_t)(kSolvePer * tid + j) * kChunk;
                    for (int v = 0; v < cnt[j]; ++v) sc[at + v] = C.gbase[base + v];
                    at += cnt[j];
                }
            } else {
                __syncthreads();   // pre[] complete
                if (nch <= nwarp) {
                    for (int q = 0; q < nch; ++q) {
                        const int b = pre[q], n = pre[q + 1] - b;
                        for (int v = tid; v < n; v += blockDim.x) sc[b + v] = C.gbase[(int64_t)q * kChunk + v];
                    }
                } else {
                    for (int q = warp; q < nch; q += nwarp) {
                        const int b = pre[q], n = pre[q + 1] - b;
                        for (int v = lane; v < n; v += 32) sc[b + v] = C.gbase[(int64_t)q * kChunk + v];
                    }
                }
            }
            C.smem = sc;
        }
        __syncthreads();
    } else {
        block_exclusive_scan(Ls.c_cnt + c0, nch, pre, shi);
        C.nC = pre[nch];
        if (C.nC <= cap_c) {
            for (int e = tid; e < C.nC; e += blockDim.x) sc[e] = C.at(e);
            __syncthreads();
            C.smem = sc;
        }
        for (int c = c0 + tid; c < c1; c += blockDim.x) sl += Ls.s_low[c];
    }
    // fp64 is slow on this part and C is small: the l1 partials are summed and
    // Algorithm 3 is iterated by warp 0 alone (warp shuffles only; every lane
    // carries the same scalars), then the result is broadcast.
    const double S_low = warp0_sum_double(sl, shdd);
    if (C.smem == nullptr) {
        // Large C: passes over the segment's chunks shared by the cluster.
        int buf = 0;
        auto stats = [&](float acap, float& rh, float& rl, int& rk) {
            float hi_ = 0.0f, lo_ = 0.0f;
            int k_ = 0;
            for (int q = rank * nwarp + warp; q < nch; q += ncta * nwarp) {
                const int n = pre[q + 1] - pre[q];
                const float* src = C.gbase + (int64_t)q * kChunk;
                for (int e = lane; e < n; e += 32) {
                    const float a = src[e];
                    if (a >= acap) ++k_; else two_sum_add(hi_, lo_, a);
                }
            }
            block_sum_df(hi_, lo_, k_, sh4);
            if (tid == 0) xch[buf] = make_float4(hi_, lo_, __int_as_float(k_), 0.0f);
            cluster.sync();
            rh = 0.0f;
            rl = 0.0f;
            rk = 0;
            for (int r = 0; r < ncta; ++r) {
                const float4 v = *cluster.map_shared_rank(&xch[buf], r);
                df_add(rh, rl, v.x, v.y);
                rk += __float_as_int(v.z);
            }
            buf ^= 1;
        };
        float rh, rl;
        int rk;
        stats(__int_as_float(0x7FC00000), rh, rl, rk);
        if (tid == 0) {
            const double S0 = S_low + ((double)rh + (double)rl);
            const bool run = isfinite(S0) && force_exact == 0 && S0 > 0.0;
            s_S = S0;
            s_lam = run ? budget / S0 : 0.0;
            s_go = run && iters > 0 ? 1 : 0;
            s_fresh = 1;
            s_j = 0;
            s_acap = cap_threshold_call(s_lam);
            s_K = 0.0;
            s_Su = S0;
        }
        __syncthreads();
        const bool run = isfinite(s_S) && force_exact == 0 && s_S > 0.0;
        if (run) {
            s_fresh = 0;   // the first stats were taken with no threshold
            __syncthreads();
            while (s_go) {
                stats(s_acap, rh, rl, rk);
                if (tid == 0) {
                    double lv = s_lam;
                    int go = 0, fresh = 1;
                    const double A = lv * (S_low + ((double)rh + (double)rl));
                    if (A != 0.0) {
                        const double cc = (budget - (double)rk) / A;
                        if (cc > 1.0) {
                            lv = cc * lv;
                            ++s_j;
                            go = s_j < iters;
                            fresh = 0;
                            s_acap = cap_threshold_call(lv);
                        }
                    }
                    s_lam = lv;
                    s_go = go;
                    s_fresh = fresh;
                }
                __syncthreads();
            }
            if (!s_fresh) stats(s_acap, rh, rl, rk);
            if (tid == 0) {
                s_K = (double)rk;
                s_Su = S_low + ((double)rh + (double)rl);
                s_go = s_lam > lam_up ? 1 : 0;    // exact fallback needed
            }
        } else if (tid == 0) {
            s_go = force_exact != 0 ? 1 : 0;
        }
        cluster.sync();   // no CTA may leave while a peer still reads its partials
        if (rank != 0) return;
        __syncthreads();
    } else if (rank != 0) {
        return;           // small C: rank 0 solves alone (uniform over the cluster)
    } else if (tid < 32) {
        float rh, rl;
        int rk;
        warp_c_stats(C, __int_as_float(0x7FC00000), rh, rl, rk);
        const double S0 = S_low + ((double)rh + (double)rl);
        double lv = 0.0;
        int jj = 0;
        bool ex = force_exact != 0;
        float acap = __int_as_float(0x7F800000);
        if (isfinite(S0) && !ex && S0 > 0.0) {
            lv = budget / S0;
            acap = warp_cap_threshold(lv);
            bool fresh = false;   // (rh, rl, rk) are the stats at acap
            while (jj < iters) {
                warp_c_stats(C, acap, rh, rl, rk);
                fresh = true;
                const double A = lv * (S_low + ((double)rh + (double)rl));
                if (A == 0.0) break;
                const double cc = (budget - (double)rk) / A;
                if (!(cc > 1.0)) break;
                lv = cc * lv;
                ++jj;
                acap = warp_cap_threshold(lv);
                fresh = false;
            }
            if (!fresh) warp_c_stats(C, acap, rh, rl, rk);
            // The lists are exact only while lambda stays within the bound.
            if (lv > lam_up) ex = true;
        }
        if (tid == 0) {
            s_S = S0;
            s_lam = lv;
            s_acap = acap;   // the threshold of lv (reused for the segment's parameters)
            s_j = jj;
            s_go = ex ? 1 : 0;
            s_K = (double)rk;
            s_Su = S_low + ((double)rh + (double)rl);
        }
    }
    __syncthreads();
    double S = s_S;
    double lam = s_lam, K = s_K, Su = s_Su;
    int j = s_j;
    bool exact = s_go != 0;
    if (!isfinite(S)) {
        flags |= kSegNonfinite;
        if (tid == 0) atomicOr(status, kStNonfinite);
    }

    if (exact && isfinite(S)) {
        flags |= kSegExact;
        solve_exact(Lo, Ls, m, lo, hi, c0, c1, budget, iters, shd, S, lam, K, Su, j);
    }
    // The solve's own threshold holds for its final lambda, except after the
    // exact fallback (or a non-finite sum, where lambda is 0).
    float a_cap = s_acap;
    if ((flags & kSegExact) || !isfinite(S) || !(lam > 0.0)) {
        if (tid < 32) a_cap = warp_cap_threshold(lam);
        else a_cap = 0.0f;   // unused
    }

    if (tid == 0) {
        SegParam& P = sp[s];
        P.lam = lam;
        P.lam32 = (float)lam;
        P.a_cap = a_cap;
        P.inv_lam32 = lam > 0.0 ? (float)(1.0 / lam) : 0.0f;
        P.l1 = S;
        P.capped = (long long)K;
        P.sum_p = lam > 0.0 ? K + lam * Su : 0.0;
        P.iters_run = j;
        P.flags = flags;
        if (info) {
            info[s].lambda = lam;
            info[s].sum_p = P.sum_p;
            info[s].capped = (int64_t)K;
            info[s].iters_run = j;
            info[s].flags = (flags & kSegExact) ? 1 : 0;
        }
    }
}

// ---------------------------------------------------------------------------
// The hybrid code's compaction, in two steps with no waits between chunks:
//   k_decide       one warp per chunk: draws each candidate's Philox word
//                  again, records its decision as one bit (a warp ballot per
//                  32 candidates) and the chunk's kept counts (all, and
//                  those with p = 1); the last warp to finish a worker's
//                  chunks turns its counts into output offsets;
//   k_emit_hybrid  one warp per chunk: Q_A and Q_B at their offsets.
// ---------------------------------------------------------------------------
constexpr int kEmitWarps = 8;
constexpr int kEmitBatch = 4;                            // candidate rounds whose loads are in flight together
constexpr int kBitWords = kChunk / 32;                   // decision words per chunk
constexpr int kScanPer = 8;                              // chunk counts per lane per step of the worker scan
// Resident CTAs per SM k_decide is compiled for (<= 42 registers a thread):
// its warps mostly wait on candidate loads, so more of them hide more.
constexpr int kDecideBlocks = 6;

// One warp turns n counts into their exclusive prefix in place (kScanPer
// counts per lane per step, read past L1) and returns the total.
__device__ __forceinline__ long long warp_scan_counts(int32_t* ko, int n, int lane) {
    long long carry = 0;
    for (int base = 0; base < n; base += 32 * kScanPer) {
        int v[kScanPer];
        int tot = 0;
#pragma unroll
        for (int j = 0; j < kScanPer; ++j) {
            const int i = base + lane * kScanPer + j;
            v[j] = i < n ? __ldcg(ko + i) : 0;
            tot += v[j];
        }
        int inc = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xFFFFFFFFu, inc, o);
            if (lane >= o) inc += u;
        }
        long long run = carry + (inc - tot);
#pragma unroll
        for (int j = 0; j < kScanPer; ++j) {
            const int i = base + lane * kScanPer + j;
            if (i < n) ko[i] = (int32_t)run;
            run += v[j];
        }
        carry += __shfl_sync(0xFFFFFFFFu, inc, 31);
    }
    return carry;
}

// Word j (0..3) of group q alone: rounds 1-9 of PhiloxStream::words_after,
// and of the last round only the product that word comes from (words 0 and 1
// are the high and low halves of 0xCD9E8D57 c2, words 2 and 3 those of
// 0xD2511F53 c0).
__device__ __forceinline__ uint32_t philox_word(const PhiloxStream& ph, uint32_t q, int j) {
    const uint64_t m0 = (uint64_t)0xD2511F53u * (uint64_t)q;
    uint32_t c0 = ph.x0, c1 = ph.x1, c2 = (uint32_t)(m0 >> 32) ^ ph.c3k1, c3 = (uint32_t)m0;
#pragma unroll
    for (int r = 1; r < 9; ++r) {
        const uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
        const uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
        const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ ph.rk0[r];
        const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ ph.rk1[r];
        c1 = (uint32_t)p1;
        c3 = (uint32_t)p0;
        c0 = n0;
        c2 = n2;
    }
    const bool from_c0 = (j & 2) != 0;
    const uint64_t p = (uint64_t)(from_c0 ? 0xD2511F53u : 0xCD9E8D57u) * (uint64_t)(from_c0 ? c0 : c2);
    if (j & 1) return (uint32_t)p;
    return (uint32_t)(p >> 32) ^ (from_c0 ? (c3 ^ ph.rk1[9]) : (c1 ^ ph.rk0[9]));
}

__device__ __forceinline__ Decider chunk_decider(const SegParam& P) {
    Decider dd;
    dd.lam = P.lam;
    dd.lam32 = P.lam32;
    dd.a_cap = P.a_cap;
    dd.inv_lam32 = P.inv_lam32;
    return dd;
}

__global__ void __launch_bounds__(kEmitWarps * 32, kDecideBlocks) k_decide(const __grid_constant__ Layout Lo, SegParam* sp,
                                                            const __grid_constant__ Lists Ls, int n_chunks,
                                                            int32_t* nnz, int32_t* n_a, int32_t* n_b, int64_t cap,
                                                            int* status) {
    grid_dep_wait();
    const int lane = threadIdx.x & 31;
    const int c = blockIdx.x * kEmitWarps + (threadIdx.x >> 5);
    if (c >= n_chunks) return;
    const Chunk ch = decode_chunk(Lo, c);
    const Decider dd = chunk_decider(sp[ch.seg]);
    const int n = Ls.p_cnt[c];
    // The chunk's candidates; the plain lists' kept entries are compacted in
    // place over them as (index, g_i / p_i) (a batch's candidates are all in
    // registers before its writes, which land below the next batch).
    int2* ent = Ls.p_ent + (int64_t)ch.m * Lo.d + ch.lo;
    const PhiloxStream ph(Lo, Lo.worker0 + (uint32_t)ch.m);
    const bool hybrid = Ls.k_offa != nullptr;   // the hybrid code's emit reads the decision bits instead
    uint32_t* wb = hybrid ? Ls.e_bits + (size_t)c * kBitWords : nullptr;
    int32_t* ks = Ls.k_sub ? Ls.k_sub + (size_t)c * kSubStride : nullptr;   // only when a sum follows
    const int lo32 = (int)ch.lo;
    int cnt = 0;        // kept so far
    int cnt_a = 0;      // kept with p = 1 (the hybrid code's Q_A)
    int last_sub = 0;   // slice of the last candidate seen
    for (int base = 0; base < n; base += 32 * kEmitBatch) {
        int2 e[kEmitBatch];
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const int i = base + r * 32 + lane;
            e[r] = i < n ? ent[i] : make_int2(0, 0);
        }
        // The batch's decisions first (independent Philox chains), then its ballots.
        bool keep[kEmitBatch], capped[kEmitBatch];
        float kv[kEmitBatch];   // the kept value g_i / p_i
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const int i = base + r * 32 + lane;
            const float gv = __int_as_float(e[r].y);
            capped[r] = i < n && fabsf(gv) >= dd.a_cap;   // p = 1: kept whatever the draw
            keep[r] = capped[r];
            kv[r] = gv;
            if (i < n && !capped[r]) {
                const uint32_t x = philox_word(ph, (uint32_t)e[r].x >> 2, e[r].x & 3);
                float v;
                keep[r] = dd(gv, x, v);
                kv[r] = v;
            }
        }
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const uint32_t bal = __ballot_sync(0xFFFFFFFFu, keep[r]);
            if (base + r * 32 < n) {
                if (hybrid) {
                    if (lane == 0) wb[(base >> 5) + r] = bal;
                } else if (keep[r]) {
                    ent[cnt + __popc(bal & ((1u << lane) - 1u))] = make_int2(e[r].x, __float_as_int(kv[r]));
                }
                if (ks) {
                    // Candidates are in ascending order: a candidate that opens slices
                    // (prev, sub] records the kept count before it for each of them.
                    const int i = base + r * 32 + lane;
                    const int sub = i < n ? (e[r].x - lo32) >> kSliceLog : kSlices;
                    int prev = __shfl_up_sync(0xFFFFFFFFu, sub, 1);
                    if (lane == 0) prev = last_sub;
                    const int before = cnt + __popc(bal & ((1u << lane) - 1u));
                    for (int t = prev + 1; t <= sub && t <= kSlices; ++t) ks[t] = before;
                    last_sub = __shfl_sync(0xFFFFFFFFu, sub, 31);
                }
            }
            cnt += __popc(bal);
            if (hybrid) cnt_a += __popc(__ballot_sync(0xFFFFFFFFu, capped[r]));
        }
    }
    if (ks) {
        // Slices after the last candidate (all of them if there is none).
        if (n == 0) last_sub = 0;
        if (lane <= kSlices && lane > last_sub) ks[lane] = cnt;
        if (lane == 0) ks[0] = 0;
    }
    if (lane == 0) {
        Ls.k_off[c] = cnt;
        if (hybrid) Ls.k_offa[c] = cnt_a;
    }

    // The last warp to finish one of the worker's chunks turns the worker's
    // counts into output offsets (exclusive prefix) and writes nnz.
    __threadfence();
    int last = 0;
    if (lane == 0) last = atomicAdd(&sp[ch.m * Lo.L].w_done, 1) == Lo.cpw - 1;
    if (!__shfl_sync(0xFFFFFFFFu, last, 0)) return;
    __threadfence();
    const long long total = warp_scan_counts(Ls.k_off + (size_t)ch.m * Lo.cpw, Lo.cpw, lane);
    if (Ls.k_offa) {
        // The hybrid code: Q_A offsets from the capped counts, Q_B's are the rest.
        const long long ta = warp_scan_counts(Ls.k_offa + (size_t)ch.m * Lo.cpw, Lo.cpw, lane);
        if (lane == 0) {
            n_a[ch.m] = (int32_t)ta;
            n_b[ch.m] = (int32_t)(total - ta);
            if (ta > cap || total - ta > cap) atomicOr(status, kStCapacity);
        }
    }
    if (lane == 0) {
        nnz[ch.m] = (int32_t)total;
        if (!Ls.k_offa && total > cap) atomicOr(status, kStCapacity);
    }
}

// The kept entries of chunk c, compacted in place by k_decide as (index,
// g_i / p_i), copied to their output positions (one warp; consecutive lanes
// write consecutive slots).  The chunk's count is the next chunk's offset
// minus its own (the worker's total after its last chunk).
__device__ __forceinline__ void emit_chunk(const Layout& Lo, const Lists& Ls, int c, const int32_t* nnz,
                                           int32_t* idx, float* val, int64_t cap) {
    const int lane = threadIdx.x & 31;
    const Chunk ch = decode_chunk(Lo, c);
    const int2* ent = Ls.p_ent + (int64_t)ch.m * Lo.d + ch.lo;
    const long long pos0 = Ls.k_off[c];
    const bool last = c - ch.m * Lo.cpw == Lo.cpw - 1;
    const int n = (int)((last ? (long long)nnz[ch.m] : (long long)Ls.k_off[c + 1]) - pos0);
    const int64_t out0 = (int64_t)ch.m * cap;
    for (int base = 0; base < n; base += 32 * kEmitBatch) {
        int2 en[kEmitBatch];
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const int i = base + r * 32 + lane;
            en[r] = i < n ? ent[i] : make_int2(0, 0);
        }
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const int i = base + r * 32 + lane;
            const long long pos = pos0 + i;
            if (i < n && pos < cap) {
                idx[out0 + pos] = en[r].x;
                val[out0 + pos] = __int_as_float(en[r].y);
            }
        }
    }
}

__global__ void __launch_bounds__(kEmitWarps * 32) k_emit(const __grid_constant__ Layout Lo,
                                                          const __grid_constant__ Lists Ls, int n_chunks,
                                                          const int32_t* nnz, int32_t* idx, float* val,
                                                          int64_t cap) {
    grid_dep_wait();
    const int c = blockIdx.x * kEmitWarps + (threadIdx.x >> 5);
    if (c < n_chunks) emit_chunk(Lo, Ls, c, nnz, idx, val, cap);
}

// The hybrid code of section 3.3 (eqs. 9-10) straight from the decisions: a
// kept candidate with p = 1 goes to Q_A as (index, g_i); any other kept
// candidate goes to Q_B as 2 * index + sign bit.  Offsets of both lists come
// from k_decide's two scans; chunk 0's warp writes the worker's 1 / lambda.
__global__ void __launch_bounds__(kEmitWarps * 32) k_emit_hybrid(const __grid_constant__ Layout Lo,
                                                                 const SegParam* __restrict__ sp,
                                                                 const __grid_constant__ Lists Ls, int n_chunks,
                                                                 const __grid_constant__ HybridOut H, int64_t cap) {
    grid_dep_wait();
    const int lane = threadIdx.x & 31;
    const int c = blockIdx.x * kEmitWarps + (threadIdx.x >> 5);
    if (c >= n_chunks) return;
    const Chunk ch = decode_chunk(Lo, c);
    const SegParam& P = sp[ch.seg];
    const float a_cap = P.a_cap;
    if (c == ch.m * Lo.cpw && lane == 0) H.inv_lam[ch.m] = P.inv_lam32;
    const int n = Ls.p_cnt[c];
    const int2* ent = Ls.p_ent + (int64_t)ch.m * Lo.d + ch.lo;
    const uint32_t* wb = Ls.e_bits + (size_t)c * kBitWords;
    const int64_t out0 = (int64_t)ch.m * cap;
    long long pa = Ls.k_offa[c], pb = (long long)Ls.k_off[c] - Ls.k_offa[c];
    const uint32_t below = (1u << lane) - 1u;
    for (int base = 0; base < n; base += 32 * kEmitBatch) {
        uint32_t wd[kEmitBatch];
        int2 en[kEmitBatch];
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const int i = base + r * 32 + lane;
            wd[r] = base + r * 32 < n ? wb[(base >> 5) + r] : 0u;
            en[r] = i < n ? ent[i] : make_int2(0, 0);
        }
#pragma unroll
        for (int r = 0; r < kEmitBatch; ++r) {
            const bool kept = (wd[r] >> lane) & 1u;
            const float gv = __int_as_float(en[r].y);
            const bool in_a = kept && fabsf(gv) >= a_cap;
            const uint32_t ba = __ballot_sync(0xFFFFFFFFu, in_a);
            const uint32_t bb = wd[r] & ~ba;
            if (in_a) {
                const long long q = pa + __popc(ba & below);
                if (q < cap) {
                    H.qa_idx[out0 + q] = en[r].x;
                    H.qa_val[out0 + q] = gv;
                }
            } else if (kept) {
                const long long q = pb + __popc(bb & below);
                if (q < cap) H.qb_code[out0 + q] = (uint32_t)en[r].x * 2u + (gv < 0.0f ? 1u : 0u);
            }
            pa += __popc(ba);
            pb += __popc(bb);
        }
    }
}

// ---------------------------------------------------------------------------
// The sparse sum of Algorithm 1, step 6 over the kept entries, one warp per
// 1024-coordinate slice.  The slice's entries of worker m are one contiguous
// run of m's chunk, compacted in place by k_decide (which recorded where each
// slice starts), so a warp gathers the runs of all workers (lane i takes
// entry i of a run), adds them into a private shared-memory tile worker by
// worker (a worker's entries have distinct indices; __syncwarp separates
// workers) and writes the slice once.  Entries past a worker's output
// capacity (which k_emit leaves out) are left out of the sum too.
// ---------------------------------------------------------------------------
constexpr int kSumWarps = 8;
constexpr int kSumGroup = 8;                  // workers whose entries are loaded together

__device__ __forceinline__ void sum_slice(const Layout& Lo, const Lists& Ls, int64_t cap, int gs, float div,
                                          int accumulate, float* out, float* acc) {
    const int lane = threadIdx.x & 31;
    const int k = gs / kSlices, sl = gs - k * kSlices;
    // Chunk k covers the same coordinates in every worker row (also for
    // layer-wise layouts, whose chunks start at segment starts).
    const Chunk ch = decode_chunk(Lo, k);
    const int64_t t0 = ch.lo + (int64_t)sl * kSlice;
    if (t0 >= ch.hi) return;
    const int tlen = (int)min((int64_t)kSlice, ch.hi - t0);
    if (accumulate) {
        // Continue a worker-order sum already in out (the earlier workers' part).
        for (int i = lane; i < kSlice; i += 32) acc[i] = i < tlen ? out[t0 + i] : 0.0f;
    } else {
#pragma unroll
        for (int i = 0; i < kSlice / 128; ++i)
            reinterpret_cast<float4*>(acc)[i * 32 + lane] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    }
    __syncwarp();
    for (int mb = 0; mb < Lo.M; mb += 32) {
        // Lane q describes worker mb + q: where its run starts and how long it is.
        const int nq = min(32, Lo.M - mb);
        long long a = 0;
        int cnt = 0;
        if (lane < nq) {
            const int c = (mb + lane) * Lo.cpw + k;
            const int32_t* ks = Ls.k_sub + (size_t)c * kSubStride;
            const long long room = cap - (long long)Ls.k_off[c];   // entries of the chunk that were emitted
            long long lo_ = ks[sl], hi_ = ks[sl + 1];
            lo_ = lo_ > room ? room : lo_;
            hi_ = hi_ > room ? room : hi_;
            a = (long long)(mb + lane) * Lo.d + ch.lo + lo_;
            cnt = hi_ > lo_ ? (int)(hi_ - lo_) : 0;
        }
        int maxc = cnt;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) maxc = max(maxc, __shfl_xor_sync(0xFFFFFFFFu, maxc, o));
        if (maxc <= 32) {
            // Every run fits one round: lane i takes entry i of each worker; the
            // loads of kSumGroup workers are issued together, then the adds run
            // worker by worker (a worker's entries have distinct indices).
            for (int q0 = 0; q0 < nq; q0 += kSumGroup) {
                int jj[kSumGroup];
                float vv[kSumGroup];
#pragma unroll
                for (int u = 0; u < kSumGroup; ++u) {
                    const int q = q0 + u;
                    const long long aq = __shfl_sync(0xFFFFFFFFu, a, q & 31);
                    const int cq = __shfl_sync(0xFFFFFFFFu, cnt, q & 31);
                    jj[u] = -1;
                    vv[u] = 0.0f;
                    if (q < nq && lane < cq) {
                        const int2 en = Ls.p_ent[aq + lane];
                        const int j = (int)((int64_t)en.x - t0);
                        vv[u] = __int_as_float(en.y);
                        if ((unsigned)j < (unsigned)tlen) jj[u] = j;   // always, for well-formed lists
                    }
                }
#pragma unroll
                for (int u = 0; u < kSumGroup; ++u) {
                    if (jj[u] >= 0) acc[jj[u]] += vv[u];
                    __syncwarp();
                }
            }
        } else {
            // Long runs: worker by worker, kSumGroup rounds of 32 entries loaded
            // together (a worker's entries never share an index).
            for (int q = 0; q < nq; ++q) {
                const long long aq = __shfl_sync(0xFFFFFFFFu, a, q);
                const int cq = __shfl_sync(0xFFFFFFFFu, cnt, q);
                for (int e0 = 0; e0 < cq; e0 += 32 * kSumGroup) {
                    int jj[kSumGroup];
                    float vv[kSumGroup];
#pragma unroll
                    for (int u = 0; u < kSumGroup; ++u) {
                        const int e = e0 + u * 32 + lane;
                        jj[u] = -1;
                        vv[u] = 0.0f;
                        if (e < cq) {
                            const int2 en = Ls.p_ent[aq + e];
                            const int j = (int)((int64_t)en.x - t0);
                            vv[u] = __int_as_float(en.y);
                            if ((unsigned)j < (unsigned)tlen) jj[u] = j;
                        }
                    }
#pragma unroll
                    for (int u = 0; u < kSumGroup; ++u)
                        if (jj[u] >= 0) acc[jj[u]] += vv[u];
                }
                __syncwarp();
            }
        }
    }
    // div > 0: the average of Algorithm 1 step 6 (one correctly rounded
    // division of the worker-order sum), else the sum itself.
    float* dst = out + t0;
    const bool whole = tlen == kSlice && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0;
    if (whole && !(div > 0.0f)) {
        // The sum leaves shared memory in one bulk copy (the asynchronous
        // proxy reads the tile once every lane's writes are fenced).
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) {
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
                         "r"((uint32_t)__cvta_generic_to_shared(acc)), "r"((int)(kSlice * sizeof(float)))
                         : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");   // the tile may be released
        }
        __syncwarp();
    } else if (whole) {
#pragma unroll
        for (int i = 0; i < kSlice / 128; ++i) {
            float4 t = reinterpret_cast<const float4*>(acc)[i * 32 + lane];
            if (div > 0.0f) {
                t.x = __fdiv_rn(t.x, div);
                t.y = __fdiv_rn(t.y, div);
                t.z = __fdiv_rn(t.z, div);
                t.w = __fdiv_rn(t.w, div);
            }
            reinterpret_cast<float4*>(dst)[i * 32 + lane] = t;
        }
    } else {
        for (int i = lane; i < tlen; i += 32) dst[i] = div > 0.0f ? __fdiv_rn(acc[i], div) : acc[i];
    }
}

// Emit and sum in one launch: both read what k_decide wrote and neither reads
// the other's output, so their CTAs run side by side (alternating, the
// longer role's surplus last).
__global__ void __launch_bounds__(kEmitWarps * 32) k_emit_sum(const __grid_constant__ Layout Lo,
                                                              const __grid_constant__ Lists Ls, int n_chunks,
                                                              const int32_t* nnz, int32_t* idx, float* val,
                                                              int64_t cap, int n_slices, float div, int accumulate,
                                                              float* out, int n_emit_blocks, int n_sum_blocks) {
    grid_dep_wait();
    static_assert(kEmitWarps == kSumWarps, "one block shape for both roles");
    __shared__ __align__(16) float tile[kSumWarps][kSlice];
    const int w = threadIdx.x >> 5;
    const int b = blockIdx.x, pairs = min(n_emit_blocks, n_sum_blocks);
    bool emit;
    int rb;
    if (b < 2 * pairs) {
        emit = (b & 1) == 0;
        rb = b >> 1;
    } else {
        emit = n_emit_blocks > n_sum_blocks;
        rb = pairs + (b - 2 * pairs);
    }
    if (emit) {
        const int c = rb * kEmitWarps + w;
        if (c < n_chunks) emit_chunk(Lo, Ls, c, nnz, idx, val, cap);
    } else {
        const int gs = rb * kSumWarps + w;
        if (gs < n_slices) sum_slice(Lo, Ls, cap, gs, div, accumulate, out, tile[w]);
    }
}

// ---------------------------------------------------------------------------
// Dense probabilities of one worker: p_i = min(lambda |g_i|, 1).
// ---------------------------------------------------------------------------
__global__ void k_prob(Layout Lo, const SegParam* __restrict__ sp, float* p) {
    grid_dep_wait();
    const SegParam P = sp[0];
    const int64_t n = Lo.d;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const float a = fabsf(load_one(Lo, 0, i));
        p[i] = (a >= P.a_cap) ? 1.0f : P.lam32 * a;
    }
}

// Random words of coordinates i0 .. i0 + n - 1 (one Philox call per thread per word).
__global__ void k_words(uint64_t seed, uint32_t step, uint32_t worker, int64_t i0, int64_t n, uint32_t* out) {
    grid_dep_wait();
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n; k += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = i0 + k;
        out[k] = word_of(group_words(seed, step, worker, i >> 2), (int)(i & 3));
    }
}

// ---------------------------------------------------------------------------
// Sparse sum.  k_bucket finds, for every worker list and output tile, the
// first entry at or after the tile (validating order and range); k_tiles
// gathers each tile's entries of all workers at once and adds them into a
// shared-memory tile worker by worker, in order.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_bucket(const __grid_constant__ AggArgs A, int32_t* off, int nt,
                                                int* status) {
    grid_dep_wait();
    constexpr int kUnroll = 8;   // entries per thread whose loads are in flight together
    const int m = blockIdx.y;
    const int32_t* __restrict__ idx = A.idx[m];
    long long n = A.nnz[m];
    if (n > A.cap) n = A.cap;
    if (n < 0) n = 0;
    int32_t* o = off + (int64_t)m * (nt + 1);
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long e0 = (long long)blockIdx.x * blockDim.x + threadIdx.x; e0 <= n; e0 += stride * kUnroll) {
        int32_t cur[kUnroll], prev[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const long long e = e0 + u * stride;
            cur[u] = e < n ? idx[e] : 0;
            prev[u] = (e > 0 && e <= n) ? idx[e - 1] : 0;
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const long long e = e0 + u * stride;
            if (e > n) break;
            long long t_cur = nt;
            if (e < n) {
                if (cur[u] < 0 || (int64_t)cur[u] >= A.d) {
                    atomicOr(status, kStInvalid);
                    continue;
                }
                t_cur = cur[u] / kAggTile;
            }
            long long t_prev = -1;
            if (e > 0) {
                if (prev[u] < 0 || (int64_t)prev[u] >= A.d) continue;
                if (e < n && prev[u] >= cur[u]) {
                    atomicOr(status, kStInvalid);
                    continue;
                }
                t_prev = prev[u] / kAggTile;
            }
            for (long long t = t_prev + 1; t <= t_cur; ++t) o[t] = (int32_t)e;
        }
    }
}

constexpr int kAggPer = 8;   // entries each thread holds per batch

// Tiles of kTile coordinates.  off[m * off_stride + t] is the first entry of
// worker m at or after tile t; the end of the last tile is the list length.
template <int kTile>
__global__ void __launch_bounds__(kThreads) k_tiles(const __grid_constant__ AggArgs A,
                                                    const int32_t* __restrict__ off, int off_stride, int nt,
                                                    float* out) {
    grid_dep_wait();
    extern __shared__ float acc[];   // kTile floats
    __shared__ int32_t s_pre[kMaxAggM + 1];
    __shared__ long long s_lo[kMaxAggM];
    __shared__ int shi[33];
    __shared__ int32_t s_cnt[kMaxAggM];
    const int M = A.M;
    for (int t = blockIdx.x; t < nt; t += gridDim.x) {
        const int64_t base = (int64_t)t * kTile;
        const int len = (int)min((int64_t)kTile, A.d - base);
        for (int k = threadIdx.x; k < kTile / 4; k += kThreads)
            reinterpret_cast<float4*>(acc)[k] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        for (int m = threadIdx.x; m < M; m += kThreads) {
            long long n = A.nnz[m];
            if (n > A.cap) n = A.cap;
            if (n < 0) n = 0;
            const int32_t* o = off + (int64_t)m * off_stride;
            long long lo = o[t], hi = t + 1 < nt ? o[t + 1] : n;
            lo = lo < 0 ? 0 : (lo > n ? n : lo);
            hi = hi < lo ? lo : (hi > n ? n : hi);
            s_lo[m] = lo;
            s_cnt[m] = (int32_t)(hi - lo);
        }
        __syncthreads();
        block_exclusive_scan(s_cnt, M, s_pre, shi);
        const int total = s_pre[M];
        for (int b = 0; b < total; b += kThreads * kAggPer) {
            int mm[kAggPer];
            int ii[kAggPer];
            float vv[kAggPer];
#pragma unroll
            for (int j = 0; j < kAggPer; ++j) {
                const int e = b + j * kThreads + threadIdx.x;
                mm[j] = -1;
                if (e < total) {
                    const int m = upper_slot(s_pre, M + 1, e);
                    const long long pos = s_lo[m] + (e - s_pre[m]);
                    ii[j] = (int)((int64_t)A.idx[m][pos] - base);
                    vv[j] = A.val[m][pos];
                    mm[j] = m;
                }
            }
            const int e_last = min(total, b + kThreads * kAggPer) - 1;
            const int m_first = upper_slot(s_pre, M + 1, b), m_last = upper_slot(s_pre, M + 1, e_last);
            for (int m = m_first; m <= m_last; ++m) {
#pragma unroll
                for (int j = 0; j < kAggPer; ++j)
                    if (mm[j] == m && ii[j] >= 0 && ii[j] < len) acc[ii[j]] += vv[j];
                __syncthreads();
            }
        }
        float* dst = out + base;
        if (len == kTile && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
            for (int k = threadIdx.x; k < kTile / 4; k += kThreads)
                reinterpret_cast<float4*>(dst)[k] = reinterpret_cast<const float4*>(acc)[k];
        } else {
            for (int k = threadIdx.x; k < len; k += kThreads) dst[k] = acc[k];
        }
        __syncthreads();
    }
}

int sm_count() { return device_sm_count(); }

}  // namespace

int device_sm_count() {
    constexpr int kMaxDev = 64;
    static std::atomic<int> cache[kMaxDev];   // 0 = not looked up yet (static storage: zero-initialised)
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    int n = (dev >= 0 && dev < kMaxDev) ? cache[dev].load(std::memory_order_relaxed) : 0;
    if (n > 0) return n;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    if (dev >= 0 && dev < kMaxDev) cache[dev].store(n, std::memory_order_relaxed);   // same value from any thread
    return n;
}

// ---------------------------------------------------------------------------
// Host launchers
// ---------------------------------------------------------------------------
cudaError_t launch_bound(const Layout& Lo, SegParam* sp, int n_seg, double kappa, int ns, int force_exact,
                         cudaStream_t st) {
    set_launch_error_site("k_bound launch");
    // One worker row (or a few): clusters of kBoundCTAs CTAs share each
    // segment's random sample loads.  Layer-wise calls have many short
    // segments: one CTA each (every CTA of a cluster would hold the whole
    // sample buffer, and clusters of 8 would take many waves).
    const size_t smem = (size_t)ns * sizeof(float);
    const bool one = Lo.L > 1;
    auto kern = one ? k_bound<1> : k_bound<kBoundCTAs>;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    // Short segments of a layer-wise call share CTAs, a warp each, when the
    // sample buffer holds at least one short segment per warp slice.
    int grid = n_seg * (one ? 1 : kBoundCTAs), per = 0;
    if (one && Lo.bnd_seg != nullptr && n_seg == Lo.M * Lo.L && ns >= kBoundWarpMax) {
        per = std::min(kBoundCtaThreads / 32, ns / kBoundWarpMax);
        const int n_short = Lo.M * (Lo.L - Lo.bnd_long);
        grid = Lo.M * Lo.bnd_long + (n_short + per - 1) / per;
    }
    TraceScope ts(kKBound, st);
    return launch_dep(kern, dim3(grid), dim3(kBoundCtaThreads), smem, st, Lo, sp, kappa, ns, force_exact, per);
}

cudaError_t launch_stream(const Layout& Lo, const SegParam* sp, const Lists& Ls, int n_chunks, bool build_p,
                          cudaStream_t st) {
    set_launch_error_site("k_stream launch");
    const int grid = std::min(n_chunks, sm_count() * 8);
    TraceScope ts(kKStream, st);
    return launch_dep(k_stream, dim3(grid), dim3(kThreads), 0, st, Lo, sp, Ls, n_chunks, build_p ? 1 : 0);
}

cudaError_t launch_solve(const Layout& Lo, SegParam* sp, const Lists& Ls, int n_seg, double kappa, int iters,
                         int force_exact, int* status, gs_info_dev* info, cudaStream_t st, int64_t max_seg_len) {
    set_launch_error_site("k_solve launch");
    // Shared memory for the largest segment only: its chunk prefix and at most
    // as many candidate values as it has coordinates (short layers then leave
    // room for more resident CTAs).
    const int64_t maxch = (max_seg_len + kChunk - 1) / kChunk + 1;
    const int cap_chunks = (int)std::min<int64_t>(kSolveSmemChunks, maxch);
    const int cap_c = (int)std::min<int64_t>(kSolveSmemC, max_seg_len);
    const size_t smem = sizeof(int32_t) * (cap_chunks + 4) + sizeof(float) * cap_c;
    cudaError_t e = cudaFuncSetAttribute(k_solve, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_solve, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    TraceScope ts(kKSolve, st);
    // C holds about the capped coordinates, whose count the budget kappa d
    // bounds at the fixed point: segments with a budget above 2^20 (where C can
    // hold millions of values) get a cluster of kSolveCTAs CTAs, others one.
    const int ncta = (Lo.L == 1 && kappa * (double)Lo.d > (double)(1 << 20)) ? kSolveCTAs : 1;
    if (ncta == 1)
        return launch_dep(k_solve, dim3(n_seg), dim3(kThreads), smem, st, Lo, sp, Ls, kappa, iters, force_exact,
                          status, info, cap_chunks, cap_c);
    return launch_dep_cluster(k_solve, dim3(n_seg * ncta), dim3(kSolveClusterThreads), smem, ncta, st, Lo, sp, Ls, kappa, iters,
                              force_exact, status, info, cap_chunks, cap_c);
}

cudaError_t launch_compact(const Layout& Lo, const SegParam* sp, const Lists& Ls, int n_chunks, int32_t* idx,
                           float* val, int32_t* nnz, int64_t cap, int* status, cudaStream_t st, float* sum_out,
                           const HybridOut* hybrid, bool average, bool accumulate) {
    const int blocks = (n_chunks + kEmitWarps - 1) / kEmitWarps;
    cudaError_t e;
    {
        set_launch_error_site("k_decide launch");
        TraceScope ts(kKDecide, st);
        Lists Ld = Ls;
        if (!sum_out || hybrid) Ld.k_sub = nullptr;   // the slice table serves the sum only
        e = launch_dep(k_decide, dim3(blocks), dim3(kEmitWarps * 32), 0, st, Lo, const_cast<SegParam*>(sp), Ld,
                       n_chunks, nnz, hybrid ? hybrid->n_a : nullptr, hybrid ? hybrid->n_b : nullptr, cap, status);
    }
    if (e != cudaSuccess) return e;
    if (hybrid) {
        set_launch_error_site("k_emit_hybrid launch");
        TraceScope ts(kKEmit, st);
        return launch_dep(k_emit_hybrid, dim3(blocks), dim3(kEmitWarps * 32), 0, st, Lo, sp, Ls, n_chunks, *hybrid,
                          cap);
    }
    if (!sum_out) {
        set_launch_error_site("k_emit launch");
        TraceScope ts(kKEmit, st);
        return launch_dep(k_emit, dim3(blocks), dim3(kEmitWarps * 32), 0, st, Lo, Ls, n_chunks,
                          static_cast<const int32_t*>(nnz), idx, val, cap);
    }
    // The output lists and the sparse sum of the M rows (one warp per slice),
    // side by side in one launch.
    const int n_slices = Lo.cpw * kSlices;
    const int sblocks = (n_slices + kSumWarps - 1) / kSumWarps;
    set_launch_error_site("k_emit_sum launch");
    TraceScope ts(kKEmitSum, st);
    return launch_dep(k_emit_sum, dim3(blocks + sblocks), dim3(kEmitWarps * 32), 0, st, Lo, Ls, n_chunks,
                      static_cast<const int32_t*>(nnz), idx, val, cap, n_slices, average ? (float)Lo.M : 0.0f,
                      accumulate ? 1 : 0, sum_out, blocks, sblocks);
}

cudaError_t launch_prob(const Layout& Lo, const SegParam* sp, float* p, cudaStream_t st) {
    set_launch_error_site("k_prob launch");
    const int64_t blocks = std::min<int64_t>((Lo.d + 255) / 256, (int64_t)sm_count() * 16);
    TraceScope ts(kKProb, st);
    return launch_dep(k_prob, dim3((int)blocks), dim3(256), 0, st, Lo, sp, p);
}

cudaError_t launch_words(uint64_t seed, uint32_t step, uint32_t worker, int64_t i0, int64_t n, uint32_t* out,
                         cudaStream_t st) {
    set_launch_error_site("k_words launch");
    const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, (int64_t)sm_count() * 8));
    TraceScope ts(kKWords, st);
    k_words<<<(int)blocks, 256, 0, st>>>(seed, step, worker, i0, n, out);
    return cudaGetLastError();
}

cudaError_t launch_aggregate(const AggArgs& A, int32_t* off, float* out, int* status, cudaStream_t st) {
    set_launch_error_site("k_bucket launch");
    const int nt = (int)((A.d + kAggTile - 1) / kAggTile);
    // Bucket: a few blocks per worker, grid-stride over its entries.
    const int bx = std::max(1, std::min((sm_count() * 4 + A.M - 1) / A.M, (int)((A.d + 255) / 256 + 1)));
    dim3 grid(bx, A.M);
    {
        TraceScope ts(kKBucket, st);
        k_bucket<<<grid, 256, 0, st>>>(A, off, nt, status);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    set_launch_error_site("k_tiles launch");
    const int tg = std::min(nt, sm_count() * 4);
    TraceScope ts(kKTiles, st);
    k_tiles<kAggTile><<<tg, kThreads, kAggTile * sizeof(float), st>>>(A, off, nt + 1, nt, out);
    return cudaGetLastError();
}

int agg_tiles(int64_t d) { return (int)((d + kAggTile - 1) / kAggTile); }
int chunk_size() { return kChunk; }
int bound_short_max() { return kBoundWarpMax; }

}  // namespace gs
