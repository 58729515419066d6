// gs_eps.cu -- Algorithm 2 (section 3.2) on the GPU: lambda for a variance
// budget eps (problem (4)) instead of a density budget.
//
// With t = 1 / lambda and p_i = min(|g_i| / t, 1) (Proposition 1), the
// variance of (4) is sum_{|g| >= t} g^2 + t sum_{|g| < t} |g|, so the active
// constraint reads
//     phi(t) = sum_i |g_i| (t - |g_i|)_+ = eps S,     S = sum_i g_i^2.
// phi is continuous, convex and non-decreasing in t.  Condition (6) at k is
// phi(a_{k+1}) <= eps S for the sorted magnitudes a_1 >= a_2 >= ..., so the
// smallest such k puts the root t* in [a_{k+1}, a_k], and (7) is lambda = 1/t*
// with t* = (eps S + sum_{i>k} a_i^2) / sum_{i>k} a_i: the root of the linear
// piece of phi between those two magnitudes.  No sort is needed to find it:
//
//   k_eps_hist     one read of g.  Per segment, a count histogram of |g| over
//                  2048 bins of its fp32 bit pattern (8 exponent and 3
//                  mantissa bits: 1/8-octave bins; one shared-memory copy per
//                  CTA, integer atomics) and S in partials of 4096
//                  coordinates (fma partials of 32 squares, error-free sum).
//   k_eps_bracket  one CTA per segment.  From the counts alone, bounds of phi
//                  at every bin edge; the largest edge whose upper bound stays
//                  below eps S is a certain lower bound t_c of t* (the
//                  streaming pass's C threshold; lambda_up = 1 / t_c), the
//                  smallest edge whose lower bound reaches eps S an upper
//                  bound t_up.
//   k_stream[_tma] C = {|g| >= t_c}, S_low = sum of |g| below t_c, B_low =
//                  sum of g^2 below t_c, and the keep candidates for lambda_up.
//   k_solve_eps    Newton's method on phi(t) = eps S from t_up, each step one
//                  pass over C (everything below t_c is summed in S_low).
//                  From the right, Newton's steps on a convex piecewise-linear
//                  function never pass the root, and a step that leaves the
//                  set {|g| < t} unchanged has landed on it exactly.  Where
//                  they crawl (eps = 0, where phi is flat at the root, or more
//                  than 24 steps) a bisection over the fp32 bit patterns of t
//                  finishes in at most 31 more passes.
// Then the decide / emit (or probabilities) kernels of Algorithm 3 run as is.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {

namespace {

constexpr int kHistShift = 20;
constexpr int kHistBins = 1 << (31 - kHistShift);    // 2048
constexpr int kEdgeFirst = 16;    // lowest edge used (2^-125): below it halving is not 8 bins
constexpr int kEdgeLast = 2039;   // highest finite lower edge (bin 2039 ends at +inf)
constexpr int kUnitLog = 12;
constexpr int kUnit = 1 << kUnitLog;                 // coordinates per S partial
constexpr int kUnitsPerChunk = kChunk / kUnit;
constexpr int kHistWarps = 8;
constexpr int kHistBatch = 8;     // 16-byte loads per lane in flight
constexpr int kHistCtasPerSm = 5;   // 48 registers x 256 threads
constexpr int kBrThreads = 256;
constexpr int kBrPer = kHistBins / kBrThreads;
constexpr int kEpsNewtonMax = 24;
constexpr int kEpsBisectMax = 32;   // a bisection over fp32 bit patterns ends within 31 passes
constexpr int kEpsCTAs = 8;       // cluster size of k_solve_eps for long segments
constexpr int kPassUnroll = 8;    // loads per lane in flight in the passes over C

static_assert(kChunk % kUnit == 0, "units tile a chunk");
static_assert(kHistBins % kBrThreads == 0, "bins split evenly over the bracket CTA");

__device__ __forceinline__ float bin_lo(int b) { return __uint_as_float((uint32_t)b << kHistShift); }

__device__ __forceinline__ void hist_count(uint32_t* h, float x) {
    atomicAdd(&h[(__float_as_uint(x) & 0x7FFFFFFFu) >> kHistShift], 1u);
}

// Counts and squares of 8 fp32 lanes' values (one 16-byte load each of 4).
__device__ __forceinline__ float hist_batch_f32(uint32_t* h, const float4 (&v)[kHistBatch]) {
    float s0 = 0.0f, s1 = 0.0f, s2 = 0.0f, s3 = 0.0f;
#pragma unroll
    for (int r = 0; r < kHistBatch; ++r) {
        hist_count(h, v[r].x);
        hist_count(h, v[r].y);
        hist_count(h, v[r].z);
        hist_count(h, v[r].w);
        s0 = fmaf(v[r].x, v[r].x, s0);
        s1 = fmaf(v[r].y, v[r].y, s1);
        s2 = fmaf(v[r].z, v[r].z, s2);
        s3 = fmaf(v[r].w, v[r].w, s3);
    }
    return (s0 + s1) + (s2 + s3);
}

// The same for bf16: each 16-byte load holds 8 values.
__device__ __forceinline__ float hist_batch_bf16(uint32_t* h, const uint4 (&v)[kHistBatch]) {
    float s[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
    for (int r = 0; r < kHistBatch; ++r) {
        const uint32_t w[4] = {v[r].x, v[r].y, v[r].z, v[r].w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float a = bf16_bits_to_float(w[k] & 0xFFFFu), b = bf16_bits_to_float(w[k] >> 16);
            hist_count(h, a);
            hist_count(h, b);
            s[k] = fmaf(a, a, s[k]);
            s[k] = fmaf(b, b, s[k]);
        }
    }
    return (s[0] + s[1]) + (s[2] + s[3]);
}

// gx CTAs per segment (block x: segment x / gx).  The CTAs of a segment share
// its 4096-coordinate units (one warp per unit at a time); each CTA keeps one
// shared-memory histogram, added into
// the segment's global histogram at the end (integer atomics: the order does
// not matter).  Each unit's sum of squares is one fixed computation (lane
// assignment, fma partials of 32 values, error-free running sum, fixed
// shuffle tree), written to u_sq[unit].
__global__ void __launch_bounds__(kHistWarps * 32) k_eps_hist(const __grid_constant__ Layout Lo, uint32_t* ghist,
                                                              double* u_sq, int gx) {
    grid_dep_wait();
    __shared__ uint32_t h[kHistBins];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int b = tid; b < kHistBins; b += blockDim.x) h[b] = 0u;
    __syncthreads();
    const int s = blockIdx.x / gx, bx = blockIdx.x - s * gx;
    int m, l, c0, c1;
    int64_t slo, shi;
    seg_range(Lo, s, m, l, slo, shi, c0, c1);
    const int u_end = c1 * kUnitsPerChunk;
    for (int u = c0 * kUnitsPerChunk + bx * kHistWarps + warp; u < u_end; u += gx * kHistWarps) {
        const int c = u / kUnitsPerChunk;
        const Chunk ch = decode_chunk(Lo, c);
        const int64_t lo = ch.lo + (int64_t)(u - c * kUnitsPerChunk) * kUnit;
        const int64_t hi = min(ch.hi, lo + kUnit);
        float sh = 0.0f, sl = 0.0f;
        const int64_t flat = (int64_t)m * Lo.d + lo;
        if (Lo.dtype == 0 && hi - lo == kUnit &&
            (reinterpret_cast<uintptr_t>(static_cast<const float*>(Lo.g) + flat) & 15u) == 0) {
            const float4* p4 = reinterpret_cast<const float4*>(static_cast<const float*>(Lo.g) + flat);
#pragma unroll 1
            for (int k0 = 0; k0 < kUnit / 128; k0 += kHistBatch) {   // 32 loads of 16 bytes per lane
                float4 v[kHistBatch];
#pragma unroll
                for (int r = 0; r < kHistBatch; ++r) v[r] = __ldcs(p4 + (k0 + r) * 32 + lane);
                two_sum_add(sh, sl, hist_batch_f32(h, v));
            }
        } else if (Lo.dtype == 1 && hi - lo == kUnit &&
                   (reinterpret_cast<uintptr_t>(static_cast<const uint16_t*>(Lo.g) + flat) & 15u) == 0) {
            const uint4* p8 = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(Lo.g) + flat);
#pragma unroll 1
            for (int k0 = 0; k0 < kUnit / 256; k0 += kHistBatch) {   // 16 loads of 16 bytes per lane
                uint4 v[kHistBatch];
#pragma unroll
                for (int r = 0; r < kHistBatch; ++r) v[r] = __ldcs(p8 + (k0 + r) * 32 + lane);
                two_sum_add(sh, sl, hist_batch_bf16(h, v));
            }
        } else if (lo < hi) {
            // Ragged or unaligned unit: 4-coordinate groups with a validity mask.
            const int64_t q0 = lo >> 2, q1 = (hi - 1) >> 2;
            for (int64_t gq = q0 + lane; gq <= q1; gq += 32) {
                float v[4];
                const int mk = load_group(Lo, m, gq, lo, hi, v);
                float s4 = 0.0f;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    if ((mk >> k) & 1) {
                        hist_count(h, v[k]);
                        s4 = fmaf(v[k], v[k], s4);
                    }
                }
                two_sum_add(sh, sl, s4);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float oh = __shfl_xor_sync(0xFFFFFFFFu, sh, o);
            const float ol = __shfl_xor_sync(0xFFFFFFFFu, sl, o);
            df_add(sh, sl, oh, ol);
        }
        if (lane == 0) u_sq[u] = (double)sh + (double)sl;
    }
    __syncthreads();
    uint32_t* gh = ghist + (size_t)s * kHistBins;
    for (int b = tid; b < kHistBins; b += blockDim.x) {
        const uint32_t n = h[b];
        if (n) atomicAdd(gh + b, n);
    }
}

// Exclusive prefix over the block of four doubles per thread (inclusive
// shuffle scan in each warp, warps added in order); returns the block totals.
__device__ __forceinline__ void block_exscan4(double v[4], double tot[4], double (*sw)[4]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    double inc[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) inc[k] = v[k];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const double t = __shfl_up_sync(0xFFFFFFFFu, inc[k], o);
            if (lane >= o) inc[k] += t;
        }
    }
    if (lane == 31) {
#pragma unroll
        for (int k = 0; k < 4; ++k) sw[warp][k] = inc[k];
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        double before = 0.0, all = 0.0;
        for (int w = 0; w < nw; ++w) {
            if (w < warp) before += sw[w][k];
            all += sw[w][k];
        }
        v[k] = before + inc[k] - v[k];
        tot[k] = all;
    }
    __syncthreads();
}

// Bounds of phi at an edge t = lo_b (b >= kEdgeFirst) from the counts n_j of
// the bins below it.  t / 2 is the edge of bin b - 8, so bins j < b - 8 lie
// in [0, t/2], where a (t - a) grows with a (largest at hi_j, smallest at
// lo_j), and bins b-8 <= j < b lie in [t/2, t], where it falls (largest at
// lo_j, smallest at hi_j).  pre[0..3][x] = sum_{j < x} of n hi, n lo, n hi^2,
// n lo^2.
__global__ void __launch_bounds__(kBrThreads) k_eps_bracket(const __grid_constant__ Layout Lo, SegParam* sp,
                                                            const uint32_t* __restrict__ ghist,
                                                            const double* __restrict__ u_sq, double eps,
                                                            int take_all) {
    grid_dep_wait();
    extern __shared__ double pre[];   // [4][kHistBins + 1]
    __shared__ double shd[33];
    __shared__ double sw[kBrThreads / 32][4];
    __shared__ int shb[2][kBrThreads / 32];
    const int s = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int m, l, c0, c1;
    int64_t lo, hi;
    seg_range(Lo, s, m, l, lo, hi, c0, c1);
    double acc = 0.0;
    for (int64_t u = (int64_t)c0 * kUnitsPerChunk + tid; u < (int64_t)c1 * kUnitsPerChunk; u += kBrThreads)
        acc += u_sq[u];
    const double S = block_sum(acc, shd);

    const uint32_t* hg = ghist + (size_t)s * kHistBins;
    double v[kBrPer][4];
    double own[4] = {0.0, 0.0, 0.0, 0.0};
#pragma unroll
    for (int r = 0; r < kBrPer; ++r) {
        const int j = tid * kBrPer + r;
        const double n = j < kEdgeLast ? (double)hg[j] : 0.0;   // bins from 2039 up never lie below a used edge
        const double bl = (double)bin_lo(j), bh = j < kEdgeLast ? (double)bin_lo(j + 1) : 0.0;
        v[r][0] = n > 0.0 ? n * bh : 0.0;
        v[r][1] = n > 0.0 ? n * bl : 0.0;
        v[r][2] = n > 0.0 ? n * bh * bh : 0.0;
        v[r][3] = n > 0.0 ? n * bl * bl : 0.0;
#pragma unroll
        for (int k = 0; k < 4; ++k) own[k] += v[r][k];
    }
    double tot[4];
    block_exscan4(own, tot, sw);
#pragma unroll
    for (int r = 0; r < kBrPer; ++r) {
        const int j = tid * kBrPer + r;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            pre[k * (kHistBins + 1) + j] = own[k];
            own[k] += v[r][k];
        }
    }
    if (tid == 0) {
#pragma unroll
        for (int k = 0; k < 4; ++k) pre[k * (kHistBins + 1) + kHistBins] = tot[k];
    }
    __syncthreads();

    // The targets carry a margin for the rounding of S (fp32 partials of 32
    // squares, ~2^-20 relative at worst) and of the bounds (fp64 sums of up
    // to 2^31 terms, one cancellation each).
    const double eS = eps * S;
    const double slack = 0x1p-16 * eS + 0x1p-40 * S;
    const double lo_target = eS - slack, hi_target = eS + slack;
    const double* P0 = pre;
    const double* P1 = pre + (kHistBins + 1);
    const double* P2 = pre + 2 * (kHistBins + 1);
    const double* P3 = pre + 3 * (kHistBins + 1);
    int bc = -1, bu = 0x7FFFFFFF;
#pragma unroll
    for (int r = 0; r < kBrPer; ++r) {
        const int b = tid * kBrPer + r;
        if (b < kEdgeFirst || b > kEdgeLast) continue;
        const double t = (double)bin_lo(b);
        const int h = b - 8;
        const double phi_max = t * (P0[h] + (P1[b] - P1[h])) - (P2[h] + (P3[b] - P3[h]));
        const double phi_min = t * (P1[h] + (P0[b] - P0[h])) - (P3[h] + (P2[b] - P2[h]));
        if (phi_max <= lo_target) bc = max(bc, b);
        if (phi_min >= hi_target) bu = min(bu, b);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        bc = max(bc, __shfl_xor_sync(0xFFFFFFFFu, bc, o));
        bu = min(bu, __shfl_xor_sync(0xFFFFFFFFu, bu, o));
    }
    if (lane == 0) {
        shb[0][warp] = bc;
        shb[1][warp] = bu;
    }
    __syncthreads();
    if (tid == 0) {
        for (int w = 0; w < kBrThreads / 32; ++w) {
            bc = max(bc, shb[0][w]);
            bu = min(bu, shb[1][w]);
        }
        const float kInfF = __int_as_float(0x7F800000);
        SegParam& P = sp[s];
        P.done = 0;
        P.w_done = 0;
        P.next_chunk = 0;
        P.sq = S;
        P.l1 = 0.0;
        int flags = 0;
        float t_c = 0.0f, up32 = kInfF;
        if (!isfinite(S)) {
            flags = kSegNonfinite | kSegTakeAll;
        } else if (take_all || !(S > 0.0) || bc < 0 || !(lo_target > 0.0)) {
            flags = kSegTakeAll;   // every coordinate a candidate
        } else {
            t_c = bin_lo(bc);
            up32 = __frcp_ru(t_c);  // lambda = 1 / t* <= 1 / t_c <= up32
        }
        P.t_c = t_c;
        P.lam_up32 = up32;
        P.lam_up = (double)up32;
        P.t_up = (isfinite(S) && bu <= kEdgeLast) ? bin_lo(bu) : kInfF;
        P.flags = flags;
    }
}

struct EpsPart {
    float uh, ul;           // sum |g| of C below the threshold (double-float)
    float bh, bl;           // sum g^2 of C below it
    float qh, ql;           // sum g^2 of C at or above it
    int below, above;       // counts of C below / at or above
};

// Launched with clusters of 1 or kEpsCTAs CTAs per segment.  Every CTA of a
// cluster walks a share of the segment's C chunks in each pass; the CTA
// partials are exchanged through distributed shared memory and added in rank
// order, so every thread of the cluster holds the same sums and runs the same
// scalar Newton iteration.
__global__ void __launch_bounds__(kThreads) k_solve_eps(const __grid_constant__ Layout Lo, SegParam* sp,
                                                        const __grid_constant__ Lists Ls, double eps, int* status,
                                                        gs_info_dev* info) {
    grid_dep_wait();
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int ncta = (int)cluster.num_blocks(), rank = (int)cluster.block_rank();
    __shared__ double shd[33];
    __shared__ float4 sh4[33];
    __shared__ EpsPart xch[2];
    const int s = blockIdx.x / ncta, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int m, l, c0, c1;
    int64_t lo, hi;
    seg_range(Lo, s, m, l, lo, hi, c0, c1);
    const int nch = c1 - c0;
    const double S_hist = sp[s].sq;   // the histogram pass's sum (non-finite check only)
    const float t_up = sp[s].t_up;
    const double lam_up = sp[s].lam_up;
    int flags = sp[s].flags & (kSegTakeAll | kSegNonfinite);

    double sl = 0.0, bq = 0.0;
    for (int c = c0 + tid; c < c1; c += blockDim.x) {
        sl += Ls.s_low[c];
        bq += Ls.b_low[c];
    }
    const double S_low = block_sum(sl, shd);
    const double B_low = block_sum(bq, shd);
    const float* cb = Ls.c_val + (int64_t)m * Lo.d + lo;

    int buf = 0;
    // One pass over C at threshold tau: below = #{C : |g| < tau}, U = S_low +
    // their sum of |g|, Q = B_low + their sum of g^2, and Qa the sum of g^2
    // over the rest of C.  Every sum is of positive terms (no cancellation).
    auto pass = [&](float tau, int& below, int& above, double& U, double& Q, double& Qa) {
        float uh = 0.0f, ul = 0.0f, bh = 0.0f, bl = 0.0f, qh = 0.0f, ql = 0.0f;
        int kb = 0, ka = 0;
        for (int q = rank * kWarps + warp; q < nch; q += ncta * kWarps) {
            const int n = Ls.c_cnt[c0 + q];
            const float* src = cb + (int64_t)q * kChunk;
            // kPassUnroll loads per lane in flight, then the sums in index order.
            for (int e0 = 0; e0 < n; e0 += 32 * kPassUnroll) {
                float av[kPassUnroll];
#pragma unroll
                for (int u = 0; u < kPassUnroll; ++u) {
                    const int e = e0 + u * 32 + lane;
                    av[u] = e < n ? src[e] : 0.0f;
                }
#pragma unroll
                for (int u = 0; u < kPassUnroll; ++u) {
                    if (e0 + u * 32 + lane >= n) continue;
                    const float a = av[u];
                    const float p = a * a;
                    if (a < tau) {
                        ++kb;
                        two_sum_add(uh, ul, a);
                        two_sum_add(bh, bl, p);
                        bl += fmaf(a, a, -p);
                    } else {
                        ++ka;
                        two_sum_add(qh, ql, p);
                        ql += fmaf(a, a, -p);
                    }
                }
            }
        }
        block_sum_df(uh, ul, kb, sh4);
        block_sum_df(qh, ql, ka, sh4);
        int unused = 0;
        block_sum_df(bh, bl, unused, sh4);
        if (tid == 0) xch[buf] = EpsPart{uh, ul, bh, bl, qh, ql, kb, ka};
        cluster.sync();
        float ruh = 0.0f, rul = 0.0f, rbh = 0.0f, rbl = 0.0f, rqh = 0.0f, rql = 0.0f;
        int rb = 0, ra = 0;
        for (int r = 0; r < ncta; ++r) {
            const EpsPart v = *cluster.map_shared_rank(&xch[buf], r);
            df_add(ruh, rul, v.uh, v.ul);
            df_add(rbh, rbl, v.bh, v.bl);
            df_add(rqh, rql, v.qh, v.ql);
            rb += v.below;
            ra += v.above;
        }
        buf ^= 1;
        below = rb;
        above = ra;
        U = S_low + ((double)ruh + (double)rul);
        Q = B_low + ((double)rbh + (double)rbl);
        Qa = (double)rqh + (double)rql;
    };

    double lam = 0.0, U = 0.0, Q = 0.0, Qa = 0.0;
    int below = 0, above = 0, it = 0;
    bool bad = false;
    float tau = t_up;
    if (!(flags & kSegNonfinite) && isfinite(S_hist) && S_hist > 0.0) pass(tau, below, above, U, Q, Qa);
    // S = sum g^2 from the sums of this pass (finer than the histogram's).
    const double S = Q + Qa;
    if ((flags & kSegNonfinite) || !isfinite(S_hist) || !isfinite(S) || !isfinite(U)) {
        flags |= kSegNonfinite;
        if (rank == 0 && tid == 0) atomicOr(status, kStNonfinite);
    } else if (S > 0.0) {
        const double eS = eps * S;
        if (!(U > 0.0) || !((double)tau * U - Q > eS)) {
            // Nothing below t_up, or phi(t_up) not above eps S (only possible
            // for eps = 0 or by rounding): start from the top.
            tau = __int_as_float(0x7F800000);
            pass(tau, below, above, U, Q, Qa);
        }
        bool conv = false;
        // eps = 0 makes phi flat at the root, where Newton's steps are only
        // weighted means: go straight to the bisection.
        const int newton_max = eps > 0.0 ? kEpsNewtonMax : 0;
        while (it < newton_max) {
            // The root of the piece of phi just left of tau.  a < tau1 holds
            // exactly when a < t1 for every float a (tau1 = t1 rounded up).
            const double t1 = (eS + Q) / U;
            const float tau1 = __double2float_ru(t1);
            if (tau1 == tau) {
                conv = true;
                break;
            }
            int b1, a1;
            double U1, Q1, Qa1;
            pass(tau1, b1, a1, U1, Q1, Qa1);
            ++it;
            // No C value between tau and tau1: phi is linear there and t1 is the
            // root (a start left of the root, which only rounding of the bracket
            // could give, moves right and then converges from the right).
            if (b1 == below) {
                conv = true;
                break;
            }
            tau = tau1;
            below = b1;
            above = a1;
            U = U1;
            Q = Q1;
        }
        if (!conv) {
            // Bisection over the fp32 bit patterns of the threshold, keeping
            // phi(lo) <= eps S < phi(hi) (t_c, or 0, is a valid lo; tau a valid
            // hi): it ends on the smallest float hi with phi(hi) > eps S, and
            // the piece of phi left of hi holds the largest root.
            uint32_t blo = __float_as_uint(sp[s].t_c), bhi = __float_as_uint(tau);
            while (bhi - blo > 1u && it < kEpsNewtonMax + kEpsBisectMax) {
                const uint32_t mid = blo + ((bhi - blo) >> 1);
                const float tm = __uint_as_float(mid);
                int b1, a1;
                double U1, Q1, Qa1;
                pass(tm, b1, a1, U1, Q1, Qa1);
                ++it;
                if ((double)tm * U1 - Q1 > eS) {
                    bhi = mid;
                    below = b1;
                    above = a1;
                    U = U1;
                    Q = Q1;
                } else {
                    blo = mid;
                }
            }
            conv = bhi - blo <= 1u;
        }
        lam = U / (eS + Q);
        // Not converged, or lambda beyond the bound the lists were built for:
        // neither should happen; the call reports an internal error.
        if (!conv || !(lam <= lam_up)) bad = true;
    }
    cluster.sync();   // no CTA may leave while a peer still reads its partials
    if (rank != 0 || tid != 0) return;
    if (bad) {
        flags |= kSegExact;
        atomicOr(status, kStInternal);
    }
    SegParam& P = sp[s];
    P.lam = lam;
    P.lam32 = (float)lam;
    P.a_cap = cap_threshold(lam);
    P.inv_lam32 = lam > 0.0 ? (float)(1.0 / lam) : 0.0f;
    P.capped = lam > 0.0 ? above : 0;
    P.sum_p = lam > 0.0 ? (double)above + lam * U : 0.0;
    P.iters_run = it;
    P.flags = flags;
    if (info) {
        info[s].lambda = lam;
        info[s].sum_p = P.sum_p;
        info[s].capped = P.capped;
        info[s].iters_run = it;
        info[s].flags = bad ? 1 : 0;
    }
}

int sm_count_eps() { return device_sm_count(); }

}  // namespace

size_t eps_hist_words(int n_seg) { return (size_t)n_seg * kHistBins; }
size_t eps_units(int n_chunks) { return (size_t)n_chunks * kUnitsPerChunk; }

cudaError_t launch_eps_bracket(const Layout& Lo, SegParam* sp, uint32_t* hist, double* u_sq, int n_seg, int n_chunks,
                               double eps, int take_all, cudaStream_t st) {
    set_launch_error_site("k_eps_hist memset");
    cudaError_t e = cudaMemsetAsync(hist, 0, sizeof(uint32_t) * eps_hist_words(n_seg), st);
    if (e != cudaSuccess) return e;
    // Every segment gets the same number of CTAs, at most one warp per unit.
    int max_units = 0;
    if (Lo.L == 1) {
        max_units = Lo.cpw * kUnitsPerChunk;
    } else {
        max_units = n_chunks * kUnitsPerChunk;   // a bound; CTAs without a unit exit at once
    }
    const int want = (sm_count_eps() * kHistCtasPerSm + n_seg - 1) / n_seg;
    const int gx = std::max(1, std::min(want, (max_units + kHistWarps - 1) / kHistWarps));
    {
        set_launch_error_site("k_eps_hist launch");
        // A plain launch: its predecessor in the stream is the memset.
        TraceScope ts(kKEpsHist, st);
        k_eps_hist<<<gx * n_seg, kHistWarps * 32, 0, st>>>(Lo, hist, u_sq, gx);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return e;
    set_launch_error_site("k_eps_bracket launch");
    const size_t smem = sizeof(double) * 4 * (kHistBins + 1);
    e = cudaFuncSetAttribute(k_eps_bracket, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    TraceScope ts(kKEpsBracket, st);
    return launch_dep(k_eps_bracket, dim3(n_seg), dim3(kBrThreads), smem, st, Lo, sp,
                      static_cast<const uint32_t*>(hist), static_cast<const double*>(u_sq), eps, take_all);
}

cudaError_t launch_solve_eps(const Layout& Lo, SegParam* sp, const Lists& Ls, int n_seg, double eps, int* status,
                             gs_info_dev* info, cudaStream_t st) {
    set_launch_error_site("k_solve_eps launch");
    TraceScope ts(kKSolveEps, st);
    // Long segments can put millions of values in C: a cluster of kEpsCTAs
    // CTAs shares each pass.
    const int ncta = (Lo.L == 1 && Lo.d > (1 << 20)) ? kEpsCTAs : 1;
    if (ncta == 1) return launch_dep(k_solve_eps, dim3(n_seg), dim3(kThreads), 0, st, Lo, sp, Ls, eps, status, info);
    return launch_dep_cluster(k_solve_eps, dim3(n_seg * ncta), dim3(kThreads), 0, ncta, st, Lo, sp, Ls, eps, status,
                              info);
}

}  // namespace gs
