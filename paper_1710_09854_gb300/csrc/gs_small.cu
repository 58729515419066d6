// gs_small.cu -- the cluster-resident path for short gradients (d up to
// 2^21 per worker), Wangni et al., arXiv:1710.09854.
//
// The chunked path (gs_kernels.cu, gs_stream_tma.cu) gives every
// 16384-coordinate chunk to one warp and runs six kernels; a gradient of
// 65536 coordinates is then four warps' work behind six launches, and one of
// 2^20 coordinates sixty-four.  Here one thread-block cluster of up to 12
// CTAs owns one worker: each CTA holds a contiguous share of the worker's
// coordinates (in shared memory when the share fits, else re-read from L2),
// and the passes of Algorithm 3 are plain walks over those shares, combined
// across the cluster in rank order through distributed shared memory:
//
//   pass 0        S = sum |g| (section 3.2, Algorithm 3 step 3);
//   passes 1..j   K_j = #{i : fl64(lam_j |g_i|) >= 1} and the uncapped
//                 mass, then lam_{j+1} = c lam_j (steps 4-10; `iters`
//                 rescalings at most, stopping at c <= 1);
//   decide        one Philox4x32-10 call per 4 coordinates, Z_i = [u_i < p_i]
//                 (section 3) as a kept bit per coordinate (with its sign and
//                 capped bits), the kept counts per 128-coordinate tile and
//                 the statistics at the final lambda;
//   emit          kept coordinates at their output offsets (tile scan plus
//                 the cluster's exclusive prefix in rank order), value g_i / p_i
//                 (g_i when capped, sign(g_i) / lambda otherwise, section 5.3);
//                 for one worker the dense sum (Algorithm 1 step 6) as well.
//
// k_small_sum adds M > 1 workers' kept values in worker order from their
// kept, sign and capped bits (Algorithm 1 step 6).  Every sum is in a fixed
// order: on this path a worker's result is a function of (g, kappa, iters,
// seed, step, worker) and of d, not of M or of the other workers in the call.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "gs_decide.cuh"
#include "gs_device.cuh"
#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {

namespace {

constexpr int kTile = 128;               // coordinates per warp step (4 consecutive per lane)
constexpr int kBatch = 4;                // tiles whose loads a warp has in flight together
// Cluster size the automatic shape stops at: eight 12-CTA clusters of 1024
// threads are resident together on a GB300, while only seven of 13, 14 or
// 16 are (a ninth worker's cluster would wait for a second wave).
constexpr int kAutoCtas = 12;
constexpr int kMaxThreads = 1024;
constexpr int kCacheFloats = 40960;      // shares up to 160 KiB stay in shared memory
constexpr int kSumThreads = 256;
constexpr int kSumStage = 64;            // workers whose parameters k_small_sum stages in shared memory
constexpr int kSumGroup = 8;             // workers whose decision words k_small_sum loads together

struct SmallArgs {
    Layout Lo;
    double kappa;
    int iters;
    int n_per;            // coordinates per CTA (a multiple of kTile)
    int cache;            // 1: each CTA keeps its share of g in shared memory
    int32_t* idx;         // [M][cap] ascending kept indices (worker-local)
    float* val;           // [M][cap] kept values g_i / p_i
    int32_t* nnz;         // [M]
    int64_t cap;
    int* status;
    gs_info_dev* info;    // [M] or NULL
    SegParam* sp;         // [M] parameters for k_small_sum, or NULL
    uint32_t* bits;       // [3][M][wpr] kept / sign / capped bits for k_small_sum, or NULL
    int64_t wpr;          // words per worker row of each plane of `bits`
    float* out;           // M == 1: the dense sum, written here; else NULL
    float div;            // > 0: out is divided by div (the average of Algorithm 1 step 6)
    int accumulate;       // 1: out continues a worker-order sum already in out
};

// Coordinates i0 .. i0 + 3 of worker row m, zero past `hi` (plain cached
// loads: later passes re-read the same lines from L2).
__device__ __forceinline__ void load4(const Layout& Lo, int m, int64_t i0, int64_t hi, float v[4]) {
    const int64_t flat = (int64_t)m * Lo.d + i0;
    if (Lo.dtype == 0) {
        const float* g = static_cast<const float*>(Lo.g) + flat;
        if (i0 + 4 <= hi && (reinterpret_cast<uintptr_t>(g) & 15u) == 0) {
            const float4 t = *reinterpret_cast<const float4*>(g);
            v[0] = t.x;
            v[1] = t.y;
            v[2] = t.z;
            v[3] = t.w;
            return;
        }
#pragma unroll
        for (int s = 0; s < 4; ++s) v[s] = i0 + s < hi ? g[s] : 0.0f;
    } else {
        const uint16_t* g = static_cast<const uint16_t*>(Lo.g) + flat;
        if (i0 + 4 <= hi && (reinterpret_cast<uintptr_t>(g) & 7u) == 0) {
            const uint2 t = *reinterpret_cast<const uint2*>(g);
            v[0] = bf16_bits_to_float(t.x & 0xFFFFu);
            v[1] = bf16_bits_to_float(t.x >> 16);
            v[2] = bf16_bits_to_float(t.y & 0xFFFFu);
            v[3] = bf16_bits_to_float(t.y >> 16);
            return;
        }
#pragma unroll
        for (int s = 0; s < 4; ++s) v[s] = i0 + s < hi ? bf16_bits_to_float(g[s]) : 0.0f;
    }
}

// One CTA's walk over its tiles, in the same order in every pass: warp w
// takes the batches of kBatch consecutive tiles starting at w * kBatch,
// stepping by the CTA's warps; lane l holds coordinates 4l .. 4l + 3 of a
// tile.  The loads of a batch are issued before `f` runs on its tiles: while
// a batch lies wholly inside the share and the row sits on the vector grid,
// with unconditional vector loads (so that all of them are in flight
// together), after that through the bounds-checked loader.  `f(t, v)` is
// called with every lane of the warp (warp-uniform tile test).
template <typename F>
__device__ __forceinline__ void walk(const Layout& Lo, int m, int64_t lo, int64_t hi, int nt, const float4* gc,
                                     F&& f) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int t0 = warp * kBatch;
    if (gc) {
        for (; t0 < nt; t0 += nw * kBatch) {
            float4 x[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                x[u] = t0 + u < nt ? gc[(t0 + u) * 32 + lane] : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const float v[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
                if (t0 + u < nt) f(t0 + u, v);
            }
        }
        return;
    }
    const int64_t base = (int64_t)m * Lo.d + lo;   // flat index of the share's first coordinate
    const int full = (int)((hi - lo) / kTile);     // tiles wholly inside the share
    if (Lo.dtype == 0) {
        const float* g = static_cast<const float*>(Lo.g) + base;
        if ((reinterpret_cast<uintptr_t>(g) & 15u) == 0) {
            for (; t0 + kBatch <= full; t0 += nw * kBatch) {
                float4 x[kBatch];
#pragma unroll
                for (int u = 0; u < kBatch; ++u)
                    x[u] = *reinterpret_cast<const float4*>(g + (int64_t)(t0 + u) * kTile + 4 * lane);
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const float v[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
                    f(t0 + u, v);
                }
            }
        }
    } else {
        const uint16_t* g = static_cast<const uint16_t*>(Lo.g) + base;
        if ((reinterpret_cast<uintptr_t>(g) & 7u) == 0) {
            for (; t0 + kBatch <= full; t0 += nw * kBatch) {
                uint2 x[kBatch];
#pragma unroll
                for (int u = 0; u < kBatch; ++u)
                    x[u] = *reinterpret_cast<const uint2*>(g + (int64_t)(t0 + u) * kTile + 4 * lane);
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const float v[4] = {bf16_bits_to_float(x[u].x & 0xFFFFu), bf16_bits_to_float(x[u].x >> 16),
                                        bf16_bits_to_float(x[u].y & 0xFFFFu), bf16_bits_to_float(x[u].y >> 16)};
                    f(t0 + u, v);
                }
            }
        }
    }
    for (; t0 < nt; t0 += nw * kBatch) {
        float v[kBatch][4];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int t = t0 + u;
            load4(Lo, m, lo + (int64_t)t * kTile + 4 * lane, t < nt ? hi : lo, v[u]);
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u)
            if (t0 + u < nt) f(t0 + u, v[u]);
    }
}

// Block sum of a double-float pair and two ints (butterflies inside warps,
// warps in order); every thread gets the totals.  `sh` holds 33 float4.
__device__ __forceinline__ void block_reduce4(float& h, float& l, int& k, int& x, float4* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xFFFFFFFFu, h, o);
        const float ol = __shfl_xor_sync(0xFFFFFFFFu, l, o);
        df_add(h, l, oh, ol);
        k += __shfl_xor_sync(0xFFFFFFFFu, k, o);
        x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    }
    __syncthreads();
    if (lane == 0) sh[warp] = make_float4(h, l, __int_as_float(k), __int_as_float(x));
    __syncthreads();
    if (warp == 0) {
        const float4 t = lane < nw ? sh[lane] : make_float4(0.0f, 0.0f, __int_as_float(0), __int_as_float(0));
        float hh = t.x, ll = t.y;
        int kk = __float_as_int(t.z), xx = __float_as_int(t.w);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float oh = __shfl_xor_sync(0xFFFFFFFFu, hh, o);
            const float ol = __shfl_xor_sync(0xFFFFFFFFu, ll, o);
            df_add(hh, ll, oh, ol);
            kk += __shfl_xor_sync(0xFFFFFFFFu, kk, o);
            xx += __shfl_xor_sync(0xFFFFFFFFu, xx, o);
        }
        if (lane == 0) sh[32] = make_float4(hh, ll, __int_as_float(kk), __int_as_float(xx));
    }
    __syncthreads();
    const float4 r = sh[32];
    h = r.x;
    l = r.y;
    k = __float_as_int(r.z);
    x = __float_as_int(r.w);
}

// The cluster's totals of (h, l, k) and, for x, the sum over the ranks below
// this CTA and over all ranks.  Each CTA posts its block totals in its own
// shared memory; warp 0 of every CTA reads all posts and adds them in rank
// order, so every CTA holds bit-identical totals.  `post` is double-buffered:
// a post is overwritten two exchanges later, after a cluster barrier that
// every reader of it has passed.
struct Exchange {
    float4 post[2];
    float4 total;     // (h, l, k, x summed over all ranks)
    int x_before;     // x summed over the ranks below this one
};

__device__ __forceinline__ void cluster_reduce(cooperative_groups::cluster_group& cluster, Exchange& ex, int& buf,
                                               float& h, float& l, int& k, int& x, int& x_before, float4* sh) {
    block_reduce4(h, l, k, x, sh);
    const int ncta = (int)cluster.num_blocks(), rank = (int)cluster.block_rank();
    if (threadIdx.x == 0) ex.post[buf] = make_float4(h, l, __int_as_float(k), __int_as_float(x));
    cluster.sync();
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        float4 p = make_float4(0.0f, 0.0f, __int_as_float(0), __int_as_float(0));
        if (lane < ncta) p = *cluster.map_shared_rank(&ex.post[buf], lane);
        float hh = 0.0f, ll = 0.0f;
        int kk = 0, xx = 0, xb = 0;
        for (int r = 0; r < ncta; ++r) {
            const float ph = __shfl_sync(0xFFFFFFFFu, p.x, r);
            const float pl = __shfl_sync(0xFFFFFFFFu, p.y, r);
            const int pk = __shfl_sync(0xFFFFFFFFu, __float_as_int(p.z), r);
            const int px = __shfl_sync(0xFFFFFFFFu, __float_as_int(p.w), r);
            df_add(hh, ll, ph, pl);
            kk += pk;
            if (r < rank) xb += px;
            xx += px;
        }
        if (lane == 0) {
            ex.total = make_float4(hh, ll, __int_as_float(kk), __int_as_float(xx));
            ex.x_before = xb;
        }
    }
    __syncthreads();
    h = ex.total.x;
    l = ex.total.y;
    k = __float_as_int(ex.total.z);
    x = __float_as_int(ex.total.w);
    x_before = ex.x_before;
    buf ^= 1;
}

// Exclusive prefix of cnt[0 .. n) in place (one block; n <= 32 * blockDim.x
// values, each thread scanning a run of consecutive ones).
__device__ __forceinline__ void block_scan_inplace(int32_t* cnt, int n, int* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const int per = (n + (int)blockDim.x - 1) / (int)blockDim.x;
    const int b = threadIdx.x * per, e = min(n, b + per);
    int s = 0;
    for (int i = b; i < e; ++i) s += cnt[i];
    int inc = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += u;
    }
    if (lane == 31) sh[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int w = lane < nw ? sh[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xFFFFFFFFu, w, o);
            if (lane >= o) w += u;
        }
        if (lane < nw) sh[lane] = w;   // inclusive warp totals
    }
    __syncthreads();
    int run = (warp > 0 ? sh[warp - 1] : 0) + inc - s;
    for (int i = b; i < e; ++i) {
        const int c = cnt[i];
        cnt[i] = run;
        run += c;
    }
    __syncthreads();
}

// One cluster per worker (blockIdx.x / cluster size); CTA rank r owns the
// coordinates [r n_per, min(d, (r + 1) n_per)).  Dynamic shared memory:
// the share's values (when cached), one decision bit per coordinate, one
// kept count per tile.  No CTA leaves before the last cluster barrier, so
// every post stays readable while a peer may read it.
__global__ void __launch_bounds__(kMaxThreads) k_small(const __grid_constant__ SmallArgs A) {
    grid_dep_wait();
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int ncta = (int)cluster.num_blocks(), rank = (int)cluster.block_rank();
    const int m = blockIdx.x / ncta;
    const int lane = threadIdx.x & 31;
    const Layout& Lo = A.Lo;
    const int64_t d = Lo.d;
    const int64_t lo = (int64_t)rank * A.n_per;
    const int64_t hi = min(d, lo + (int64_t)A.n_per);
    const int n = hi > lo ? (int)(hi - lo) : 0;
    const int nt = (n + kTile - 1) / kTile;

    extern __shared__ __align__(16) unsigned char dsm[];
    float4* gc = A.cache ? reinterpret_cast<float4*>(dsm) : nullptr;
    uint32_t* bm = reinterpret_cast<uint32_t*>(dsm + (A.cache ? sizeof(float) * A.n_per : 0));   // kept
    uint32_t* bs = bm + A.n_per / 32;   // sign of g
    uint32_t* bc = bs + A.n_per / 32;   // capped (p = 1) and kept
    int32_t* tc = reinterpret_cast<int32_t*>(bc + A.n_per / 32);
    __shared__ float4 sh4[33];
    __shared__ int shi[33];
    __shared__ Exchange ex;
    int buf = 0, xb = 0;

    // Pass 0: S = sum |g| (an unordered NaN threshold sends every value into the sum).
    float h = 0.0f, l = 0.0f;
    int k = 0, x = 0;
    walk(Lo, m, lo, hi, nt, nullptr, [&](int t, const float v[4]) {
        if (gc) gc[t * 32 + lane] = make_float4(v[0], v[1], v[2], v[3]);
        two_sum_add(h, l, (fabsf(v[0]) + fabsf(v[1])) + (fabsf(v[2]) + fabsf(v[3])));
    });
    cluster_reduce(cluster, ex, buf, h, l, k, x, xb, sh4);

    // Algorithm 3's scalar recurrence runs on warp 0 alone (fp64 is slow on
    // this part: every other thread repeating it would cost each step
    // thousands of cycles) and reaches the CTA through shared memory.  Every
    // CTA of the cluster takes the same decisions from the same totals, so
    // the passes (and their barriers) stay in step.
    __shared__ struct {
        double S, lam;
        float acap, lam32, inv32;
        int j, go;
    } sc;
    const double budget = A.kappa * (double)d;
    if (threadIdx.x < 32) {
        const double S0 = (double)h + (double)l;
        const double lam0 = isfinite(S0) && S0 > 0.0 ? budget / S0 : 0.0;
        const float a0 = warp_cap_threshold(lam0);
        if (lane == 0) {
            sc.S = S0;
            sc.lam = lam0;
            sc.acap = a0;
            sc.j = 0;
            sc.go = lam0 > 0.0 && A.iters > 0 ? 1 : 0;
        }
    }
    __syncthreads();
    const double S = sc.S;
    const bool finite = isfinite(S);

    while (sc.go) {
        const float acap_j = sc.acap;
        h = 0.0f;
        l = 0.0f;
        k = 0;
        x = 0;
        walk(Lo, m, lo, hi, nt, gc, [&](int, const float v[4]) {
            float u[4];
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                const float a = fabsf(v[s]);
                const bool c = a >= acap_j;
                k += c ? 1 : 0;
                u[s] = c ? 0.0f : a;
            }
            two_sum_add(h, l, (u[0] + u[1]) + (u[2] + u[3]));
        });
        cluster_reduce(cluster, ex, buf, h, l, k, x, xb, sh4);   // (ends with a block barrier)
        if (threadIdx.x < 32) {
            double lv = sc.lam;
            const int j = sc.j;
            int go = 0;
            float a_new = acap_j;
            const double Aa = lv * ((double)h + (double)l);
            if (Aa != 0.0) {
                const double c = (budget - (double)k) / Aa;
                if (c > 1.0) {
                    lv = c * lv;
                    go = j + 1 < A.iters ? 1 : 0;
                    a_new = warp_cap_threshold(lv);
                    if (lane == 0) {
                        sc.lam = lv;
                        sc.acap = a_new;
                        sc.j = j + 1;
                    }
                }
            }
            if (lane == 0) sc.go = go;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        sc.lam32 = (float)sc.lam;
        sc.inv32 = sc.lam > 0.0 ? (float)(1.0 / sc.lam) : 0.0f;
    }
    __syncthreads();
    const double lam = sc.lam;
    const float acap = sc.acap;
    const int j = sc.j;

    // Decide: one bit per coordinate, kept counts per tile, and the capped
    // count and uncapped mass at the final lambda.  A non-finite gradient keeps nothing.
    Decider dd;
    dd.lam = lam;
    dd.lam32 = sc.lam32;
    dd.a_cap = acap;
    dd.inv_lam32 = sc.inv32;
    const bool any = finite && lam > 0.0;
    const PhiloxStream ph(Lo, Lo.worker0 + (uint32_t)m);
    h = 0.0f;
    l = 0.0f;
    k = 0;
    x = 0;
    walk(Lo, m, lo, hi, nt, gc, [&](int t, const float v[4]) {
        const int64_t i0 = lo + (int64_t)t * kTile + 4 * lane;
        const uint4 w = ph.words((uint32_t)(i0 >> 2));
        uint32_t nib = 0, sgn = 0, cap = 0;
        float u[4];
#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const float a = fabsf(v[s]);
            const bool c = a >= acap;
            k += c ? 1 : 0;
            u[s] = c ? 0.0f : a;
            float vv;
            if (any && dd(v[s], word_of(w, s), vv)) nib |= 1u << s;
            sgn |= (__float_as_uint(v[s]) >> 31) << s;
            cap |= (c ? 1u : 0u) << s;
        }
        two_sum_add(h, l, (u[0] + u[1]) + (u[2] + u[3]));
        // Lanes 8q .. 8q + 7 hold the 32 coordinates of word q of the tile.
        const int sft = 4 * (lane & 7);
        uint32_t wk = nib << sft, ws = sgn << sft, wc = cap << sft;
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) {
            wk |= __shfl_xor_sync(0xFFFFFFFFu, wk, o);
            ws |= __shfl_xor_sync(0xFFFFFFFFu, ws, o);
            wc |= __shfl_xor_sync(0xFFFFFFFFu, wc, o);
        }
        if ((lane & 7) == 0) {
            const int wi = t * 4 + (lane >> 3);
            bm[wi] = wk;
            bs[wi] = ws;
            bc[wi] = wc & wk;   // capped and kept
        }
        const int c = __reduce_add_sync(0xFFFFFFFFu, __popc(nib));
        if (lane == 0) tc[t] = c;
        x += lane == 0 ? c : 0;
    });
    cluster_reduce(cluster, ex, buf, h, l, k, x, xb, sh4);   // (ends with a block barrier: bitmaps, tc complete)
    const int64_t total = x;
    block_scan_inplace(tc, nt, shi);

    // Emit: a lane per 32-coordinate word, each kept coordinate at the
    // cluster's prefix + its tile block's offset + the lane's rank in the
    // block, its value g_i when capped (the only read of g here) and
    // sign(g_i) / lambda otherwise.  Entries past the capacity are not
    // written and (as in the chunked path, whose sum reads the written lists)
    // not summed either: their bits are cleared before any sum reads them.
    const int64_t row = (int64_t)m * A.cap;
    const float inv = dd.inv_lam32;
    const float* gcf = reinterpret_cast<const float*>(gc);
    auto g_at = [&](int64_t i) { return gcf ? gcf[i - lo] : load_one(Lo, m, i); };
    {
        const int warp = threadIdx.x >> 5, nw = blockDim.x >> 5, nwords = nt * 4;
        for (int b = warp; b * 32 < nwords; b += nw) {
            const int wi = b * 32 + lane;
            uint32_t kw = wi < nwords ? bm[wi] : 0u;
            const uint32_t sw = wi < nwords ? bs[wi] : 0u, cw = wi < nwords ? bc[wi] : 0u;
            const int cnt = __popc(kw);
            int inc = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                if (lane >= o) inc += y;
            }
            int64_t pos = (int64_t)xb + tc[b * 8] + (inc - cnt);
            uint32_t drop = 0, rest = kw;
            while (rest) {
                const int sb = __ffs(rest) - 1;
                rest &= rest - 1u;
                const int64_t i = lo + (int64_t)wi * 32 + sb;
                if (pos < A.cap) {
                    A.idx[row + pos] = (int32_t)i;
                    A.val[row + pos] = (cw >> sb) & 1u ? g_at(i) : ((sw >> sb) & 1u ? -inv : inv);
                } else {
                    drop |= 1u << sb;
                }
                ++pos;
            }
            if (drop) bm[wi] = kw & ~drop;   // this lane's own word
        }
    }
    __syncthreads();

    float* out = A.out;
    if (out) {
        // One worker: the dense sum (Algorithm 1 step 6) from the bits, four
        // consecutive coordinates per lane.
        const int warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
        const int q = lane >> 3, sft = 4 * (lane & 7);
        for (int t = warp; t < nt; t += nw) {
            const int wi = t * 4 + q;
            const uint32_t kn = (bm[wi] >> sft) & 0xFu, sn = (bs[wi] >> sft) & 0xFu, cn = (bc[wi] >> sft) & 0xFu;
            const int64_t i0 = lo + (int64_t)t * kTile + 4 * lane;
            float o[4];
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                float acc = A.accumulate && i0 + s < hi ? out[i0 + s] : 0.0f;
                if ((kn >> s) & 1u) acc += (cn >> s) & 1u ? g_at(i0 + s) : ((sn >> s) & 1u ? -inv : inv);
                o[s] = A.div > 0.0f ? __fdiv_rn(acc, A.div) : acc;
            }
            float* dst = out + i0;
            if (i0 + 4 <= hi && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
                *reinterpret_cast<float4*>(dst) = make_float4(o[0], o[1], o[2], o[3]);
            } else {
#pragma unroll
                for (int s = 0; s < 4; ++s)
                    if (i0 + s < hi) dst[s] = o[s];
            }
        }
    }

    if (A.bits) {
        // The bits of the written entries (kept, sign, capped) for the
        // worker-order sum of M > 1 workers.
        const size_t w0 = (size_t)(lo >> 5);
        uint32_t* dk = A.bits + (size_t)m * A.wpr + w0;
        uint32_t* ds = A.bits + ((size_t)A.Lo.M + m) * A.wpr + w0;
        uint32_t* dc = A.bits + ((size_t)2 * A.Lo.M + m) * A.wpr + w0;
        for (int i = threadIdx.x; i < nt * 4; i += blockDim.x) {
            if (w0 + i < (size_t)A.wpr) {
                dk[i] = bm[i];
                ds[i] = bs[i];
                dc[i] = bc[i] & bm[i];
            }
        }
    }

    if (rank == 0 && threadIdx.x == 0) {
        const double Su = (double)h + (double)l;
        const double K = (double)k;
        const double sum_p = lam > 0.0 ? K + lam * Su : 0.0;
        A.nnz[m] = (int32_t)total;
        if (total > A.cap) atomicOr(A.status, kStCapacity);
        if (!finite) atomicOr(A.status, kStNonfinite);
        if (A.sp) {
            SegParam& P = A.sp[m];
            P.lam = lam;
            P.lam32 = dd.lam32;
            P.a_cap = acap;
            P.inv_lam32 = inv;
            P.l1 = S;
            P.capped = (long long)K;
            P.sum_p = sum_p;
            P.iters_run = j;
            P.flags = finite ? 0 : kSegNonfinite;
        }
        if (A.info) {
            A.info[m].lambda = lam;
            A.info[m].sum_p = sum_p;
            A.info[m].capped = (int64_t)K;
            A.info[m].iters_run = j;
            A.info[m].flags = 0;
        }
    }
    cluster.sync();   // peers may still read this CTA's posts until here
}

// Algorithm 1 step 6 for M > 1 workers of the small path: out_i = the fp32
// sum, in worker order, of the kept values of coordinate i (g_i when capped,
// sign(g_i) / lambda otherwise), from each worker's kept / sign / capped bits
// (`bits` holds the three planes [3][M][wpr]); g is read for capped entries
// only.  The same adds, in the same order, as the chunked path's sum over
// compacted lists.
__global__ void __launch_bounds__(kSumThreads) k_small_sum(const __grid_constant__ Layout Lo,
                                                           const SegParam* __restrict__ sp,
                                                           const uint32_t* __restrict__ bits, int64_t wpr,
                                                           float div, int accumulate, float* out) {
    grid_dep_wait();
    __shared__ float s_inv[kSumStage];
    for (int m = threadIdx.x; m < min(Lo.M, kSumStage); m += blockDim.x) s_inv[m] = sp[m].inv_lam32;
    __syncthreads();
    const int64_t d = Lo.d, nq = (d + 3) >> 2;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i0 = q * 4;
        float acc[4];
#pragma unroll
        for (int s = 0; s < 4; ++s) acc[s] = accumulate && i0 + s < d ? out[i0 + s] : 0.0f;
        const int sh = (int)(i0 & 31);
        for (int m0 = 0; m0 < Lo.M; m0 += kSumGroup) {
            // The group's words of all three planes first (independent
            // loads), then the kept values in worker order.
            uint32_t kw[kSumGroup], sw[kSumGroup], cw[kSumGroup];
#pragma unroll
            for (int u = 0; u < kSumGroup; ++u) {
                kw[u] = sw[u] = cw[u] = 0u;
                if (m0 + u < Lo.M) {
                    const size_t wi = (size_t)(m0 + u) * wpr + (i0 >> 5);
                    kw[u] = __ldg(bits + wi);
                    sw[u] = __ldg(bits + (size_t)Lo.M * wpr + wi);
                    cw[u] = __ldg(bits + (size_t)2 * Lo.M * wpr + wi);
                }
            }
#pragma unroll
            for (int u = 0; u < kSumGroup; ++u) {
                const uint32_t nib = (kw[u] >> sh) & 0xFu;
                if (nib == 0u) continue;
                const int m = m0 + u;
                const float inv = m < kSumStage ? s_inv[m] : sp[m].inv_lam32;
#pragma unroll
                for (int s = 0; s < 4; ++s) {
                    if ((nib >> s) & 1u)
                        acc[s] += (cw[u] >> (sh + s)) & 1u ? load_one(Lo, m, i0 + s)
                                                          : ((sw[u] >> (sh + s)) & 1u ? -inv : inv);
                }
            }
        }
        if (div > 0.0f) {
#pragma unroll
            for (int s = 0; s < 4; ++s) acc[s] = __fdiv_rn(acc[s], div);
        }
        float* dst = out + i0;
        if (i0 + 4 <= d && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
            *reinterpret_cast<float4*>(dst) = make_float4(acc[0], acc[1], acc[2], acc[3]);
        } else {
#pragma unroll
            for (int s = 0; s < 4; ++s)
                if (i0 + s < d) dst[s] = acc[s];
        }
    }
}

// Cluster size and share per CTA for a row of d coordinates: shares of about
// 4096 coordinates, up to kAutoCtas CTAs, and never above kMaxShare (whose
// three bitmaps and tile counts take 208 KiB).  A function of d alone: the
// shape fixes the order of every sum, so a row's result depends on nothing
// else.
constexpr int64_t kMaxShare = (int64_t)1 << 19;
void small_shape(int64_t d, int& ncta, int& n_per) {
    ncta = (int)std::min<int64_t>(kAutoCtas, std::max<int64_t>(1, (d + 4095) / 4096));
    ncta = (int)std::max<int64_t>(ncta, (d + kMaxShare - 1) / kMaxShare);
    const int64_t per = (d + ncta - 1) / ncta;
    n_per = (int)((per + kTile - 1) / kTile * kTile);
}

}  // namespace

bool small_path_eligible(int64_t d) { return d >= 1 && d <= kSmallMaxD; }

size_t small_scratch_bytes(int M, int64_t d) {
    const size_t wpr = (size_t)((d + 31) / 32);
    return ((sizeof(SegParam) * (size_t)M + 255) & ~(size_t)255) + 3 * sizeof(uint32_t) * wpr * (size_t)M;
}

cudaError_t launch_small(const Layout& Lo, double kappa, int iters, int32_t* idx, float* val, int32_t* nnz,
                         int64_t cap, int* status, gs_info_dev* info, float* out, bool average, bool accumulate,
                         void* scratch, cudaStream_t st) {
    int ncta, n_per;
    small_shape(Lo.d, ncta, n_per);
    const int nt = n_per / kTile;
    const bool cache = n_per <= kCacheFloats;
    int threads = 32 * ((nt + kBatch - 1) / kBatch);
    threads = std::max(64, std::min(kMaxThreads, threads));
    const size_t smem = (cache ? sizeof(float) * (size_t)n_per : 0) + 3 * sizeof(uint32_t) * (size_t)(n_per / 32) +
                        sizeof(int32_t) * (size_t)nt;
    SmallArgs A;
    A.Lo = Lo;
    A.kappa = kappa;
    A.iters = iters;
    A.n_per = n_per;
    A.cache = cache ? 1 : 0;
    A.idx = idx;
    A.val = val;
    A.nnz = nnz;
    A.cap = cap;
    A.status = status;
    A.info = info;
    A.sp = nullptr;
    A.bits = nullptr;
    A.wpr = (Lo.d + 31) / 32;
    A.out = nullptr;
    A.div = average ? (float)Lo.M : 0.0f;
    A.accumulate = accumulate ? 1 : 0;
    const bool sum_kernel = out != nullptr && Lo.M > 1;
    if (out && !sum_kernel) A.out = out;
    if (sum_kernel) {
        A.sp = static_cast<SegParam*>(scratch);
        A.bits = reinterpret_cast<uint32_t*>(static_cast<char*>(scratch) +
                                             ((sizeof(SegParam) * (size_t)Lo.M + 255) & ~(size_t)255));
    }
    set_launch_error_site("k_small launch");
    cudaError_t e = cudaFuncSetAttribute(k_small, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_small, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    {
        TraceScope ts(kKSmall, st);
        e = launch_dep_cluster(k_small, dim3(Lo.M * ncta), dim3(threads), smem, ncta, st, A);
    }
    if (e != cudaSuccess || !sum_kernel) return e;
    set_launch_error_site("k_small_sum launch");
    const int64_t nq = (Lo.d + 3) / 4;
    const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>((nq + kSumThreads - 1) / kSumThreads,
                                                                   (int64_t)device_sm_count() * 8));
    TraceScope ts(kKSmallSum, st);
    return launch_dep(k_small_sum, dim3(blocks), dim3(kSumThreads), 0, st, Lo, static_cast<const SegParam*>(A.sp),
                      static_cast<const uint32_t*>(A.bits), A.wpr, A.div, A.accumulate, out);
}

}  // namespace gs
