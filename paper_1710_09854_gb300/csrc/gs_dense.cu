// gs_dense.cu -- the dense code of Q(g) (section 3.3, last paragraph): the
// vector q~ in {0, +1, -1, 2}^d (0: dropped; sign(g_i): kept with p_i < 1;
// 2: kept with p_i = 1) entropy coded under the static model the paper
// prices it with, P(s) = d_s / d, whose ideal length is
// sum_s d_s log2(d / d_s) <= 2d bits.
//
// The model is coded one non-zero symbol at a time: the run g of zeros
// before it under the model's geometric law P(g) = (1 - p0) p0^g
// (p0 = d_0 / d), then its value t under P(t) = d_t / (d - d_0).  The run is
// sent as v = g + 1: its bit length l = floor(log2 v) with
// P(l) = p0^(2^l - 1) (1 - p0^(2^l)), then its l bits below the leading one
// (most significant first), bit k being 1 with probability
// p0^(2^k) / (1 + p0^(2^k)); given l these bits are independent and their
// probabilities multiply back to P(g), so the events cost exactly what the
// symbols would one by one.
//
// Format of one vector (16-bit words; two-word integers low word first):
//   header     d, d_{+1}, d_{-1}, d_2 (two words each), log2 K (one word)
//   directory  per chunk of K consecutive non-zero symbols: the index of its
//              first non-zero (two words) and its stream length (one word)
//   streams    one rANS stream per chunk, in chunk order; the chunk's first
//              non-zero is placed by the directory (its run is not coded).
// rANS: integer frequencies over 2^15 (model below), state x in
// [2^15, 2^31), 16-bit renormalisation words.  A chunk's coding steps, in
// decode order, are (run bit length, run bits) for every non-zero but the
// first, then the value; the encoder visits them last to first starting from
// x = 2^15, emitting x's low word (x >>= 16) while x >= f 2^16 and setting
// x = floor(x / f) 2^15 + (x mod f) + c; the stream is the final state (high
// word first) followed by the emitted words last to first.
//
// Frequencies from the counts, in exactly rounded fp64 in this order:
// p0 = d_0 / d; s_0 = p0, s_{k+1} = s_k s_k; bit k: r = s_k / (1 + s_k),
// f_1 = (floor(r 2^16) + 1) >> 1 clamped to [1, 2^15 - 1]; length l:
// P = pi_l (1 - s_l), pi_0 = 1, pi_{l+1} = pi_l s_l; value t: n_t / nz; in a
// multi-symbol model every symbol that can occur gets max(1, floor(P 2^15))
// and the largest (first on ties) absorbs the difference to 2^15.
//
// Work is per non-zero symbol (about 2 + log2 of its run coding steps), not
// per coordinate.  The two hybrid lists (Q_A: p = 1; Q_B: the rest) are
// first merged into one ascending sequence of (index, value) per worker (a
// warp per chunk, merge-path placement in shared memory); then one thread
// per chunk runs the chunk's rANS chain from the end of its stretch, once to
// count its words and, after a per-worker scan of the counts, once to write
// them.  The decoder runs one thread per chunk too.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "gs_device.cuh"
#include "gs_launch.h"
#include "gs_trace.h"

namespace gs {
namespace {

constexpr int kScale = 15;
constexpr uint32_t kM = 1u << kScale;          // total frequency
constexpr uint32_t kLow = 1u << 15;            // lower end of the state interval
constexpr int kLens = 31;                      // run bit lengths 0 .. 30
constexpr int kBitModels = 30;
constexpr int kHeaderWords = 9;
constexpr int kDirWords = 3;

// One symbol of a model: frequency, cumulative start, and the exact
// reciprocal pair for floor(x / f) = (x * rcp) >> sh on x < 2^31.
struct Sym {
    uint32_t f, c, rcp, sh;
};

struct DenseModel {
    Sym len[kLens];
    Sym bit0[kBitModels], bit1[kBitModels];
    Sym val[3];                 // +1, -1, 2
    uint32_t len_c[kLens + 1];  // cumulative starts for the decoder's search
    uint8_t len_lut[256];       // the length whose range holds slot 128 b: where the decoder's search starts
    int64_t n_pos, n_neg, n_cap, nz;
    int64_t n_chunks, chunk0;   // chunks of this worker, and the chunks of all workers before it
    int64_t words;              // total words of the worker's code (after the scan)
    int log2_k;                 // non-zero symbols per chunk (log2)
    int status;                 // unused
};

// floor(x / f) = (x * rcp) >> sh for every x < 2^31, with s = ceil(log2 f),
// rcp = ceil(2^(31+s) / f), sh = 31 + s: rcp = 2^(31+s)/f + e (0 <= e < 1), so
// the product overshoots x / f by x e / 2^(31+s) < 2^-s <= 1 / f, less than the
// gap between x / f and the next integer.
__device__ __forceinline__ Sym make_sym(uint32_t f, uint32_t c) {
    Sym y;
    y.f = f;
    y.c = c;
    int s = 0;
    while ((1u << s) < f) ++s;
    y.sh = 31 + s;
    y.rcp = f ? (uint32_t)((((unsigned long long)1 << y.sh) + f - 1) / f) : 0u;
    return y;
}

// max(1, floor(P 2^15)) for the symbols that can occur; the largest absorbs the rest.
__device__ void quantise(const double* P, const bool* can, int n, uint32_t* f) {
    long long sum = 0;
    int best = 0;
    for (int s = 0; s < n; ++s) {
        uint32_t q = 0;
        if (can[s]) {
            const double t = floor(__dmul_rn(P[s], (double)kM));
            q = t < 1.0 ? 1u : (uint32_t)t;
        }
        f[s] = q;
        sum += q;
        if (q > f[best]) best = s;
    }
    f[best] = (uint32_t)((long long)f[best] + (long long)kM - sum);
}

// A worker's model, built by a whole block (any blockDim >= 32) from its
// symbol counts: p0 = d_0 / d; the bit-length model P(l) = p0^(2^l - 1)
// (1 - p0^(2^l)) and the bit models P(bit k = 1) = s_k / (1 + s_k) with
// s_k = p0^(2^k), each quantised as the oracle does; the value model d_t / nz.  The two serial
// chains (the repeated squaring of p0 and the running product before each
// length) stay on thread 0; the frequencies' divisions run side by side.
__device__ void build_model_block(int64_t d, int64_t n_pos, int64_t n_neg, int64_t n_cap, DenseModel& m) {
    __shared__ double s_sq[kLens], s_P[kLens];
    __shared__ uint32_t s_f[kLens], s_c[kLens + 1], s_fv[3], s_cv[3];
    const int tid = threadIdx.x;
    const int64_t nz = n_pos + n_neg + n_cap;
    if (tid == 0) {
        m.n_pos = n_pos;
        m.n_neg = n_neg;
        m.n_cap = n_cap;
        m.nz = nz;
        double sq = __ddiv_rn((double)(d - nz), (double)d);
        double pi = 1.0;
        for (int l = 0; l < kLens; ++l) {
            s_sq[l] = sq;
            s_P[l] = __dmul_rn(pi, __dsub_rn(1.0, sq));
            pi = __dmul_rn(pi, sq);
            sq = __dmul_rn(sq, sq);
        }
    }
    __syncthreads();
    for (int k = tid; k < kBitModels; k += blockDim.x) {
        const double r = __ddiv_rn(s_sq[k], __dadd_rn(1.0, s_sq[k]));
        uint32_t f1 = ((uint32_t)floor(__dmul_rn(r, 65536.0)) + 1u) >> 1;
        f1 = min(max(f1, 1u), kM - 1u);
        m.bit0[k] = make_sym(kM - f1, 0u);
        m.bit1[k] = make_sym(f1, kM - f1);
    }
    for (int l = tid; l < kLens; l += blockDim.x) {
        const double t = floor(__dmul_rn(s_P[l], (double)kM));
        s_f[l] = t < 1.0 ? 1u : (uint32_t)t;
    }
    __syncthreads();
    if (tid == 0) {
        // quantise's remainder to the first most probable length, then the starts
        long long sum = 0;
        int best = 0;
        for (int l = 0; l < kLens; ++l) {
            sum += s_f[l];
            if (s_f[l] > s_f[best]) best = l;
        }
        s_f[best] = (uint32_t)((long long)s_f[best] + (long long)kM - sum);
        uint32_t c = 0;
        for (int l = 0; l < kLens; ++l) {
            s_c[l] = c;
            c += s_f[l];
        }
        s_c[kLens] = c;
        // the value model (three symbols)
        const int64_t nt[3] = {n_pos, n_neg, n_cap};
        double Pv[3];
        bool cv[3];
        for (int t = 0; t < 3; ++t) {
            Pv[t] = nz > 0 ? __ddiv_rn((double)nt[t], (double)nz) : 0.0;
            cv[t] = nt[t] > 0;
        }
        if (nz == 0) cv[0] = true;   // an unused model still sums to 2^15
        uint32_t fv[3];
        quantise(Pv, cv, 3, fv);
        uint32_t cc = 0;
        for (int t = 0; t < 3; ++t) {
            s_fv[t] = fv[t];
            s_cv[t] = cc;
            cc += fv[t];
        }
    }
    __syncthreads();
    for (int l = tid; l <= kLens; l += blockDim.x) {
        m.len_c[l] = s_c[l];
        if (l < kLens) m.len[l] = make_sym(s_f[l], s_c[l]);
    }
    for (int b = tid; b < 256; b += blockDim.x) {
        const uint32_t slot = (uint32_t)b << 7;
        int l = 0;
        while (l + 1 < kLens && s_c[l + 1] <= slot) ++l;
        m.len_lut[b] = (uint8_t)l;
    }
    for (int t = tid; t < 3; t += blockDim.x) m.val[t] = make_sym(s_fv[t], s_cv[t]);
    __syncthreads();
}

// The two hybrid lists of one worker, ascending: Q_A indices (value 2) and
// Q_B codes 2 i + [g_i < 0] (value -1 or +1).
struct Lists2 {
    const int32_t* a;
    const uint32_t* b;
    int na, nb;
    __device__ __forceinline__ int bi(int j) const { return (int)(b[j] >> 1); }
};

// Number of Q_A entries among the r smallest indices of the merge.
__device__ __forceinline__ int merge_split(const Lists2& L, int r) {
    int lo = max(0, r - L.nb), hi = min(r, L.na);
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (L.a[mid] < L.bi(r - mid - 1)) lo = mid + 1; else hi = mid;
    }
    return lo;
}

// One rANS coding step on the encoder's state; `w` (NULL while counting)
// receives emitted word number n at w[-n] (the stream is stored last-first).
__device__ __forceinline__ void put(uint32_t& x, const Sym& s, uint16_t* w, int& n) {
    if (x >= (s.f << 16)) {
        if (w) w[-n] = (uint16_t)(x & 0xFFFFu);
        ++n;
        x >>= 16;
    }
    const uint32_t q = (uint32_t)(((unsigned long long)x * s.rcp) >> s.sh);
    x += s.c + q * (kM - s.f);
}

// Shared memory of one warp's chunk: the worker's model, the chunk's
// stretches of the two lists, and their merge (indices and value symbols).
constexpr int kDenseWarps = 4;   // chunks (warps) per block

__host__ __device__ constexpr size_t model_bytes() { return (sizeof(DenseModel) + 15) & ~(size_t)15; }
__host__ __device__ constexpr size_t warp_bytes(int K) {
    return model_bytes() + (size_t)K * (sizeof(int32_t) + sizeof(uint32_t) + sizeof(int32_t) + 1) + 16;
}

struct Staged {
    DenseModel* md;
    int32_t* sa;     // the chunk's Q_A stretch
    uint32_t* sb;    // its Q_B stretch
    int32_t* idx;    // merged indices
    uint8_t* typ;    // merged value symbols (0: +1, 1: -1, 2: 2)
};

__device__ __forceinline__ Staged staged_at(unsigned char* base, int K) {
    Staged t;
    t.md = reinterpret_cast<DenseModel*>(base);
    t.sa = reinterpret_cast<int32_t*>(base + model_bytes());
    t.sb = reinterpret_cast<uint32_t*>(t.sa + K);
    t.idx = reinterpret_cast<int32_t*>(t.sb + K);
    t.typ = reinterpret_cast<uint8_t*>(t.idx + K);
    return t;
}


// The warp stages the merge ranks [r0, r1) of worker lists L: both lists'
// stretches are loaded, then each lane places its output positions by a
// merge-path search in shared memory.
__device__ void stage_merge(const Lists2& L, int r0, int r1, const Staged& t, int lane) {
    int ia0 = 0, ia1 = 0;
    if (lane == 0) ia0 = merge_split(L, r0);
    if (lane == 1) ia1 = merge_split(L, r1);
    ia0 = __shfl_sync(0xFFFFFFFFu, ia0, 0);
    ia1 = __shfl_sync(0xFFFFFFFFu, ia1, 1);
    const int ib0 = r0 - ia0, na = ia1 - ia0, nb = (r1 - ia1) - ib0;
    for (int i = lane; i < na; i += 32) t.sa[i] = L.a[ia0 + i];
    for (int i = lane; i < nb; i += 32) t.sb[i] = L.b[ib0 + i];
    __syncwarp();
    for (int p = lane; p < r1 - r0; p += 32) {
        int lo = max(0, p - nb), hi = min(p, na);   // A entries among the p smallest
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (t.sa[mid] < (int)(t.sb[p - mid - 1] >> 1)) lo = mid + 1; else hi = mid;
        }
        const bool from_a = lo < na && (p - lo >= nb || t.sa[lo] < (int)(t.sb[p - lo] >> 1));
        if (from_a) {
            t.idx[p] = t.sa[lo];
            t.typ[p] = 2;
        } else {
            const uint32_t code = t.sb[p - lo];
            t.idx[p] = (int32_t)(code >> 1);
            t.typ[p] = (uint8_t)(code & 1u);
        }
    }
    __syncwarp();
}

__device__ __forceinline__ void put32(uint16_t* w, uint32_t v) {
    w[0] = (uint16_t)(v & 0xFFFFu);
    w[1] = (uint16_t)(v >> 16);
}
__device__ __forceinline__ uint32_t get32(const uint16_t* w) { return (uint32_t)w[0] | ((uint32_t)w[1] << 16); }

// Per-worker count of the -1 symbols among the Q_B codes (grid: x over the
// list, y over workers).
__global__ void k_dense_count(const uint32_t* __restrict__ qb, const int32_t* __restrict__ n_b, int64_t cap,
                              unsigned long long* neg) {
    grid_dep_wait();
    const int m = blockIdx.y;
    const int64_t n = min((int64_t)n_b[m], cap);
    const uint32_t* b = qb + (int64_t)m * cap;
    int cnt = 0;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += (int64_t)gridDim.x * blockDim.x)
        cnt += (int)(b[j] & 1u);
    cnt = warp_sum(cnt);
    if ((threadIdx.x & 31) == 0 && cnt) atomicAdd(neg + m, (unsigned long long)cnt);
}

// One block per worker: its model and chunk count, the header words, and
// the chunks of all workers before it (from the list lengths, which every
// block reads; the last block writes the total).
__device__ __forceinline__ bool lists_ok(int64_t na, int64_t nb, int64_t cap, int64_t d) {
    return !(na > cap || nb > cap || na < 0 || nb < 0 || na + nb > d);
}

__global__ void k_dense_setup(const int32_t* __restrict__ n_a, const int32_t* __restrict__ n_b,
                              const unsigned long long* __restrict__ neg, int M, int64_t d, int64_t cap, int log2_k,
                              DenseModel* md, uint16_t* words, int64_t word_cap, int64_t* total_chunks, int* status) {
    grid_dep_wait();
    __shared__ long long s_red[32];
    const int m = blockIdx.x, tid = threadIdx.x;
    const int64_t na = n_a[m], nb = n_b[m];
    const bool ok = lists_ok(na, nb, cap, d);
    DenseModel& mm = md[m];
    if (ok) build_model_block(d, nb - (int64_t)neg[m], (int64_t)neg[m], na, mm);
    else build_model_block(d, 0, 0, 0, mm);
    // chunks of the workers before this one
    long long before = 0;
    for (int j = tid; j < m; j += blockDim.x) {
        const int64_t a = n_a[j], bb = n_b[j];
        if (lists_ok(a, bb, cap, d)) before += (a + bb + ((int64_t)1 << log2_k) - 1) >> log2_k;
    }
    before = warp_sum(before);
    if ((tid & 31) == 0) s_red[tid >> 5] = before;
    __syncthreads();
    if (tid == 0) {
        long long c0 = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) c0 += s_red[w];
        mm.n_chunks = ok ? (mm.nz + ((int64_t)1 << log2_k) - 1) >> log2_k : 0;
        mm.chunk0 = c0;
        mm.log2_k = log2_k;
        mm.status = 0;
        if (!ok) atomicOr(status, kStInvalid);   // lists that overflowed their capacity cannot be coded
        if (word_cap >= kHeaderWords) {
            uint16_t* w = words + (int64_t)m * word_cap;
            put32(w, (uint32_t)d);
            put32(w + 2, (uint32_t)mm.n_pos);
            put32(w + 4, (uint32_t)mm.n_neg);
            put32(w + 6, (uint32_t)mm.n_cap);
            w[8] = (uint16_t)log2_k;
        }
        if (m == M - 1) *total_chunks = c0 + mm.n_chunks;
    }
}

// The worker of global chunk g (chunk0 ascending).
__device__ __forceinline__ int chunk_worker(const DenseModel* md, int M, int64_t g) {
    int a = 0, b = M - 1;
    while (a < b) {
        const int mid = (a + b + 1) >> 1;
        if (md[mid].chunk0 <= g) a = mid; else b = mid - 1;
    }
    return a;
}

// The merge of every worker's two lists into one ascending sequence of
// (index, value symbol), one warp per chunk: the warp stages the chunk's
// stretches in shared memory, merges them there, and writes the chunk's
// stretch of the merged sequence (worker m's at m * stride).
__global__ void __launch_bounds__(kDenseWarps * 32)
    k_dense_merge(const int32_t* __restrict__ qa, const uint32_t* __restrict__ qb, const DenseModel* __restrict__ md,
                  int M, int64_t cap, int log2_k, const int64_t* __restrict__ total_chunks, int32_t* m_idx,
                  uint8_t* m_typ, int64_t stride) {
    grid_dep_wait();
    extern __shared__ __align__(16) unsigned char dsm[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int K = 1 << log2_k;
    const Staged t = staged_at(dsm + warp * warp_bytes(K), K);
    const int64_t total = *total_chunks;
    for (int64_t g = (int64_t)blockIdx.x * kDenseWarps + warp; g < total; g += (int64_t)gridDim.x * kDenseWarps) {
        const int m = chunk_worker(md, M, g);
        const int64_t i = g - md[m].chunk0;
        const int r0 = (int)(i << log2_k), r1 = (int)min((int64_t)r0 + K, md[m].nz);
        Lists2 L;
        L.a = qa + (int64_t)m * cap;
        L.b = qb + (int64_t)m * cap;
        L.na = (int)md[m].n_cap;
        L.nb = (int)(md[m].n_pos + md[m].n_neg);
        stage_merge(L, r0, r1, t, lane);
        int32_t* oi = m_idx + (int64_t)m * stride + r0;
        uint8_t* ot = m_typ + (int64_t)m * stride + r0;
        for (int p = lane; p < r1 - r0; p += 32) {
            oi[p] = t.idx[p];
            ot[p] = t.typ[p];
        }
        __syncwarp();
    }
}

// rANS encoding of merge ranks [r0, r1) of one worker from its merged
// sequence (one thread): returns the number of emitted words; with out,
// writes the stream there (n_emitted from the counting pass).  Symbols are
// coded last to first; the value symbols and preceding indices of the next
// four are loaded while the current four are coded.
struct Batch {
    uint32_t typ4;   // value symbols of ranks j, j-1, j-2, j-3 (a byte each)
    int prev[4];     // index of rank j-u-1 (the end of rank j-u's run)
};

__device__ __forceinline__ Batch load_batch(const int32_t* idx, const uint8_t* typ, int j, int r0) {
    Batch b;
    b.typ4 = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int jj = j - u;
        if (jj >= r0) b.typ4 |= (uint32_t)typ[jj] << (8 * u);
        b.prev[u] = jj - 1 >= r0 ? idx[jj - 1] : 0;
    }
    return b;
}

__device__ __forceinline__ int encode_seq(const DenseModel& md, const int32_t* idx, const uint8_t* typ, int r0,
                                          int r1, uint16_t* out, int n_emitted) {
    uint32_t x = kLow;
    int n = 0;
    uint16_t* w = out ? out + 2 + (n_emitted - 1) : nullptr;
    int cur = idx[r1 - 1];
    Batch b = load_batch(idx, typ, r1 - 1, r0);
    for (int j = r1 - 1; j >= r0; j -= 4) {
        const Batch nb = j - 4 >= r0 ? load_batch(idx, typ, j - 4, r0) : b;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int jj = j - u;
            if (jj < r0) break;
            put(x, md.val[(b.typ4 >> (8 * u)) & 0xFFu], w, n);
            if (jj == r0) break;
            const int prev = b.prev[u];
            const uint32_t v = (uint32_t)(cur - prev);   // run of zeros + 1
            const int l = 31 - __clz(v);
            for (int k = 0; k < l; ++k) put(x, ((v >> k) & 1u) ? md.bit1[k] : md.bit0[k], w, n);
            put(x, md.len[l], w, n);
            cur = prev;
        }
        b = nb;
    }
    if (out) {
        out[0] = (uint16_t)(x >> 16);
        out[1] = (uint16_t)(x & 0xFFFFu);
    }
    return n;
}

// The models of the workers whose chunks one block handles, staged in
// shared memory: the coding steps read them there, where the global stores
// of the coded words cannot alias them (a generic pointer could, which
// would make every step reload its symbol).  kStageModels workers cover a
// block's 128 consecutive chunks unless workers have fewer chunks than that.
constexpr int kStageModels = 4;

__device__ __forceinline__ void stage_models(DenseModel* dst, const DenseModel* __restrict__ src, int n) {
    const int words = n * (int)(sizeof(DenseModel) / 4);
    const uint32_t* s = reinterpret_cast<const uint32_t*>(src);
    uint32_t* d = reinterpret_cast<uint32_t*>(dst);
    for (int i = threadIdx.x; i < words; i += blockDim.x) d[i] = s[i];
}

// Counting pass (kWrite false): each chunk's stream length and first index.
// Writing pass: each chunk's stream at its offset (codes that fit only).
// One thread per chunk, reading the merged sequence.
template <bool kWrite>
__global__ void __launch_bounds__(128)
    k_dense_encode(const int32_t* __restrict__ m_idx, const uint8_t* __restrict__ m_typ, int64_t stride,
                   const DenseModel* __restrict__ md, int M, int log2_k, const int64_t* __restrict__ total_chunks,
                   int32_t* ch_len, int32_t* ch_first, const int64_t* __restrict__ ch_off, uint16_t* words,
                   int64_t word_cap) {
    grid_dep_wait();
    __shared__ DenseModel s_md[kStageModels];
    const int64_t total = *total_chunks;
    for (int64_t g0 = (int64_t)blockIdx.x * blockDim.x; g0 < total; g0 += (int64_t)gridDim.x * blockDim.x) {
        const int m_lo = chunk_worker(md, M, g0);
        const int m_hi = chunk_worker(md, M, min(g0 + (int64_t)blockDim.x, total) - 1);
        __syncthreads();   // the previous round's readers are done
        stage_models(s_md, md + m_lo, min(m_hi - m_lo + 1, kStageModels));
        __syncthreads();
        const int64_t g = g0 + threadIdx.x;
        if (g >= total) continue;
        const int m = chunk_worker(md, M, g);
        const DenseModel& gm = md[m];
        if (kWrite && gm.words > word_cap) continue;
        const int64_t i = g - gm.chunk0;
        const int r0 = (int)(i << log2_k), r1 = (int)min((int64_t)r0 + ((int64_t)1 << log2_k), gm.nz);
        const int32_t* idx = m_idx + (int64_t)m * stride;
        const uint8_t* typ = m_typ + (int64_t)m * stride;
        uint16_t* out = kWrite ? words + (int64_t)m * word_cap + kHeaderWords + kDirWords * gm.n_chunks + ch_off[g]
                               : nullptr;
        const int n_em = kWrite ? ch_len[g] - 2 : 0;
        int n;
        if (m - m_lo < kStageModels) n = encode_seq(s_md[m - m_lo], idx, typ, r0, r1, out, n_em);
        else n = encode_seq(gm, idx, typ, r0, r1, out, n_em);
        if (!kWrite) {
            ch_len[g] = n + 2;
            ch_first[g] = idx[r0];
        }
    }
}

// One block per worker: stream offsets of its chunks (exclusive scan of the
// lengths), the directory, the worker's total words and the capacity check.
__global__ void k_dense_scan(DenseModel* md, const int32_t* __restrict__ ch_len, const int32_t* __restrict__ ch_first,
                             int64_t* ch_off, uint16_t* words, int64_t word_cap, int64_t* n_words, int* status) {
    grid_dep_wait();
    __shared__ int64_t s_tot[33];
    const int m = blockIdx.x;
    DenseModel& mm = md[m];
    const int64_t n = mm.n_chunks, c0 = mm.chunk0;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int64_t run = 0;
    for (int64_t b0 = 0; b0 < n; b0 += blockDim.x) {
        const int64_t i = b0 + threadIdx.x;
        const int64_t v = i < n ? ch_len[c0 + i] : 0;
        int64_t inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t t = __shfl_up_sync(0xFFFFFFFFu, inc, o);
            if (lane >= o) inc += t;
        }
        if (lane == 31) s_tot[warp] = inc;
        __syncthreads();
        int64_t before = 0, all = 0;
        for (int w = 0; w < nw; ++w) {
            before += w < warp ? s_tot[w] : 0;
            all += s_tot[w];
        }
        if (i < n) ch_off[c0 + i] = run + before + inc - v;
        run += all;
        __syncthreads();
    }
    const int64_t total = kHeaderWords + kDirWords * n + run;
    if (threadIdx.x == 0) {
        mm.words = total;
        n_words[m] = total;
        if (total > word_cap) atomicOr(status, kStCapacity);
    }
    if (total <= word_cap) {
        uint16_t* dir = words + (int64_t)m * word_cap + kHeaderWords;
        for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
            put32(dir + kDirWords * i, (uint32_t)ch_first[c0 + i]);
            dir[kDirWords * i + 2] = (uint16_t)ch_len[c0 + i];
        }
    }
}

// ---------------------------------------------------------------------------
// Decoder
// ---------------------------------------------------------------------------
// Worker m's header read back: its counts and chunk size, and its chunk
// count (0 for a malformed header or a code too short for its directory).
struct Header {
    int64_t np, nn, nc, n_chunks;
    int lk;
    bool ok;
};

__device__ Header read_header(const uint16_t* __restrict__ words, const int64_t* __restrict__ n_words, int m,
                              int64_t d, int64_t word_cap) {
    Header h = {0, 0, 0, 0, 4, false};
    const uint16_t* w = words + (int64_t)m * word_cap;
    const int64_t nw = n_words[m];
    bool ok = nw >= kHeaderWords && nw <= word_cap;
    if (ok) {
        h.np = get32(w + 2);
        h.nn = get32(w + 4);
        h.nc = get32(w + 6);
        h.lk = w[8];
        ok = (int64_t)get32(w) == d && h.lk >= 4 && h.lk <= 10 && h.np + h.nn + h.nc <= d;
    }
    if (ok) {
        h.n_chunks = (h.np + h.nn + h.nc + ((int64_t)1 << h.lk) - 1) >> h.lk;
        if (nw < kHeaderWords + kDirWords * h.n_chunks) ok = false;
    }
    if (!ok) {
        h.np = h.nn = h.nc = h.n_chunks = 0;
    }
    h.ok = ok;
    return h;
}

// One block per worker: its header read back and its model rebuilt, and the
// chunks of all workers before it (from their headers; the last block writes
// the total).  A malformed header records kStInvalid and leaves that worker
// with no chunk.
__global__ void k_dense_dsetup(const uint16_t* __restrict__ words, const int64_t* __restrict__ n_words, int M,
                               int64_t d, int64_t word_cap, DenseModel* md, int64_t* total_chunks, int* status) {
    grid_dep_wait();
    __shared__ long long s_red[32];
    const int m = blockIdx.x, tid = threadIdx.x;
    const Header h = read_header(words, n_words, m, d, word_cap);
    DenseModel& mm = md[m];
    build_model_block(d, h.np, h.nn, h.nc, mm);
    long long before = 0;
    for (int j = tid; j < m; j += blockDim.x) before += read_header(words, n_words, j, d, word_cap).n_chunks;
    before = warp_sum(before);
    if ((tid & 31) == 0) s_red[tid >> 5] = before;
    __syncthreads();
    if (tid == 0) {
        long long c0 = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) c0 += s_red[w];
        mm.log2_k = h.lk;
        mm.n_chunks = h.n_chunks;
        mm.chunk0 = c0;
        if (!h.ok) atomicOr(status, kStInvalid);
        if (m == M - 1) *total_chunks = c0 + h.n_chunks;
    }
}

// One block per worker: offsets of the chunk streams from the directory's
// lengths; the streams must fill the code exactly.
__global__ void k_dense_dscan(DenseModel* md, const uint16_t* __restrict__ words, const int64_t* __restrict__ n_words,
                              int64_t word_cap, int64_t* ch_off, int* status) {
    grid_dep_wait();
    __shared__ int64_t s_tot[33];
    const int m = blockIdx.x;
    DenseModel& mm = md[m];
    const int64_t n = mm.n_chunks, c0 = mm.chunk0;
    const uint16_t* dir = words + (int64_t)m * word_cap + kHeaderWords;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int64_t run = 0;
    for (int64_t b0 = 0; b0 < n; b0 += blockDim.x) {
        const int64_t i = b0 + threadIdx.x;
        const int64_t v = i < n ? dir[kDirWords * i + 2] : 0;
        int64_t inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t t = __shfl_up_sync(0xFFFFFFFFu, inc, o);
            if (lane >= o) inc += t;
        }
        if (lane == 31) s_tot[warp] = inc;
        __syncthreads();
        int64_t before = 0, all = 0;
        for (int w = 0; w < nw; ++w) {
            before += w < warp ? s_tot[w] : 0;
            all += s_tot[w];
        }
        if (i < n) ch_off[c0 + i] = run + before + inc - v;
        run += all;
        __syncthreads();
    }
    if (threadIdx.x == 0 && n > 0 && kHeaderWords + kDirWords * n + run != n_words[m]) {
        atomicOr(status, kStInvalid);
        mm.n_chunks = 0;   // (no chunk of this worker is decoded)
    }
}

// One rANS decoding step: the symbol whose [c, c + f) holds x's low 15 bits.
// The stream's next words wait in a register window (four words, refilled
// four at a time from loads issued one window ahead), so a renormalisation
// rarely waits on memory.
struct Dec {
    const uint16_t* w;
    int pos, len;       // next word to load into the window, stream length
    uint64_t win, nxt;  // current and next window, low word first
    int nwin, nnxt;     // words left in each
    uint32_t x;
    bool bad;
    __device__ __forceinline__ void fetch(uint64_t& v, int& n) {
        v = 0;
        n = 0;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (pos + k < len) {
                v |= (uint64_t)w[pos + k] << (16 * k);
                ++n;
            }
        }
        pos += n;
    }
    __device__ __forceinline__ void start() {
        fetch(win, nwin);
        fetch(nxt, nnxt);
    }
    __device__ __forceinline__ void step(uint32_t f, uint32_t c, uint32_t slot) {
        x = f * (x >> kScale) + slot - c;
        if (x < kLow) {
            if (nwin == 0 && nnxt > 0) {
                win = nxt;
                nwin = nnxt;
                fetch(nxt, nnxt);
            }
            if (nwin > 0) {
                x = (x << 16) | (uint32_t)(win & 0xFFFFu);
                win >>= 16;
                --nwin;
            } else {
                bad = true;
            }
        }
    }
    __device__ __forceinline__ bool done() const { return nwin == 0 && nnxt == 0 && pos == len; }
};

// Decodes chunk i of worker m into its dense q~ row; false when the
// stream is malformed.
__device__ __forceinline__ bool decode_chunk(const DenseModel& mm, const uint16_t* base, int64_t i, int64_t off,
                                             int64_t d, int8_t* row) {
    const uint16_t* dir = base + kHeaderWords + kDirWords * i;
    const int64_t K = (int64_t)1 << mm.log2_k;
    const int64_t cnt = min(K, mm.nz - i * K);
    Dec r;
    r.w = base + kHeaderWords + kDirWords * mm.n_chunks + off;
    r.len = dir[2];
    r.bad = r.len < 2;
    r.x = r.bad ? kLow : (((uint32_t)r.w[0] << 16) | r.w[1]);
    r.pos = r.bad ? r.len : 2;
    r.start();
    int64_t idx = get32(dir);
    for (int64_t j = 0; j < cnt && !r.bad; ++j) {
        if (j > 0) {
            // run bit length: the last l with len_c[l] <= slot, searched
            // forward from the table's start for the slot's top 8 bits
            const uint32_t slot = r.x & (kM - 1u);
            int a = mm.len_lut[slot >> 7];
            while (a + 1 < kLens && mm.len_c[a + 1] <= slot) ++a;
            r.step(mm.len[a].f, mm.len[a].c, slot);
            uint32_t v = 1;
            for (int k = a - 1; k >= 0; --k) {
                const uint32_t sl = r.x & (kM - 1u);
                const uint32_t f0 = mm.bit0[k].f;
                const uint32_t bit = sl >= f0 ? 1u : 0u;
                if (bit) r.step(mm.bit1[k].f, mm.bit1[k].c, sl); else r.step(f0, 0u, sl);
                v = 2u * v + bit;
            }
            idx += v;
        }
        const uint32_t sl = r.x & (kM - 1u);
        const int t = sl < mm.val[1].c ? 0 : (sl < mm.val[2].c ? 1 : 2);
        r.step(mm.val[t].f, mm.val[t].c, sl);
        if (idx < 0 || idx >= d) {
            r.bad = true;
            break;
        }
        row[idx] = t == 0 ? (int8_t)1 : (t == 1 ? (int8_t)-1 : (int8_t)2);
    }
    return !(r.bad || r.x != kLow || !r.done());
}

// Decodes every chunk into the dense q~ rows (int8, zeroed beforehand), one
// thread per chunk, with the block's models staged in shared memory.
__global__ void __launch_bounds__(128)
    k_dense_decode(const uint16_t* __restrict__ words, const DenseModel* __restrict__ md, int M, int64_t d,
                   int64_t word_cap, const int64_t* __restrict__ total_chunks, const int64_t* __restrict__ ch_off,
                   int8_t* qt, int* status) {
    grid_dep_wait();
    __shared__ DenseModel s_md[kStageModels];
    const int64_t total = *total_chunks;
    for (int64_t g0 = (int64_t)blockIdx.x * blockDim.x; g0 < total; g0 += (int64_t)gridDim.x * blockDim.x) {
        const int m_lo = chunk_worker(md, M, g0);
        const int m_hi = chunk_worker(md, M, min(g0 + (int64_t)blockDim.x, total) - 1);
        __syncthreads();   // the previous round's readers are done
        stage_models(s_md, md + m_lo, min(m_hi - m_lo + 1, kStageModels));
        __syncthreads();
        const int64_t g = g0 + threadIdx.x;
        if (g >= total) continue;
        const int m = chunk_worker(md, M, g);
        const DenseModel& gm = md[m];
        const int64_t i = g - gm.chunk0;
        if (i >= gm.n_chunks) continue;   // a worker whose directory did not add up
        const uint16_t* base = words + (int64_t)m * word_cap;
        int8_t* row = qt + (int64_t)m * d;
        const bool ok = m - m_lo < kStageModels ? decode_chunk(s_md[m - m_lo], base, i, ch_off[g], d, row)
                                                : decode_chunk(gm, base, i, ch_off[g], d, row);
        if (!ok) atomicOr(status, kStInvalid);
    }
}

}  // namespace

// ---------------------------------------------------------------------------
// Host launchers.  The workspace holds, in order: the per-worker -1 counts,
// the per-worker models, the chunk total, and per chunk its stream length,
// first index and stream offset.
// ---------------------------------------------------------------------------
namespace {
struct DenseWs {
    unsigned long long* neg;
    DenseModel* md;
    int64_t* total;
    int32_t* len;
    int32_t* first;
    int64_t* off;
    int32_t* m_idx;    // encoder: each worker's merged sequence (row stride `stride`)
    uint8_t* m_typ;
};

size_t up256(size_t b) { return (b + 255) & ~(size_t)255; }

DenseWs carve_dense(void* base, int M, int64_t max_chunks, int64_t stride, bool encode, size_t* bytes) {
    DenseWs w;
    char* p = static_cast<char*>(base);
    size_t o = 0;
    auto take = [&](size_t n) {
        char* r = p ? p + o : nullptr;
        o += up256(n);
        return r;
    };
    w.neg = reinterpret_cast<unsigned long long*>(take(sizeof(unsigned long long) * M));
    w.md = reinterpret_cast<DenseModel*>(take(sizeof(DenseModel) * M));
    w.total = reinterpret_cast<int64_t*>(take(sizeof(int64_t)));
    w.len = reinterpret_cast<int32_t*>(take(encode ? sizeof(int32_t) * max_chunks : 0));
    w.first = reinterpret_cast<int32_t*>(take(encode ? sizeof(int32_t) * max_chunks : 0));
    w.off = reinterpret_cast<int64_t*>(take(sizeof(int64_t) * max_chunks));
    w.m_idx = reinterpret_cast<int32_t*>(take(encode ? sizeof(int32_t) * (size_t)M * stride : 0));
    w.m_typ = reinterpret_cast<uint8_t*>(take(encode ? (size_t)M * stride : 0));
    if (bytes) *bytes = o;
    return w;
}

int grid_for(int64_t items, int threads, int per_sm) {
    const int64_t b = (items + threads - 1) / threads;
    return (int)std::max<int64_t>(1, std::min<int64_t>(b, (int64_t)device_sm_count() * per_sm));
}
}  // namespace

size_t dense_workspace_bytes(int M, int64_t max_chunks, int64_t stride, bool encode) {
    size_t b = 0;
    carve_dense(nullptr, M, max_chunks, stride, encode, &b);
    return b;
}

cudaError_t launch_dense_encode(const int32_t* qa, const uint32_t* qb, const int32_t* n_a, const int32_t* n_b, int M,
                                int64_t d, int64_t cap, int log2_k, uint16_t* words, int64_t word_cap,
                                int64_t* n_words, void* ws, int64_t max_chunks, int* status, cudaStream_t st) {
    const int64_t stride = std::min<int64_t>(d, 2 * cap);   // at most this many non-zero symbols per worker
    const DenseWs w = carve_dense(ws, M, max_chunks, stride, true, nullptr);
    cudaError_t e;
    set_launch_error_site("dense code: count reset");
    e = cudaMemsetAsync(w.neg, 0, sizeof(unsigned long long) * M, st);
    if (e != cudaSuccess) return e;
    {
        set_launch_error_site("k_dense_count launch");
        TraceScope ts(kKDenseCount, st);
        const int bx = std::max(1, std::min(grid_for(cap, 1024, 1), std::max(1, device_sm_count() * 4 / M)));
        e = launch_dep(k_dense_count, dim3(bx, M), dim3(1024), 0, st, qb, n_b, cap, w.neg);
        if (e != cudaSuccess) return e;
    }
    {
        set_launch_error_site("k_dense_setup launch");
        TraceScope ts(kKDenseSetup, st);
        e = launch_dep(k_dense_setup, dim3(M), dim3(128), 0, st, n_a, n_b, (const unsigned long long*)w.neg, M, d, cap,
                       log2_k, w.md, words, word_cap, w.total, status);
        if (e != cudaSuccess) return e;
    }
    const size_t smem = kDenseWarps * warp_bytes(1 << log2_k);
    set_launch_error_site("k_dense_merge shared-memory attribute");
    e = cudaFuncSetAttribute(k_dense_merge, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    {
        set_launch_error_site("k_dense_merge launch");
        TraceScope ts(kKDenseMerge, st);
        e = launch_dep(k_dense_merge, dim3(grid_for(max_chunks, kDenseWarps, 16)), dim3(kDenseWarps * 32), smem, st,
                       qa, qb, (const DenseModel*)w.md, M, cap, log2_k, (const int64_t*)w.total, w.m_idx, w.m_typ,
                       stride);
        if (e != cudaSuccess) return e;
    }
    const int gb = grid_for(max_chunks, 128, 16);
    {
        set_launch_error_site("k_dense_encode (count) launch");
        TraceScope ts(kKDenseEncode, st);
        e = launch_dep(k_dense_encode<false>, dim3(gb), dim3(128), 0, st, (const int32_t*)w.m_idx,
                       (const uint8_t*)w.m_typ, stride, (const DenseModel*)w.md, M, log2_k, (const int64_t*)w.total,
                       w.len, w.first, (const int64_t*)w.off, words, word_cap);
        if (e != cudaSuccess) return e;
    }
    {
        set_launch_error_site("k_dense_scan launch");
        TraceScope ts(kKDenseScan, st);
        e = launch_dep(k_dense_scan, dim3(M), dim3(512), 0, st, w.md, (const int32_t*)w.len,
                       (const int32_t*)w.first, w.off, words, word_cap, n_words, status);
        if (e != cudaSuccess) return e;
    }
    set_launch_error_site("k_dense_encode (write) launch");
    TraceScope ts(kKDenseEncode, st);
    return launch_dep(k_dense_encode<true>, dim3(gb), dim3(128), 0, st, (const int32_t*)w.m_idx,
                      (const uint8_t*)w.m_typ, stride, (const DenseModel*)w.md, M, log2_k, (const int64_t*)w.total,
                      w.len, w.first, (const int64_t*)w.off, words, word_cap);
}

cudaError_t launch_dense_decode(const uint16_t* words, const int64_t* n_words, int M, int64_t d, int64_t word_cap,
                                int8_t* qt, void* ws, int64_t max_chunks, int* status, cudaStream_t st) {
    const DenseWs w = carve_dense(ws, M, max_chunks, 0, false, nullptr);
    cudaError_t e;
    set_launch_error_site("dense decode: output reset");
    e = cudaMemsetAsync(qt, 0, (size_t)M * (size_t)d, st);
    if (e != cudaSuccess) return e;
    {
        set_launch_error_site("k_dense_dsetup launch");
        TraceScope ts(kKDenseSetup, st);
        e = launch_dep(k_dense_dsetup, dim3(M), dim3(128), 0, st, words, n_words, M, d, word_cap, w.md, w.total,
                       status);
        if (e != cudaSuccess) return e;
    }
    {
        set_launch_error_site("k_dense_dscan launch");
        TraceScope ts(kKDenseScan, st);
        e = launch_dep(k_dense_dscan, dim3(M), dim3(512), 0, st, w.md, words, n_words, word_cap, w.off, status);
        if (e != cudaSuccess) return e;
    }
    set_launch_error_site("k_dense_decode launch");
    TraceScope ts(kKDenseDecode, st);
    return launch_dep(k_dense_decode, dim3(grid_for(max_chunks, 128, 16)), dim3(128), 0, st, words,
                      (const DenseModel*)w.md, M, d, word_cap, (const int64_t*)w.total, (const int64_t*)w.off, qt,
                      status);
}

}  // namespace gs
