/*
 * gs.h -- C ABI of the GB300 gradient-sparsification library (libgs.so).
 *
 * The library computes, on one GPU, the data-parallel hot path of the
 * gradient sparsification of Wangni, Wang, Liu and Zhang (arXiv:1710.09854):
 * for each of M simulated workers with a dense gradient g (length d)
 *   (1) the l1 sums of g (section 3.2, Algorithm 3, step 3),
 *   (2) keep probabilities p_i = min(lambda |g_i|, 1) (Proposition 1) with
 *       lambda from the greedy rescaling of Algorithm 3,
 *   (3) one Bernoulli(p_i) draw per coordinate (section 3),
 *   (4) amplification of kept entries to g_i / p_i (section 3),
 *   (5) compaction of the kept entries to (int32 index, fp32 value) pairs
 *       (the plain coding of section 3.3),
 * and (6) the sum of the M sparse vectors into a dense fp32 vector
 * (Algorithm 1, step 6, as a sum: the caller applies the 1/M).
 *
 * Conventions shared by every entry point:
 *  - Array arguments are DEVICE pointers unless a parameter says "host".
 *    The caller owns all of them; the library never frees caller memory.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call is asynchronous with respect to the host and
 *    ordered on `stream`.
 *  - Argument errors found on the host are returned at once and nothing is
 *    enqueued.  Errors that only the GPU can see (non-finite gradients,
 *    output capacity, malformed sparse input, a bounded wait that ran out)
 *    are recorded in a per-device status word; gs_sync_status() waits for
 *    the stream and returns (and clears) them.
 *  - Scratch memory is taken stream-ordered from a memory pool owned by the
 *    library (cudaMallocAsync / cudaFreeAsync on `stream`).
 *  - The random draw of coordinate i of worker w at step t is word i mod 4
 *    of Philox4x32-10 (Salmon et al., SC'11) with key = (seed lo, seed hi)
 *    and counter = (q lo, q hi, w, t), q = i / 4; u_i = word * 2^-32 and
 *    coordinate i is kept iff u_i < p_i.  Results are therefore a pure
 *    function of (g, kappa, iters, seed, step, worker) and bit-identical
 *    across runs and launch configurations.
 *  - kappa is the density budget (the paper's rho, Algorithm 3): the
 *    expected number of kept coordinates is at most kappa * d.  It must lie
 *    in (0, 1].  iters >= 0 is the maximum number of rescalings of
 *    Algorithm 3 (the paper's experiments use 2, section 5).
 */
#ifndef GS_H
#define GS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    GS_OK = 0,
    GS_ERR_INVALID_ARG = 1, /* bad argument (host) or malformed sparse input (device) */
    GS_ERR_CUDA = 2,        /* a CUDA runtime call failed */
    GS_ERR_CAPACITY = 3,    /* more kept entries than the output capacity */
    GS_ERR_NONFINITE = 4,   /* a gradient contains NaN or Inf */
    GS_ERR_TIMEOUT = 5,     /* a bounded device-side wait ran out */
    GS_ERR_INTERNAL = 6,    /* library invariant violated */
    GS_ERR_ABORTED = 7      /* a bounded wait ran out and a kernel then left with copies into its
                               shared memory still in flight (the memory system stopped answering):
                               every result since the previous status check is suspect */
} gs_status;

typedef enum { GS_DTYPE_F32 = 0, GS_DTYPE_BF16 = 1 } gs_dtype;

/* Per-worker (per-segment for layer-wise calls) record of the greedy solve,
 * written to device memory by the calls that take a `gs_info*`. */
typedef struct {
    double lambda;      /* final lambda of Proposition 1 */
    double sum_p;       /* sum_i p_i at the final lambda (<= kappa d, Algorithm 3) */
    int64_t capped;     /* #{i : p_i = 1} at the final lambda */
    int32_t iters_run;  /* rescalings performed (<= iters) */
    int32_t flags;      /* bit 0: the exact fallback solve was used */
} gs_info;

/* Human-readable name of a status code.  Never NULL. */
const char* gs_status_string(int status);

/* Text of the last CUDA failure seen by this thread inside the library (the
 * call that failed and the CUDA error name), "" if none.  Never NULL. */
const char* gs_last_error(void);

/* Library version as 10000*major + 100*minor + patch. */
int gs_version(void);

/* Wait for `stream`, then return the first device-side error recorded since
 * the last call to gs_sync_status (GS_OK if none) and clear the record. */
gs_status gs_sync_status(void* stream);

/*
 * Keep probabilities of one gradient (Proposition 1 with lambda from
 * Algorithm 3):  p[i] = min(lambda |g[i]|, 1), rounded to fp32.
 *   g     device, d fp32 values (read only)
 *   d     length, 1 <= d < 2^31
 *   p     device, d fp32 values (written)
 */
gs_status gs_probabilities(const float* g, int64_t d, double kappa, int iters, float* p, void* stream);

/* gs_probabilities plus the solve record: `info` is a device pointer to one
 * gs_info (may be NULL). */
gs_status gs_probabilities_ex(const float* g, int64_t d, double kappa, int iters, float* p, gs_info* info,
                              void* stream);

/*
 * Sparsify one worker's gradient (section 3): kept coordinates in
 * ascending index order as idx[0..nnz) / val[0..nnz), val = g_i / p_i.
 *   g      device, d fp32 values
 *   idx    device, capacity d int32 (written)
 *   val    device, capacity d fp32 (written)
 *   nnz    device, one int32 (written)
 * Equals row `worker` of gs_batched_sparsify(..., worker0 = worker, M = 1).
 */
gs_status gs_sparsify(const float* g, int64_t d, double kappa, int iters, uint64_t seed, uint32_t step,
                      uint32_t worker, int32_t* idx, float* val, int32_t* nnz, void* stream);

/*
 * Sparsify M workers' gradients in one call (Algorithm 1, steps 4-5 for
 * every worker).
 *   g      device, M x d row-major; fp32 or bf16 per `dtype` (row m is
 *          worker worker0 + m)
 *   idx    device, M x cap int32: row m holds worker m's kept indices
 *   val    device, M x cap fp32: the matching values g_i / p_i
 *   nnz    device, M int32: kept count of each worker.  If a count exceeds
 *          cap, only the first cap entries are written, nnz holds the true
 *          count and GS_ERR_CAPACITY is recorded.
 *   cap    row capacity, 1 <= cap <= d (cap = d can never overflow)
 *   info   device, M gs_info records, or NULL
 */
gs_status gs_batched_sparsify(const void* g, int dtype, int M, int64_t d, double kappa, int iters, uint64_t seed,
                              uint32_t step, uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
                              gs_info* info, void* stream);

/*
 * Algorithm 1, steps 4-7 in one call: every worker's Q(g^m) as in
 * gs_sparsify_aggregate, their average v = (1/M) sum_m Q(g^m) (step 6: the
 * fp32 sum in worker order, then one correctly rounded fp32 division by M per
 * coordinate), and step 7's optional re-sparsification v <- Q(v) with its own
 * density budget kappa_v and iters_v, drawn from the Philox stream of worker
 * id worker_v (give it an id no worker uses, or the two stages share draws).
 *   v                  device, d fp32: the average (written)
 *   idx_v, val_v, nnz_v  device: Q(v) as ascending (index, value) pairs,
 *                      capacity d, and its count
 *   info               device, M + 1 gs_info records (the workers', then v's),
 *                      or NULL
 * Other arguments as in gs_sparsify_aggregate (1 <= M <= 512).
 */
gs_status gs_sparsify_average_sparsify(const void* g, int dtype, int M, int64_t d, double kappa, int iters,
                                       uint64_t seed, uint32_t step, uint32_t worker0, int32_t* idx, float* val,
                                       int32_t* nnz, int64_t cap, float* v, double kappa_v, int iters_v,
                                       uint32_t worker_v, int32_t* idx_v, float* val_v, int32_t* nnz_v,
                                       gs_info* info, void* stream);

/*
 * gs_batched_sparsify with the hybrid code of section 3.3 (eqs. 9-10) in
 * place of the plain (index, value) lists: the kept coordinates with p_i = 1
 * (the capped set S_k) go to Q_A as (index, value g_i); every other kept
 * coordinate has value sign(g_i) / lambda, so Q_B holds only its code
 * 2 * index + (g_i < 0), and one fp32 1/lambda per worker gives the
 * magnitude.  Both lists are in ascending index order; merged (a Q_B entry
 * becoming +-inv_lam) they are exactly gs_batched_sparsify's idx / val.
 *   qa_idx, qa_val  device, M x cap: row m holds worker m's Q_A
 *   qb_code         device, M x cap uint32: row m holds worker m's Q_B
 *   n_a, n_b        device, M int32: the lengths (a length above cap writes
 *                   only cap entries and records GS_ERR_CAPACITY)
 *   inv_lam         device, M fp32: fl32(1 / lambda) of each worker
 *   cap             row capacity, >= 1 (cap = d can never overflow)
 * Other arguments as in gs_batched_sparsify.  Q_A needs 8 bytes per entry,
 * Q_B 4 (the index limit d < 2^31 leaves room for the sign bit).
 */
gs_status gs_batched_sparsify_hybrid(const void* g, int dtype, int M, int64_t d, double kappa, int iters,
                                     uint64_t seed, uint32_t step, uint32_t worker0, int32_t* qa_idx, float* qa_val,
                                     uint32_t* qb_code, int32_t* n_a, int32_t* n_b, float* inv_lam, int64_t cap,
                                     gs_info* info, void* stream);

/*
 * The dense code of section 3.3 (last paragraph): per worker, the vector
 * q~ in {0, +1, -1, 2}^d -- 0 where a coordinate is dropped, sign(g_i) where
 * it is kept with p_i < 1, 2 where p_i = 1 -- entropy coded under the static
 * model P(s) = d_s / d (d_s coordinates hold symbol s), whose ideal length
 * sum_s d_s log2(d / d_s) is at most 2d bits.  Together with Q_A's values
 * and 1 / lambda it carries Q(g) exactly.  Each non-zero symbol is coded as
 * the run of zeros before it (geometric in p0 = d_0 / d: its bit length, then
 * its bits below the leading one) and its value (P(t) = d_t / (d - d_0)),
 * which costs exactly what the model charges the symbols; the coder is rANS
 * with 15-bit frequencies and 16-bit words, in independent chunks of
 * K = 2^log2_k non-zero symbols so that both directions run in parallel.
 * A worker's code, in 16-bit words (two-word integers low word first):
 *   header     d, d_{+1}, d_{-1}, d_2 (two words each), log2_k (one word)
 *   directory  per chunk: index of its first non-zero (two words), stream
 *              length in words (one word)
 *   streams    per chunk: the rANS final state (high word first), then the
 *              renormalisation words in the order the decoder reads them.
 * Overhead over the model's length: 144 bits per worker, 96 bits at most per
 * chunk (directory and final state; the run of each chunk's first non-zero
 * and the zeros after the last are not coded), plus the rounding of the
 * frequencies.
 *
 * gs_dense_encode
 *   qa_idx, qb_code, n_a, n_b  the hybrid lists of gs_batched_sparsify_hybrid
 *              (device; rows of `cap` entries; lengths n_a, n_b <= cap)
 *   log2_k     4 .. 10
 *   words      device, M x word_cap uint16: row m receives worker m's code
 *   n_words    device, M int64: each code's length in words.  A code longer
 *              than word_cap is not written past its header; its length is
 *              still reported and GS_ERR_CAPACITY recorded.
 * gs_dense_decode
 *   words, n_words, word_cap   codes as gs_dense_encode writes them
 *   qt         device, M x d int8: q~ of each worker (written)
 *   A malformed code (header, directory, or a stream that does not end in the
 *   encoder's initial state) records GS_ERR_INVALID_ARG.
 */
gs_status gs_dense_encode(const int32_t* qa_idx, const uint32_t* qb_code, const int32_t* n_a, const int32_t* n_b,
                          int M, int64_t d, int64_t cap, int log2_k, uint16_t* words, int64_t word_cap,
                          int64_t* n_words, void* stream);
gs_status gs_dense_decode(const uint16_t* words, const int64_t* n_words, int M, int64_t d, int64_t word_cap,
                          int8_t* qt, void* stream);

/*
 * Algorithm 2 (section 3.2): the closed-form solution of problem (4) for a
 * variance budget eps >= 0 instead of a density budget.  lambda is the one
 * for which sum_i g_i^2 / p_i = (1 + eps) sum_i g_i^2 with
 * p_i = min(lambda |g_i|, 1): (7) with the smallest k satisfying (6).  It is
 * found without a sort (a histogram pass over g brackets 1 / lambda, then
 * Newton steps over the values above the bracket's lower end), so each call
 * reads g twice.  eps = 0 keeps every non-zero coordinate.  sum_i g_i^2 is
 * accumulated in fp32 pairs: a |g_i| above ~1.8e19 (g_i^2 overflows fp32)
 * is reported as GS_ERR_NONFINITE, as are NaN / Inf.  In the gs_info records
 * `iters_run` counts the Newton steps and `capped` is k.
 *   p      device, d fp32: p_i rounded to fp32 (gs_probabilities_eps)
 * Other arguments as in gs_probabilities_ex / gs_batched_sparsify.
 */
gs_status gs_probabilities_eps(const float* g, int64_t d, double eps, float* p, gs_info* info, void* stream);
gs_status gs_batched_sparsify_eps(const void* g, int dtype, int M, int64_t d, double eps, uint64_t seed, uint32_t step,
                                  uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap, gs_info* info,
                                  void* stream);

/*
 * The training loop of the convex experiments of section 5.1 (l2-regularised
 * logistic regression, eq. (14), by SGD over M simulated workers).  These are
 * the loop's own kernels around the sparsifier, not part of it:
 *
 * gs_logreg_grad: worker m's minibatch gradient
 *   G[m] = (1/B) sum_j grad_n_j + 2 lam2 w,
 *   grad_n = -b_n a_n sigma(-b_n a_n^T w) / ln 2 (eq. (14) uses log2),
 * over the rows n_j = batch[m * B + j] of X, and gsq[m] = ||G[m]||^2.
 *   X      device, N x d fp32 row-major (rows a_n);  y  device, N fp32 labels in {-1, +1}
 *   w      device, d fp32;  batch  device, M x B int32 row indices
 *   G      device, M x d fp32 (written);  gsq  device, M fp32 (written)
 *   1 <= B <= 64.  An index outside [0, N) is skipped and recorded as
 *   GS_ERR_INVALID_ARG in the status word.
 */
gs_status gs_logreg_grad(const float* X, const float* y, int N, int d, const float* w, const int32_t* batch, int M,
                         int B, float lam2, float* G, float* gsq, void* stream);

/* margins[n] = b_n a_n^T w for all N rows (the objective of eq. (14) is
 * mean(log2(1 + exp(-margins))) + lam2 ||w||^2).  margins: device, N fp32. */
gs_status gs_logreg_margins(const float* X, const float* y, int N, int d, const float* w, float* margins,
                            void* stream);

/* out[m] = sum of val[m * cap + e]^2 over e < min(nnz[m], cap): ||Q(g^m)||^2
 * from the plain lists.  All device pointers. */
gs_status gs_row_sq_norms(const float* val, const int32_t* nnz, int M, int64_t cap, float* out, void* stream);

/* v = sum of the M rows of G (M x d, device), in row order: the dense
 * (unsparsified) aggregate. */
gs_status gs_sum_rows(const float* G, int M, int64_t d, float* v, void* stream);

/* One SGD step of section 5.1: w -= eta_t * scale * v with the step size
 * divided by the variance factor, eta_t = eta0 / ((1 + t / T0) var_t),
 * var_t = sum_m qsq[m] / sum_m gsq[m] (= ||Q(g)||^2 / ||g||^2 summed over
 * workers; pass qsq = gsq for the unsparsified baseline).  log (device, 2
 * floats, or NULL) receives (eta_t, var_t).  w, v, qsq, gsq are device
 * pointers; T0 > 0, t >= 0. */
gs_status gs_sgd_step(float* w, const float* v, int64_t d, float scale, float eta0, float T0, int t, const float* qsq,
                      const float* gsq, int M, float* log, void* stream);

/*
 * Layer-wise sparsification (section 5.2: each layer is sparsified on its
 * own).  Each worker's vector is cut into L segments by the HOST array
 * seg_offsets[0..L] (0 = seg_offsets[0] < ... < seg_offsets[L] = d); every
 * segment gets its own Algorithm 3 with budget kappa * (segment length).
 * Random words follow the worker's flat index, so each worker's output is
 * one ascending list over all its segments.  Outputs as in
 * gs_batched_sparsify; `info` (or NULL) holds M * L records, worker-major.
 */
gs_status gs_segmented_sparsify(const void* g, int dtype, int M, int64_t d, const int64_t* seg_offsets, int L,
                                double kappa, int iters, uint64_t seed, uint32_t step, uint32_t worker0, int32_t* idx,
                                float* val, int32_t* nnz, int64_t cap, gs_info* info, void* stream);

/*
 * gs_segmented_sparsify plus the sum of the M workers' sparse vectors into
 * out (d fp32, overwritten), fused with the compaction exactly as in
 * gs_sparsify_aggregate (the fp32 sum in worker order; entries beyond cap are
 * neither written nor summed).  1 <= M <= 512.
 */
gs_status gs_segmented_sparsify_aggregate(const void* g, int dtype, int M, int64_t d, const int64_t* seg_offsets,
                                          int L, double kappa, int iters, uint64_t seed, uint32_t step,
                                          uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
                                          gs_info* info, float* out, void* stream);

/*
 * Sum M sparse vectors into a dense fp32 vector (Algorithm 1, step 6):
 *   out[i] = sum_{m=0}^{M-1} Q_m[i], added in fp32 in worker order, so the
 *   result is deterministic.  `out` (device, d fp32) is overwritten.
 *   idx, val   HOST arrays of M device pointers; list m holds nnz[m]
 *              strictly ascending indices in [0, d) and their values
 *   nnz        device, M int32
 *   1 <= M <= 512.  An unsorted, duplicate or out-of-range index records
 *   GS_ERR_INVALID_ARG and leaves `out` unspecified.
 */
gs_status gs_sparse_aggregate(const int32_t* const* idx, const float* const* val, const int32_t* nnz, int M, int64_t d,
                              float* out, void* stream);

/*
 * The whole path for M workers in one call (Algorithm 1, steps 4-6):
 * gs_batched_sparsify, then the worker-order fp32 sum of the M sparse vectors
 * into `out` (device, d fp32, overwritten), exactly as gs_sparse_aggregate
 * would compute it.  The sum reuses the sparsify pass's per-chunk output
 * offsets as its tile table, so it makes no extra pass over the codes.
 * Arguments as in gs_batched_sparsify plus `out`; 1 <= M <= 512.
 */
gs_status gs_sparsify_aggregate(const void* g, int dtype, int M, int64_t d, double kappa, int iters, uint64_t seed,
                                uint32_t step, uint32_t worker0, int32_t* idx, float* val, int32_t* nnz, int64_t cap,
                                gs_info* info, float* out, void* stream);

/*
 * gs_sparsify without any allocation.  The paper has no counterpart: this is
 * a library convenience for callers that cannot allocate device memory
 * during a call -- a program that hands (nearly) all device memory to its
 * own allocator at start-up, or a timed loop in which an allocation, which
 * may block or grow the device's footprint, is not acceptable.  Everything
 * else in this library takes scratch from its memory pool.
 *
 * Result and arguments as in gs_sparsify (same idx / val / nnz, bit for
 * bit), plus:
 *   d       1 <= d <= 4194304 (2^22); a larger d returns GS_ERR_INVALID_ARG
 *           at once and gs_last_error() says why
 *   info    device, one gs_info (may be NULL)
 *   status  device, one int32 (required; NULL returns GS_ERR_INVALID_ARG):
 *           receives, in stream order, the gs_status of the device-side
 *           checks of this call (GS_OK, GS_ERR_NONFINITE, GS_ERR_TIMEOUT,
 *           ...).  It is the only place these errors are reported: they are
 *           not recorded for gs_sync_status, whose status word this call
 *           never touches (it lives in memory the library allocates).
 * Scratch is one static device array of about 48 MiB (sized for d = 2^22)
 * and one static status word; every GPU that loads the library may hold
 * them until the process exits.  The first call on a device looks up their
 * addresses (a one-time set-up that may load the library's code onto the
 * device): make that first call before any stream capture.  All calls on a
 * device share the array, and each call leaves its contents behind: calls
 * that may run at the same time (on different streams, or from host threads
 * with no ordering between them) race and return wrong results, so order
 * them, e.g. on one stream.  GS_OPT_* settings apply as for gs_sparsify;
 * with GS_OPT_KERNEL_TIMING on, the library creates CUDA events.
 */
gs_status gs_sparsify_noalloc(const float* g, int64_t d, double kappa, int iters, uint64_t seed, uint32_t step,
                              uint32_t worker, int32_t* idx, float* val, int32_t* nnz, gs_info* info, int32_t* status,
                              void* stream);

/*
 * The whole path for M workers with HOST buffers: copies g_host (M x d,
 * `dtype`) to the device, runs gs_sparsify_aggregate,
 * and copies the dense sum back to out_host (d fp32) and the kept counts to
 * nnz_host (M int32).  The copy is split into up to 8 groups of workers on two
 * library-owned copy streams, each group sparsified on `stream` as soon as it
 * has landed while the next ones copy; the sum continues across the groups in
 * worker order, so every output equals gs_sparsify_aggregate's bit for bit.
 * The read-back is split in two halves, one per copy stream, and `stream`
 * waits for both.  Calls on one device are serialised on the host (they
 * share the ordering events).  g_dev / idx / val / nnz / out are caller-owned device
 * buffers of the sizes gs_batched_sparsify / gs_sparse_aggregate require
 * (idx, val: M x cap).  Host buffers should be pinned for full copy speed.
 * Returns after enqueueing; the host buffers are valid once `stream` has
 * been synchronised.
 */
gs_status gs_pipeline_host(const void* g_host, int dtype, int M, int64_t d, double kappa, int iters, uint64_t seed,
                           uint32_t step, uint32_t worker0, void* g_dev, int32_t* idx, float* val, int32_t* nnz,
                           int64_t cap, float* out, float* out_host, int32_t* nnz_host, void* stream);

/*
 * The random words the sampler draws (section 3, Z_i ~ Bernoulli(p_i)):
 * out[k] = the Philox4x32-10 word of coordinate i0 + k of worker `worker` at
 * `step` (see the conventions above), for k in [0, n).  Coordinate i is kept
 * iff out * 2^-32 < p_i.  `out` is device memory for n uint32; i0 >= 0.
 */
gs_status gs_random_words(uint64_t seed, uint32_t step, uint32_t worker, int64_t i0, int64_t n, uint32_t* out,
                          void* stream);

/* Library options for tests and diagnostics.
 *   GS_OPT_FORCE_EXACT_SOLVE  1: skip the sampled bound and use the exact
 *                              fallback solve for every worker (slow).
 *   GS_OPT_SAMPLE_SIZE        sampled coordinates per segment for the bound
 *                              on lambda: a multiple of 8 in 256 .. 32768,
 *                              or 0 (the default): 8192 when the call's
 *                              longest segment has at most 2^25
 *                              coordinates, 16384 when it is longer.
 *   GS_OPT_KERNEL_TIMING      1: time every kernel launch (gs_kernel_times);
 *                              2: time the streaming pass only (k_small on
 *                              the cluster path).  The events
 *                              sit between launches, so a timed kernel does
 *                              not overlap its neighbours' launch (mode 2
 *                              leaves the rest of the chain overlapped).
 *   GS_OPT_STREAM_PATH        streaming pass over g: 0 automatic (the TMA
 *                              kernel whenever the layout allows it), 1 the
 *                              generic-load kernel, 2 the TMA kernel where
 *                              eligible.
 *   GS_OPT_SMALL_PATH         rows of d <= 2^21 coordinates: 0 automatic
 *                              (one thread-block cluster per worker when
 *                              also M d <= 2^24, else the chunked kernels),
 *                              1 always the chunked kernels, 2 always the
 *                              cluster path.  Calls with a forced exact
 *                              solve, probabilities, the hybrid code,
 *                              Algorithm 2 or layer-wise segments always
 *                              take the chunked kernels.  Each path is
 *                              deterministic; the two agree with the oracle
 *                              to the stated tolerances, not bit for bit
 *                              (their sums of |g| round in different orders).
 * Options are process-wide; returns GS_ERR_INVALID_ARG for an unknown
 * option or value. */
typedef enum {
    GS_OPT_FORCE_EXACT_SOLVE = 1,
    GS_OPT_SAMPLE_SIZE = 2,
    GS_OPT_KERNEL_TIMING = 3,
    GS_OPT_STREAM_PATH = 4,
    GS_OPT_SMALL_PATH = 5
} gs_option;
gs_status gs_set_option(int option, int64_t value);

/*
 * Self-test of the device-side timeouts (no counterpart in the paper).  Every
 * spin wait in the library's kernels is bounded: on expiry the kernel records
 * GS_ERR_TIMEOUT in the status word and returns.  This launches one warp that
 * waits, with a short limit, on something that never completes -- kind 0: an
 * mbarrier phase nothing arrives at (the primitive the streaming pass waits
 * with), kind 1: a device flag nothing sets -- so the next gs_sync_status()
 * returns GS_ERR_TIMEOUT and the context stays usable.  The call itself
 * returns GS_OK (GS_ERR_INVALID_ARG for another kind).
 */
gs_status gs_selftest_timeout(int kind, void* stream);

/* Tracing.  The library counts every kernel it launches; with
 * GS_OPT_KERNEL_TIMING = 1 it also brackets each launch with CUDA events
 * recorded on the launching stream.  gs_kernel_times() waits for the
 * recorded events, writes for each kernel k < n the accumulated device time
 * ms[k] and launch count launches[k] since the previous read (either array
 * may be NULL), and resets both.  Kernel k is named by gs_kernel_name(k);
 * gs_kernel_count() kernels exist. */
int gs_kernel_count(void);
const char* gs_kernel_name(int k);
gs_status gs_kernel_times(double* ms, int64_t* launches, int n);

#ifdef __cplusplus
}
#endif

#endif /* GS_H */
