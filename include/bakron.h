/*
 * bakron.h -- C ABI of the GB300 BaKron solver (libbakron.so).
 *
 * BaKron ("Babai quantization for Kronecker-factored Hessians") rounds an
 * m x n weight matrix W onto a quantisation alphabet by Babai nearest-plane /
 * GPTQ error feedback under the Hessian H = A (x) B, with A (n x n) the
 * input-side and B (m x m) the output-side SPD Kronecker factor (paper,
 * Sec. 3, Alg. 2-5).  The factors enter through their unit-lower forms
 * L^A = Cholesky(A^-1), L^B = Cholesky(B^-1) with columns scaled to a unit
 * diagonal (Alg. 1/2, first two lines), and entry (i, j) is rounded at
 *
 *     X_ij = W_ij + sum_{(p,q) < (i,j)} L^B_ip E_pq L^A_jq,   E = V - X,
 *
 * the order-free definition of the equivalence proof (Appendix, Eq.
 * canonical-antidiagonal).  All anti-diagonals i + j = k are independent, so
 * the solve takes m + n - 1 dependent rounding steps, and the bulk error
 * propagation follows Alg. 5 (recursive halving of the anti-diagonal range),
 * O(mn(m+n)) work in total (Appendix, complexity of BaKron).
 *
 * Conventions for every entry point:
 *  - Matrices are row-major.  Pointers marked "device" are CUDA device memory
 *    owned by the caller; the library never allocates, frees or retains them.
 *    State kept between calls: the per-shape schedule table of
 *    bakron_autotune, the lane streams and events of bakron_solve_batched
 *    (created on first use), the fixed scratch of bakron_solve_noalloc and
 *    the profiling counters; all live until the process exits.
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is
 *    enqueued asynchronously on it unless stated otherwise.
 *  - Arguments are validated on the host before anything is enqueued; an
 *    invalid argument returns BAKRON_ERR_INVALID_ARG and enqueues nothing.
 *  - Errors found on the device (a non-positive Cholesky pivot, a non-finite
 *    value) are recorded in a status word inside the workspace; entry points
 *    that synchronise return it, and bakron_read_status() returns it later.
 *    No kernel traps or aborts.
 *  - Only the lower triangles of A and B are read.
 */
#ifndef BAKRON_H_
#define BAKRON_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  BAKRON_OK = 0,
  BAKRON_ERR_INVALID_ARG = 1,   /* bad pointer, size, bits, group, dtype      */
  BAKRON_ERR_NOT_SPD = 2,       /* damped A or B not positive definite        */
  BAKRON_ERR_CUDA = 3,          /* a CUDA runtime call failed                 */
  BAKRON_ERR_TIMEOUT = 4,       /* a bounded device wait ran out              */
  BAKRON_ERR_WORKSPACE = 5,     /* workspace smaller than required            */
  BAKRON_ERR_NONFINITE = 6      /* NaN/Inf met while rounding                 */
} bakron_status;

typedef enum { BAKRON_F32 = 0, BAKRON_BF16 = 1 } bakron_dtype;

/* Bytes of the opaque factor buffer for an m x n problem (L^A, L^B and the
 * RevCholesky diagonals, padded to the kernels' tile size). */
size_t bakron_factors_bytes(int m, int n);

/* Bytes of scratch a call to bakron_prepare or bakron_solve needs for an
 * m x n problem (the larger of the two; one buffer serves both). */
size_t bakron_workspace_bytes(int m, int n);

/*
 * bakron_prepare -- damp A and B and build their unit-lower factors.
 * Paper: Alg. 2 first two lines; damping as in Sec. 4 and Appendix
 * "Experiments" (H + damp * mean(diag H) * I).  Computed as
 * L = RevCholesky(H_d)^-1 diag(RevCholesky(H_d)), which equals the
 * normalised Cholesky(H_d^-1) without forming the inverse.
 *   A        device, n x n fp32, input-side Gram (lower triangle read)
 *   B        device, m x m fp32, output-side Gram (lower triangle read)
 *   damp     >= 0, relative diagonal damping
 *   factors  device, bakron_factors_bytes(m, n) bytes, written
 *   workspace device, >= bakron_workspace_bytes(m, n) bytes, scratch
 * Synchronises `stream` at the end and returns BAKRON_ERR_NOT_SPD if a pivot
 * of the damped A or B was not positive (factors are then undefined).
 */
int bakron_prepare(const float* A, const float* B, int m, int n, float damp,
                   void* factors, void* workspace, size_t workspace_bytes,
                   void* stream);

/*
 * bakron_set_factors -- fill a factor buffer from given unit-lower factors.
 *   LA  device, n x n fp32 row-major; strictly-lower part read, diagonal = 1
 *   LB  device, m x m fp32 row-major; likewise
 *   rA, rB  device, length n and m, the RevCholesky diagonals (may be NULL;
 *           they are only stored for the caller)
 * Asynchronous.
 */
int bakron_set_factors(const float* LA, const float* LB, const float* rA,
                       const float* rB, int m, int n, void* factors,
                       void* stream);

/*
 * bakron_get_factors -- copy the unit-lower factors and RevCholesky
 * diagonals out of a factor buffer (device destinations; any may be NULL).
 * Asynchronous.
 */
int bakron_get_factors(const void* factors, int m, int n, float* LA,
                       float* LB, float* rA, float* rB, void* stream);

/*
 * bakron_solve -- BaKron rounding of W (paper, Alg. 5; result defined by the
 * equivalence proof's canonical recursion).
 *   W        device, m rows of n values, row stride ldw elements (>= n),
 *            dtype BAKRON_F32 or BAKRON_BF16 (bf16 is widened exactly)
 *   factors  device, from bakron_prepare or bakron_set_factors
 *   bits     1..8: the alphabet is {0, ..., 2^bits - 1}
 *   group_size 0 for one grid per row, else a divisor of n: one grid per
 *            (row, group of group_size columns)
 *   codes    device, m x n uint8, written (row stride n)
 *   scales, zeros  device, m x G fp32 (G = 1 or n / group_size), written:
 *            the grid of each row/group, from the ORIGINAL W: xmin =
 *            min(0, min w), xmax = max(0, max w) ([-1, 1] if both are 0),
 *            s = (xmax - xmin) / (2^bits - 1), z = rint(-xmin / s), all in
 *            fp32; value of code c is s * (c - z)
 *   prerounding device, m x n fp32 (row stride n), or NULL: the value each
 *            entry was rounded at (the paper's in-place workspace)
 *   workspace device, >= bakron_workspace_bytes(m, n) bytes, scratch
 *   sync     nonzero: synchronise `stream` and return the device status;
 *            zero: fully asynchronous (use bakron_read_status afterwards)
 * Codes are c = clamp(rint(x / s) + z, 0, 2^bits - 1), round half to even.
 */
int bakron_solve(const void* W, int wdtype, int m, int n, int64_t ldw,
                 const void* factors, int bits, int group_size,
                 uint8_t* codes, float* scales, float* zeros,
                 float* prerounding, void* workspace, size_t workspace_bytes,
                 int sync, void* stream);

/*
 * bakron_solve_gptq -- the solve with B = I, i.e. GPTQ (paper, Sec. 1: GPTQ
 * is BaKron with an identity output-side factor; Alg. 1 applied to every row
 * under H = A).  The rows are independent, so the recursion splits columns
 * only: one launch rounds up to four 32-column tiles of every row (one warp
 * per 32-row strip, 32 dependent steps per tile) and the errors of each
 * finished column range reach the columns after it as one tensor-core
 * product E L^A^T (3xTF32).  Arguments, outputs and errors as bakron_solve;
 * only the L^A part of `factors` is read (its L^B may be anything, e.g. from
 * bakron_prepare with B = I).  group_size must be 0 or a multiple of 32 (a
 * group covers whole tiles); BAKRON_ERR_INVALID_ARG otherwise.  The result
 * is the textbook GPTQ loop's (Alg. 1) on every row, up to fp32 rounding.
 */
int bakron_solve_gptq(const void* W, int wdtype, int m, int n, int64_t ldw,
                      const void* factors, int bits, int group_size,
                      uint8_t* codes, float* scales, float* zeros,
                      float* prerounding, void* workspace,
                      size_t workspace_bytes, int sync, void* stream);

/*
 * bakron_grid_symmetric -- the quantisation grid of the paper's experiments
 * (Appendix "Experiments"): the symmetric alphabet {-l, ..., +l}, one scale
 * per row (group_size 0) or per (row, group of group_size columns), chosen
 * from max |w| / l by a squared-error search over shrink factors in [1/2, 1]:
 *   candidate k = 0..K (K = shrink_steps):
 *     s_k = fl(amax * fl((2K - k) / (2K l)))   (K = 0: s_0 = fl(amax * fl(1/l)))
 *   error_k = sum over the row/group of (s_k clamp(rint(w / s_k), -l, l) - w)^2
 * and the least error_k wins (the first, i.e. the larger scale, on ties).  An
 * all-zero row/group uses amax = 1.  The paper's runs use l = 3 and shrink
 * the scale by at most 2x; it leaves the search's resolution open, so the
 * number of steps is the caller's (K = 50 gives factors 1.00, 0.99, ..., 0.50).
 *   W        device, as bakron_solve (read only)
 *   levels   l, 1..127 (2l + 1 codes)
 *   shrink_steps K, 0..1024
 *   scales, zeros  device, m x G fp32, written: the chosen s and z = l, so
 *            that the affine form of bakron_solve holds: code c in 0..2l has
 *            value s (c - l)
 * The quotient w / s_k is formed as w * fl(1 / s_k) and the errors are summed
 * in fp32 (per-thread partial sums, then a fixed tree); rows whose two best
 * candidates lie within that rounding may pick either.  Asynchronous on `stream`; returns BAKRON_ERR_INVALID_ARG before
 * any launch for bad arguments.  Pass the result to bakron_solve_with_grid
 * with qmax = 2 l.
 */
int bakron_grid_symmetric(const void* W, int wdtype, int m, int n, int64_t ldw,
                          int levels, int group_size, int shrink_steps,
                          float* scales, float* zeros, void* stream);

/*
 * bakron_solve_with_grid -- bakron_solve with the caller's grid instead of
 * the min-max one: the same rounding (Alg. 5) onto codes 0..qmax, code c of
 * row p / group g standing for s[p, g] (c - z[p, g]).
 *   qmax     1..255 (codes are uint8)
 *   scales, zeros  device, m x G fp32 (G = 1 or n / group_size), read only;
 *            each scale finite and > 0, each zero an integer in [0, qmax]
 *            (not checked: other values give meaningless codes, but every
 *            memory access stays in bounds)
 * Other arguments, outputs, `sync` and errors as bakron_solve.  The solve's
 * schedule comes from the same per-shape table as bakron_solve.
 */
int bakron_solve_with_grid(const void* W, int wdtype, int m, int n, int64_t ldw,
                           const void* factors, int qmax, int group_size,
                           const float* scales, const float* zeros,
                           uint8_t* codes, float* prerounding, void* workspace,
                           size_t workspace_bytes, int sync, void* stream);

/*
 * Kronecker factors of the Hessian (Sec. 4, "Choosing the Factorization";
 * appendix on the Hessian factorisation).  For H = E[a a^T (x) b b^T]:
 *   K-FAC:    A = E[a a^T], B = E[b b^T]
 *   Shampoo (one power-iteration step from identity):
 *             A = E[|b|^2 a a^T], B = E[|a|^2 b b^T]
 * Both are weighted Grams, accumulated by
 *
 * bakron_gram -- G <- beta G + alpha X^T diag(w) X.
 *   X        device, k samples (rows) of d values, row stride ldx elements
 *            (>= d), dtype BAKRON_F32 or BAKRON_BF16: the activations' tokens
 *            x features layout; a matrix sample (d x r) enters as r rows
 *   w        device, k fp32 weights, or NULL for all ones
 *   alpha, beta  scalars (K-FAC over k samples: alpha = 1/k; beta = 1 adds
 *            to a running sum; beta = 0 never reads G)
 *   G        device, d x d fp32, row stride ldg (>= d): every entry written,
 *            (i, j) and (j, i) to the same value
 *   workspace device scratch of at least bakron_gram_workspace_bytes(d, 1,
 *            w != NULL) bytes; the samples are processed in chunks of as many
 *            as fit (bakron_gram_workspace_bytes(d, c, weighted) holds c), so
 *            a larger workspace means fewer, larger launches
 *   sync     nonzero: synchronise `stream` and return the device status
 * On the tensor cores (tcgen05), FP32-accurate.  bf16 samples without
 * weights: kind::f16 MMAs on the bf16 values (products exact in fp32), each
 * 256 samples accumulated afresh in the tensor core and added in fp32.
 * Otherwise kind::tf32 with operands split x = hi + lo and A B^T ~ hi hi^T +
 * hi lo^T + lo hi^T (bf16 rows are exact in tf32, so their lo MMAs are
 * skipped), each 32 samples accumulated afresh.  Only the lower-triangle
 * 128 x 128 blocks are computed.  Returns BAKRON_ERR_INVALID_ARG (bad
 * pointer, k < 1, d outside 1..65536, strides), BAKRON_ERR_WORKSPACE, or the
 * device status (BAKRON_ERR_TIMEOUT if a bounded wait ran out).
 */
size_t bakron_gram_workspace_bytes(int d, int k_chunk, int weighted);
int bakron_gram(const void* X, int xdtype, int k, int d, int64_t ldx,
                const float* w, float alpha, float beta, float* G, int64_t ldg,
                void* workspace, size_t workspace_bytes, int sync, void* stream);

/*
 * bakron_sample_sqnorms -- out[t] = |y_t|^2 = sum_j Y[t, j]^2 for the k rows
 * of Y (device, row stride ldy >= d, fp32 or bf16), in fp32: the one-step
 * Shampoo weight tr(b_t^T b_t) of sample t.  out: device, k fp32.
 * Asynchronous; BAKRON_ERR_INVALID_ARG before any launch for bad arguments.
 */
int bakron_sample_sqnorms(const void* Y, int ydtype, int k, int d, int64_t ldy,
                          float* out, void* stream);

/*
 * bakron_solve_batched -- H independent solves of one shape m x n in one
 * call: the per-head problems of attention layers whose output-side factor
 * is block diagonal (one B per head, a shared input-side A; the local
 * attention Hessians of Sec. 4 and the BoA setting).  Problem h rounds W[h]
 * under factors[h] exactly as bakron_solve would (the same arithmetic and
 * schedule table, the same codes bit for bit).
 *   W, factors, codes, scales, zeros  HOST arrays of H device pointers (the
 *            buffers of problem h; factors[h] may repeat); the device
 *            buffers are those of bakron_solve for one m x n problem
 *   streams  S, 1..32: problems run side by side on S library-owned CUDA
 *            streams, problem h on lane h mod S, each lane in order; the
 *            lanes fork from `stream` and join back into it through events,
 *            so later work on `stream` sees every result.  With S = H >= 2
 *            (one lane per problem) the leaves of all problems share one
 *            launch per tile anti-diagonal and each tensor-core band stage
 *            one launch, on `stream` itself (unless the shape's schedule
 *            uses dataflow leaves or persistent subtrees)
 *   workspace device, >= bakron_batched_workspace_bytes(m, n, min(S, H))
 *            bytes: lane l uses slice l (bakron_workspace_bytes(m, n) rounded
 *            up to 256 bytes, at offset l times that)
 *   sync     nonzero: synchronise and return the first nonzero device status
 *            of any lane; zero: asynchronous (bakron_read_status_batched)
 * The first call on a device creates its lane streams and events (kept until
 * the process exits): make it outside any stream capture; later calls with
 * sync = 0 can be captured into a CUDA graph.  Calls from several host
 * threads are serialised while they enqueue.  Arguments are validated on
 * the host as in bakron_solve (BAKRON_ERR_INVALID_ARG, BAKRON_ERR_WORKSPACE)
 * before anything is enqueued.
 */
size_t bakron_batched_workspace_bytes(int m, int n, int streams);
int bakron_solve_batched(int H, const void* const* W, int wdtype, int m, int n,
                         int64_t ldw, const void* const* factors, int bits,
                         int group_size, uint8_t* const* codes,
                         float* const* scales, float* const* zeros,
                         void* workspace, size_t workspace_bytes, int streams,
                         int sync, void* stream);
/* Synchronise `stream`; return and clear the status words of the first
 * `streams` lane slices of a batched workspace (the first nonzero one). */
int bakron_read_status_batched(void* workspace, int m, int n, int streams,
                               void* stream);

/*
 * bakron_autotune -- choose, for this problem shape, which kernels run each
 * node of the recursion, by timing candidate schedules on the caller's data.
 * No counterpart in the paper: Alg. 5 fixes the recursion (halving of the
 * anti-diagonal range, Sec. 3.5) and its result, not how a node's band
 * product is evaluated; only that is tuned, so every choice rounds W the same
 * way up to fp32 summation order.  Three settings, in tile anti-diagonals
 * (32 x 32 tiles) spanned by a range of the recursion:
 *   leaf_block      ranges spanning at most this many (1 .. 16) run as a
 *                   block of leaves, each leaf applying what the earlier
 *                   anti-diagonals of its block send it (the nodes inside)
 *   tc_min_band     wider nodes spanning at least this many run their two
 *                   band products on the tensor cores (3xTF32); 0: never
 *   fused_max_band  narrower nodes spanning at most this many run both
 *                   products in one CUDA-core launch, wider ones in two
 * Candidates: tc_min_band in {0, 4, 6, 8, 12, 16, 24} x fused_max_band in
 * {2, 4} x leaf_block in {4, 8, 16}; each is solved three times (one warm-up)
 * and timed with CUDA events on `stream`.  The fastest is stored in a
 * process-wide table keyed by the current device and (m, n), which later
 * bakron_solve calls of that shape use; the environment variables
 * BAKRON_TC_MIN_BAND, BAKRON_FUSED_MAX_BAND and BAKRON_LEAF_BLOCK override
 * the table.  Untuned shapes use tc_min_band = 6, fused_max_band = 2,
 * leaf_block = 8.  Arguments as bakron_solve (codes, scales and zeros are
 * overwritten; no pre-rounding output); tc_min_band, fused_max_band,
 * leaf_block (host, may be NULL) receive the choice and best_ms (host, may
 * be NULL) its time.  Synchronous: it synchronises `stream` after every
 * candidate, so it cannot be captured in a CUDA graph.  Returns the first
 * nonzero status of a candidate solve.
 */
int bakron_autotune(const void* W, int wdtype, int m, int n, int64_t ldw,
                    const void* factors, int bits, int group_size,
                    uint8_t* codes, float* scales, float* zeros,
                    void* workspace, size_t workspace_bytes,
                    int* tc_min_band, int* fused_max_band, int* leaf_block,
                    float* best_ms, void* stream);

/* bakron_get_tuning -- the settings a bakron_solve of shape m x n would use
 * now (table entry or default, environment applied).  Host only. */
int bakron_get_tuning(int m, int n, int* tc_min_band, int* fused_max_band,
                      int* leaf_block);

/* bakron_autotune_clear -- forget every tuned shape. */
void bakron_autotune_clear(void);

/*
 * bakron_solve_noalloc -- bakron_solve without a caller workspace, for
 * callers that cannot allocate device memory of their own: for example a
 * plugin that a host framework hands only its input and output buffers
 * (the framework owns every allocation), or a process under a fixed device
 * memory budget that forbids allocating after start-up.  This entry point has
 * no counterpart in the paper; it is the same solve as bakron_solve.
 *
 * Scratch: a fixed array of BAKRON_NOALLOC_SCRATCH_BYTES (64 MiB) inside the
 * library, on every GPU that loads it, held until the process exits.  A
 * problem fits when the solve's scratch, bakron_workspace_bytes(m, n)'s solve
 * part -- 20 * mp * np bytes (mp, np: m and n rounded up to multiples of 128)
 * plus 4 bytes per 32 x 32 tile and 33 KiB of counters and status -- is at
 * most 64 MiB: e.g. 1792 x 1792 or 2048 x 1536; larger problems are rejected
 * with BAKRON_ERR_WORKSPACE before anything is enqueued (sides above 131072 with BAKRON_ERR_INVALID_ARG,
 * as bakron_solve does).  The call allocates nothing: no cudaMalloc/cudaFree,
 * no allocating library routine.
 *
 * The first call in a CUDA context (the current device's context at the
 * call) looks up the array's device address once (cudaGetSymbolAddress) and
 * caches it under that context's id; make that first call before any stream
 * capture on that device.  After a device reset the new context gets a new
 * id, so the address is looked up again.
 * Every call on a device shares the one array and leaves its contents behind;
 * each call clears what must start at zero (the status word) and overwrites
 * the rest before reading it.  Calls whose work overlaps on the GPU (another
 * stream, another host thread, same device) race on the array: serialise
 * them.  Arguments and outputs are those of bakron_solve.  With sync = 1 the
 * call synchronises `stream` and returns the device status; with sync = 0 it
 * returns after enqueueing, and the device status of that solve (NOT_SPD,
 * NONFINITE, TIMEOUT) is read, and cleared, by bakron_read_status_noalloc on
 * the same device before the next noalloc call clears it.
 */
#define BAKRON_NOALLOC_SCRATCH_BYTES ((size_t)64 << 20)
int bakron_solve_noalloc(const void* W, int wdtype, int m, int n, int64_t ldw,
                         const void* factors, int bits, int group_size,
                         uint8_t* codes, float* scales, float* zeros,
                         float* prerounding, int sync, void* stream);

/* bakron_read_status_noalloc -- synchronise `stream`, return and clear the
 * status word of the last bakron_solve_noalloc on the current device (it
 * lives in the fixed scratch array, whose address callers never see).
 * Allocates nothing.  No counterpart in the paper. */
int bakron_read_status_noalloc(void* stream);

/* Synchronise `stream`, return and clear the device status word kept in
 * `workspace` by the last prepare/solve that used it. */
int bakron_read_status(void* workspace, void* stream);

/*
 * Instrumentation for benchmarks (no counterpart in the paper).
 * bakron_profile_enable(1) (event mode) makes every later bakron_solve
 * bracket each of its kernel launches with CUDA events on `stream` and
 * accumulate, per kernel family, the number of launches, their device time
 * and their algorithmic floating-point work.  The events serialise the
 * launches, so these times add up to more than a solve takes.
 * bakron_profile_enable(2) (timeline mode) instead has every kernel of a
 * solve stamp, on the device, when its CTAs start their dependent work and
 * when the last one ends (global nanosecond timer), with no events between
 * the launches.  The launch sequence of the last bakron_solve enqueued (for
 * example while a CUDA graph of it is captured) is recorded; after each run
 * of that sequence (a graph replay), bakron_profile_collect(stream)
 * synchronises `stream`, turns the stamps into a partition of the run's
 * device time -- launch i owns the time from the end of launch i - 1 to its
 * own end -- adds it to the family totals and clears the stamps.  Timeline
 * mode allocates its stamp buffer (512 KiB) at the first enable(2).  It
 * records one solve at a time (a batched solve's heads overwrite each other).
 * Families:
 *   0 grid + workspace init, 1 leaf wavefront (2*32^3 flops per tile),
 *   2 / 3 band product stage 1 (M = L^B E) / stage 2 (X += M L^A^T) on CUDA
 *   cores, 4 output copy, 5 / 6 stage 1 / stage 2 on the tensor cores,
 *   7 both stages of a narrow node fused in one launch on CUDA cores,
 *   8 one persistent launch running a narrow range of the recursion (its
 *   leaves and band products, separated by grid-wide barriers; not stamped).
 *   A band stage counts 2*32^3 flops per 32x32 tile product it must form
 *   (tile pairs inside the band, triangular diagonal blocks counted whole).
 * bakron_profile_read synchronises the device, then returns the totals since
 * the last bakron_profile_enable (launches, milliseconds, flops; `flops` may
 * be NULL); family -1 returns, in timeline mode, the number of collected runs
 * and the sum of their spans (first start to last end).
 * bakron_last_launches returns the number of kernels the last bakron_solve
 * call on this host thread enqueued.
 */
int bakron_profile_enable(int on);
int bakron_profile_collect(void* stream);
/* Timeline mode: the launches of the last collected run, in enqueue order --
 * family, algorithmic flops, and start / end (us from the run's first start;
 * -1 for a launch without stamps).  Fills at most `max` entries of each
 * (host) array and returns the number of launches, or a negative status. */
int bakron_profile_launch_stamps(int max, int* family, double* flops,
                                 double* start_us, double* end_us);
int bakron_profile_read(int family, int* launches, double* ms, double* flops);
int bakron_last_launches(void);

/*
 * Diagnostic (no counterpart in the paper): C = A B^T on the tensor cores
 * with the 3xTF32 split the band products use.  A is M x K, B is N x K, C is
 * M x N, all device fp32 row-major; M and N multiples of 128, K of 32.
 * workspace >= 256 + 8 (M + N) K bytes.  Synchronises `stream` and returns
 * the device status (BAKRON_ERR_TIMEOUT if a bounded wait ran out).
 */
int bakron_diag_gemm_tf32x3(const float* A, const float* B, float* C, int M,
                            int N, int K, void* workspace,
                            size_t workspace_bytes, void* stream);

/*
 * Diagnostic (no counterpart in the paper): the measured rate of the tensor
 * core instruction the band products issue, tcgen05.mma kind::tf32 with a
 * 128 x 128 accumulator and K = 8, from operands resident in shared memory,
 * one CTA per SM, `stages` x 4 back-to-back MMAs each (timed with CUDA events
 * after a warm-up launch).  *tflops receives the whole-device tf32 rate
 * (2 * 128 * 128 * 8 flops per MMA), *cycles_per_mma (may be NULL) one SM's
 * cycles per MMA.  The FP32-effective rate of the 3xTF32 products is a third
 * of *tflops.  workspace >= 256 + 8 * (number of SMs) bytes.  Synchronous.
 */
int bakron_diag_mma_rate(int stages, void* workspace, size_t workspace_bytes,
                         double* tflops, double* cycles_per_mma, void* stream);

/*
 * Diagnostic (no counterpart in the paper): the cycles one step of the leaf's
 * dependent chain takes, alone on the GPU.  Solves the 32 x 32 problem W
 * (device, row stride 32, fp32 or bf16) with `factors` (a factor buffer of a
 * 32 x 32 problem) as one leaf tile (4-bit grid into codes, scales, zeros),
 * and returns in *cycles_per_step the chain warp's clock64 cycles over its
 * 63 in-tile steps divided by 63.  workspace >= bakron_workspace_bytes(32,
 * 32) + 256 bytes.  Synchronous; returns the device status.
 */
int bakron_diag_leaf_chain(const void* W, int wdtype, const void* factors,
                           uint8_t* codes, float* scales, float* zeros,
                           void* workspace, size_t workspace_bytes,
                           double* cycles_per_step, void* stream);

/* Static description of a status code. */
const char* bakron_strerror(int status);

/* bakron_last_cuda_error -- the CUDA runtime error behind the last
 * BAKRON_ERR_CUDA that a call of this library returned on the calling host
 * thread (0 if none).  Where the pointers are non-null, *name receives the
 * error's name (static storage), *where the library source file and *line the
 * line that saw it.  Host-only, never fails; the record is overwritten by the
 * next failure and not cleared by successes. */
int bakron_last_cuda_error(const char** name, const char** where, int* line);

#ifdef __cplusplus
}
#endif

#endif /* BAKRON_H_ */
