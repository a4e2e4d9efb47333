/*
 * dbw.h - C ABI of the GB300 (sm_103a) hot path of Dynamic Backup Workers.
 *
 * Method: C. Xu, G. Neglia, N. Sebastianelli, "Dynamic Backup Workers for
 * Parallel Machine Learning" (arXiv 2004.14696).  One synchronous
 * parameter-server (PS) iteration with n workers simulated on one GPU:
 *
 *   dbw_choose_b          Eqs. (13)-(19): b_t = n - k_t from the estimator state
 *   dbw_worker_grads      Eq. (2): every worker's minibatch gradient -> G [n, ld]
 *   dbw_select_fastest    Eq. (4): arrival order of the n gradients, the k kept
 *   dbw_aggregate_update  Eqs. (3)-(4): masked mean + SGD step, fused with the
 *                         partial sums of Eq. (10), ||g_t||^2 and ||g_j||^2
 *   dbw_grad_stats        Eqs. (10)-(12) and Sect. 3.2: finishes the statistics
 *                         and records them (and the order statistics) in the state
 *
 * Push-and-wait clock and the time estimator of Eq. (17) (Sect. 2, 3.2):
 *   dbw_psw_arrivals / dbw_psw_record / dbw_psw_estimate, dbw_choose_b_times
 *
 * A second form of the iteration skips the [n, d] matrix:
 *   dbw_received_grads_update  Eqs. (2)-(4) and the partial sums of Eqs. (10)-(11)
 *                         for the received workers only (replaces dbw_worker_grads +
 *                         dbw_aggregate_update after dbw_select_fastest)
 *
 * Conventions shared by every call:
 *  - Every pointer argument is a DEVICE pointer owned by the caller unless its
 *    comment says "host".  The library never allocates in these calls; scratch
 *    ("workspace", "partials") is caller memory sized by the *_bytes queries.
 *  - Every compute call is asynchronous on ``stream`` (a cudaStream_t passed as
 *    void*, NULL = legacy default stream) and returns an int status:
 *      DBW_OK (0), DBW_EINVAL (bad argument, detected on the host before any
 *      launch), DBW_EALIGN (a pointer or leading dimension violates the stated
 *      alignment), DBW_ECUDA (a CUDA launch error), DBW_EUNSUPPORTED (device
 *      is not sm_103).  dbw_last_error_string() describes the last failure of
 *      the calling thread.  Nothing is launched when a call returns an error.
 *  - Errors that can only be seen on the device (a device-resident b out of
 *    range, a sample index out of range) never fault: they are clamped or
 *    poisoned as documented per call and raise a bit in dbw_state.flags or
 *    produce NaN in the outputs.
 *  - Floating point: gradients, parameters and G are fp32 (GEMM operands
 *    optionally bf16 with fp32 accumulation); estimator quantities are fp64.
 */
#ifndef DBW_H
#define DBW_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DBW_OK 0
#define DBW_EINVAL (-1)
#define DBW_EALIGN (-2)
#define DBW_ECUDA (-3)
#define DBW_EUNSUPPORTED (-4)

#define DBW_PREC_FP32 0 /* fp32 GEMM operands, fp32 accumulation */
#define DBW_PREC_BF16 1 /* bf16 GEMM operands (RNE from fp32), fp32 accumulation */

#define DBW_NMAX 1024 /* maximum number of workers n */
#define DBW_DMAX 64   /* maximum window D of Eqs. (13)-(15) */
#define DBW_LMAX 8    /* maximum number of layers */

/* dbw_choose_b flags */
#define DBW_CHOOSE_BLIND 1 /* B-DBW (Sect. 4): the gain of k is k itself */

/* dbw_state.flags bits (sticky, OR-ed over iterations) */
#define DBW_FLAG_K1 (1 << 0)        /* an iteration kept k = 1: Eq. (10) undefined, not recorded */
#define DBW_FLAG_L_SKIPPED (1 << 1) /* an Eq. (12) value had denominator <= 0 or was not finite */
#define DBW_FLAG_EMPTY_MASK (1 << 2) /* dbw_grad_stats saw no received worker: nothing recorded */
#define DBW_FLAG_BAD_STATE (1 << 3)  /* state->n disagrees with the call's n (or is out of range) */

/* indices into the stats_out vector of dbw_grad_stats (DBW_STATS_LEN doubles) */
#define DBW_STAT_K 0       /* k_t, number of received gradients */
#define DBW_STAT_SS 1      /* sum_l sum_{j<=k} ([g_j - g_t]_l)^2 (double sum of Eq. (10)) */
#define DBW_STAT_GBAR_SQ 2 /* ||g_t||^2 */
#define DBW_STAT_V 3       /* V^+ of Eq. (10) (NaN if k = 1) */
#define DBW_STAT_N 4       /* ||grad F(w_t)||^2 ^+ of Eq. (11) (NaN if k = 1) */
#define DBW_STAT_F 5       /* F^_t, mean minibatch loss of the received workers (Sect. 3.1) */
#define DBW_STAT_L 6       /* L^+_t of Eq. (12) (NaN if not available / not recorded) */
#define DBW_STAT_FLAGS 7   /* DBW_FLAG_* bits raised by this iteration */
#define DBW_STAT_VCLOCK 8  /* virtual clock after this iteration: sum of T_(k_t) */
#define DBW_STATS_LEN 9

/*
 * Estimator state carried by the PS from iteration to iteration (device memory,
 * plain old data: save/restore by copying sizeof(dbw_state) bytes).
 *
 * Rings hold the most recently recorded "+" estimates of Eqs. (10), (11), (12);
 * cnt* counts all values ever recorded, the newest sits at index (cnt-1) % DMAX.
 * S[k-1] is the running sum of the k-th arrival time, c the number of observed
 * time vectors, so that T^_k = S[k-1] / c (Eq. (17) under push-and-interrupt,
 * where every k has c samples and the per-k means are already monotone).
 */
typedef struct dbw_state {
    int32_t n;        /* workers */
    int32_t D;        /* window of Eqs. (13)-(15), 1..DBW_DMAX */
    int32_t t;        /* completed iterations */
    int32_t k_last;   /* k_{t-1} */
    int32_t c;        /* time vectors observed */
    int32_t cntV, cntN, cntL;
    int32_t flags;    /* sticky DBW_FLAG_* */
    int32_t has_last; /* V_last / N_last hold iteration t-1's recorded estimates */
    int32_t k_next;   /* k_t written by the last dbw_choose_b */
    int32_t reserved;
    double F_last;    /* F^_{t-1} */
    double F_prev;    /* F^_{t-2} */
    double N_last;    /* ||grad F||^2 ^+ of iteration t-1 */
    double V_last;    /* V^+ of iteration t-1 */
    double vclock;    /* virtual clock: sum over iterations of the k_t-th arrival time */
    double ringV[DBW_DMAX];
    double ringN[DBW_DMAX];
    double ringL[DBW_DMAX];
    double S[DBW_NMAX];
} dbw_state;

/* Text of the calling thread's last error ("" if none).  Host; never fails. */
const char* dbw_last_error_string(void);

/* ABI version (incremented on any signature or layout change). */
int dbw_abi_version(void);

/* ----------------------------------------------------------------------- model
 * A fully connected ReLU network (Sect. 4 trains neural networks with the
 * cross-entropy loss): widths[0] inputs, widths[1..L-1] hidden ReLU layers,
 * widths[L] classes, L = num_layers in [1, DBW_LMAX].  Parameters are one flat
 * fp32 vector w [d] in layer order, each layer W_l [out, in] row-major then
 * b_l [out]; G rows use the same order.  widths is a HOST array.
 */

/* d for these widths, or -1 if an argument is invalid. */
int64_t dbw_param_count(int num_layers, const int32_t* widths);

/* Workspace bytes dbw_worker_grads needs for (widths, n, B, prec); 0 if invalid. */
size_t dbw_worker_grads_workspace_bytes(int num_layers, const int32_t* widths, int n, int B, int prec);

/*
 * Eq. (2): g_{i,t} = (1/B) sum_{x in B_i} grad f(x, w_t) for every worker i.
 *
 *  w       [d] fp32 parameters w_t (16-byte aligned).
 *  pool    [S, widths[0]] fp32 dataset features, row-major (16-byte aligned).
 *  labels  [S] int32 class of each pool row.
 *  idx     [n*B] int32 pool rows of the minibatches; worker i owns
 *          idx[i*B .. i*B+B-1].  An index outside [0, S) or a label outside
 *          [0, classes) makes that worker's loss and gradient NaN.
 *  G       [n, ld] fp32 output, row i = g_{i,t}; ld >= d, ld % 4 == 0, 16-byte
 *          aligned.  Columns d..ld-1 are not written.
 *  loss    [n] fp32 output: each worker's minibatch mean loss (Sect. 3.1, F^_t).
 *  ws      workspace of ws_bytes >= dbw_worker_grads_workspace_bytes(...),
 *          256-byte aligned; contents are scratch, except that its first 4
 *          bytes hold a status word once the call's device work is done: 0 on
 *          success, bit 0 set if a tensor-core pipeline wait timed out (it is
 *          bounded, never a hang), in which case G and loss are undefined.
 *  Path: with prec = DBW_PREC_BF16 and B a multiple of 32 the GEMMs run on
 *  the tcgen05 tensor cores in bf16.  With prec = DBW_PREC_FP32 the large
 *  forward and per-worker weight-gradient GEMMs run on the tcgen05 tensor
 *  cores in three tf32 passes (fp32 accuracy: each operand split into two
 *  tf32 parts), small-output and short-inner-dimension GEMMs on dedicated
 *  kernels, the rest on fp32 FFMA (SIMT) tiles; bf16 with B % 32 != 0 runs
 *  on the SIMT tiles too.
 *  prec    DBW_PREC_FP32 or DBW_PREC_BF16.
 */
int dbw_worker_grads(int num_layers, const int32_t* widths, int prec,
                     const float* w, int64_t d,
                     const float* pool, int64_t S, const int32_t* labels,
                     const int32_t* idx, int n, int B,
                     float* G, int64_t ld, float* loss,
                     void* ws, size_t ws_bytes, void* stream);

/*
 * Where dbw_worker_grads leaves the input activations of layer ``layer``
 * (1 <= layer < num_layers: the hidden activations A = ReLU(Z) of the layer
 * below) inside ``ws``: *offset bytes from ws, rows of *ld elements of
 * *elem_bytes bytes (4 = fp32, 2 = bf16), one row per sample, M = n*B rows.
 * Valid once a call's device work is done, until ws is used again.  A hidden
 * unit's ReLU derivative is 1[A > 0], so this is also where a caller reads
 * which units were active.  Host only; DBW_EINVAL for an invalid argument.
 */
int dbw_worker_grads_activations(int num_layers, const int32_t* widths, int n, int B, int prec, int layer,
                                 size_t* offset, int64_t* ld, int* elem_bytes);

/*
 * Opt-in timing of the per-worker weight-gradient launches (the GEMM epilogue
 * that writes G, the largest HBM stream of an iteration).  While enabled, every
 * such launch inside dbw_worker_grads is bracketed by CUDA events recorded on
 * the call's stream.  dbw_profile_dw(enable) turns it on or off and forgets
 * earlier records; dbw_profile_dw_read waits for the recorded events and returns
 * the summed launch durations (ms), the number of launches and their summed
 * algorithmic bytes (G written once in fp32 plus both bf16 operands read once),
 * then forgets them.  Host only; not for use during stream capture.
 */
int dbw_profile_dw(int enable);
int dbw_profile_dw_read(double* total_ms, int64_t* launches, double* total_bytes);

/*
 * Opt-in timing of the persistent tensor-core GEMMs: the forward GEMMs of every
 * layer and the input-gradient GEMMs inside dbw_worker_grads (bf16 models), and
 * in dbw_received_grads_update also the mean-gradient GEMM of every layer.  Each
 * such launch is bracketed by CUDA events on the call's stream while enabled.
 * dbw_profile_gemm(enable) turns it on or off and forgets earlier records;
 * dbw_profile_gemm_read waits for the recorded events and returns the summed
 * launch durations (ms) and the number of launches, then forgets them.  The
 * caller knows the flops: in the received form M (or K) is k*B with k read on
 * the device.  Host only; not for use during stream capture.
 */
int dbw_profile_gemm(int enable);
int dbw_profile_gemm_read(double* total_ms, int64_t* launches);

/*
 * Test hook of the bounded waits (the paper has no counterpart; for tests of the
 * failure path).  Every wait of the tensor-core kernels on a pipeline barrier is
 * bounded (2 s); when one runs out the kernel sets bit 0 of the status word,
 * stops, waits (bounded) for its own copies still in flight, releases its tensor
 * memory and returns, so that the context stays usable.  This call arms the next
 * per-worker weight-gradient launch of dbw_worker_grads (one launch, then it
 * disarms itself): its waits are bounded by wait_ms, and its first CTA does not
 * issue the TMA load of pipeline stage ``stage`` (0 = its first), so that the
 * MMA's wait for that stage runs out, as a lost copy would make it.  That call's
 * G and loss are then undefined and its status word has bit 0 set.  stage < 0
 * disarms.  Host only; DBW_EINVAL unless 0 < wait_ms <= 2000.
 */
int dbw_test_arm_wait_timeout(int stage, double wait_ms);

/*
 * Eq. (4): the PS waits for the first k = n - b gradients.
 * Arrival order is (times[i], i) ascending (ties go to the lower worker index).
 *
 *  times    [n] fp64 round-trip times of this iteration (finite, not NaN).
 *  b        device int32 scalar, the number of backup workers; values outside
 *           [0, n-1] are clamped into it.
 *  order    [n] int32 out: order[r] = worker with arrival rank r.
 *  mask     [n] uint8 out: 1 for the k received workers, else 0.
 *  tsorted  [n] fp64 out: order statistics, tsorted[r] = times[order[r]];
 *           tsorted[k-1] is the iteration's duration for every candidate k.
 *  k_out    device int32 scalar out (nullable): the k actually used.
 *  n in [1, DBW_NMAX].
 */
int dbw_select_fastest(const double* times, int n, const int32_t* b,
                       int32_t* order, uint8_t* mask, double* tsorted,
                       int32_t* k_out, void* stream);

/*
 * Layout of the partials buffer (caller-owned scratch written by
 * dbw_aggregate_update and read by dbw_grad_stats; public so that a caller can
 * also assemble the sums for dbw_grad_stats itself):
 *   int64_t header[4] = {DBW_PARTIALS_MAGIC, blocks, n, flags}
 *           flags: DBW_ALL_ROW_NORMS if every row's norm is in vals, else 0
 *   double  sums[n + 2]              reduced totals, written by dbw_grad_stats
 *   double  vals[(n + 2) * blocks]   per-block pieces, vals[q * blocks + j]:
 *           q < n: piece of ||g_q||^2 (0 for rows not received, unless the
 *           header carries DBW_ALL_ROW_NORMS),
 *           q = n: piece of the deviation sum of Eq. (10), q = n + 1: piece of ||g_t||^2.
 * dbw_grad_stats reduces each quantity in a fixed order (256 strided fp64
 * partial sums, then a pairwise tree), so equal buffers give equal results.
 * A header that does not carry the magic and this call's n yields NaN sums.
 */
#define DBW_PARTIALS_MAGIC 0x44425750415254LL

/* Bytes of the partials buffer dbw_aggregate_update needs on the current device. */
size_t dbw_aggregate_partials_bytes(int n, int64_t d);

/*
 * Eqs. (3)-(4) fused with the statistics of Sect. 3.1, one pass over G:
 *   g_t = (1/k) sum_{j: mask[j]} G[j, :]       (k = number of set mask bytes)
 *   w   = w - lr * g_t                          (in place)
 * and, into ``partials``, the per-block pieces of sum_j ||g_j||^2 (received
 * rows), sum_l sum_j (G[j,l] - g_t[l])^2 and ||g_t||^2, which dbw_grad_stats
 * reduces.  Column sums use a per-column shift (the first received row) so that
 * the deviation sum does not cancel; cross-column sums are fp64.
 *
 *  G        [n, ld] fp32, ld % 4 == 0, 16-byte aligned; only received rows read
 *           (every row with DBW_ALL_ROW_NORMS).
 *  mask     [n] uint8 from dbw_select_fastest (at least one byte set; with none
 *           set, w is left as it is and every piece is 0).
 *  w        [d] fp32, updated in place (16-byte aligned).
 *  gbar     [d] fp32 out (nullable, 16-byte aligned): g_t.
 *  flags    0, or DBW_ALL_ROW_NORMS: also read the n - k rows the mask leaves
 *           out, for their ||g_j||^2 only ((n - k) d * 4 more bytes).  g_t, w and
 *           the sums of Eq. (10) still come from the received rows alone (Eq. (10)
 *           sums over the k received gradients); dbw_grad_stats then reports
 *           every row's norm in row_sqnorm.  Other bits: DBW_EINVAL.
 *  partials scratch of partials_bytes >= dbw_aggregate_partials_bytes(n, d),
 *           256-byte aligned; consumed by the next dbw_grad_stats.
 */
#define DBW_ALL_ROW_NORMS 1
int dbw_aggregate_update(const float* G, int64_t ld, int n, int64_t d,
                         const uint8_t* mask, float lr, float* w, float* gbar, int flags,
                         double* partials, size_t partials_bytes, void* stream);

/*
 * dbw_aggregate_update_noalloc: the same fused aggregation as
 * dbw_aggregate_update, for callers that cannot provide scratch memory.  The
 * paper has no counterpart to this call; it exists for integration.
 *
 * Some callers may not allocate device memory at all: a plugin inside a host
 * application that owns the whole GPU memory budget and hands out only the
 * tensors to work on, or a latency-critical loop in which cudaMalloc (which can
 * synchronise the device) is not acceptable.  This call needs no scratch from
 * them and allocates nothing: its per-block partial sums go to one built-in
 * device array of DBW_NOALLOC_SCRATCH_BYTES that every GPU loading the library
 * holds until the process exits.  That is enough for n <= 1024 on a 152-SM GB300;
 * if (n, d) would need more on the current device the call returns DBW_EINVAL
 * (use dbw_aggregate_update with caller memory instead).
 *
 * The first call on each device looks up the array's device address (the
 * runtime's cudaGetSymbolAddress, with that device current) and caches it; make
 * that first call before any stream capture begins.  All calls on a device
 * share the array: calls whose GPU work overlaps (unordered streams) race and
 * corrupt each other's sums.  Each call clears the array's header on its stream
 * before the aggregation, so a call whose aggregation did not run yields NaN
 * sums rather than an earlier call's; nothing else in it needs to start at zero.
 *
 *  G, ld, n, d, mask, lr, w, gbar, flags   as for dbw_aggregate_update.
 *  sums_out  [n + 2] fp64 device out: sums_out[j] = ||g_j||^2 for received rows
 *            (0 otherwise; every row with DBW_ALL_ROW_NORMS), sums_out[n] = the
 *            deviation sum of Eq. (10), sums_out[n + 1] = ||g_t||^2 -- the totals
 *            dbw_grad_stats would form.
 */
#define DBW_NOALLOC_SCRATCH_BYTES ((size_t)4 << 20)
int dbw_aggregate_update_noalloc(const float* G, int64_t ld, int n, int64_t d, const uint8_t* mask, float lr,
                                 float* w, float* gbar, int flags, double* sums_out, void* stream);

/* Workspace bytes dbw_received_grads_update needs for (widths, n, B, prec); 0 if
 * the shape is invalid or the call does not support it. */
size_t dbw_received_grads_workspace_bytes(int num_layers, const int32_t* widths, int n, int B, int prec);

/* Bytes of the partials buffer dbw_received_grads_update writes for n workers
 * (the layout above with blocks = 1). */
size_t dbw_received_partials_bytes(int n);

/*
 * One PS iteration for the k received workers without the [n, d] gradient
 * matrix: the same w_{t+1} and statistics as dbw_worker_grads followed by
 * dbw_aggregate_update on the rows mask selects, computed as
 *   Eq. (2) for the received workers only: their minibatches are stacked
 *     (slot s = the s-th received worker in increasing index order) and the
 *     forward / backward GEMMs run over those k B rows (under push-and-interrupt,
 *     Sect. 3, the other workers' gradients are never used);
 *   Eqs. (3)-(4): g_t(W_l) = (1/k) dZ_l^T A_{l-1} over the k B stacked rows, one
 *     GEMM with K = k B whose epilogue applies w -= lr g_t; the bias part is
 *     (1/k) times the column sums of dZ_l over the k B rows;
 *   ||g_j||^2 of every received worker from two B x B Gram matrices per layer,
 *     ||dZ_j^T A_j||^2 + ||1^T dZ_j||^2 = <dZ_j dZ_j^T, A_j A_j^T + 1 1^T>
 *     (never forming g_j);
 *   the deviation sum of Eq. (10) by sum_j ||g_j - g_t||^2 = sum_j ||g_j||^2
 *     - k ||g_t||^2 in fp64, and ||g_t||^2, into ``partials``, which the next
 *     dbw_grad_stats reduces exactly as after dbw_aggregate_update.
 * The tensor cores carry the weight-gradient work (K = k B instead of B), and the
 * n d fp32 writes and k d reads of G disappear.  Rounding differs from the
 * two-call form: the mean is an fp32 tensor-core sum over k B rows, the norms come
 * from fp32 Gram entries, and the deviation sum is a difference, whose relative
 * error grows as sum_j ||g_j||^2 / SS.
 *
 *  num_layers, widths, pool, S, labels, idx, n, B   as for dbw_worker_grads.
 *  prec    DBW_PREC_BF16 only, with B % 32 == 0 and (128 % B == 0 or B % 128 == 0);
 *          anything else returns DBW_EUNSUPPORTED.
 *  w       [d] fp32 parameters, updated in place to w_{t+1} (16-byte aligned).
 *  mask    [n] uint8 from dbw_select_fastest; k = number of set bytes, counted on
 *          the device.  With k = 0 nothing is updated and the sums are NaN.
 *  lr      the step eta of Eq. (4).
 *  gbar    [d] fp32 out (nullable, 16-byte aligned): g_t.
 *  loss    [n] fp32 out: minibatch mean loss of each received worker; NaN for
 *          the workers mask leaves out (their loss is never computed).
 *  partials  [partials_bytes >= dbw_received_partials_bytes(n)], 256-byte aligned.
 *  ws      workspace of ws_bytes >= dbw_received_grads_workspace_bytes(...),
 *          256-byte aligned; its first 4 bytes hold the status word of
 *          dbw_worker_grads (bit 0: a bounded tensor-core wait timed out; the
 *          outputs are then undefined).  The activations of layer ``layer`` are
 *          where dbw_worker_grads_activations(..., DBW_PREC_BF16, ...) says, with
 *          slot s at rows s B .. s B + B - 1 (rows of slots >= k are scratch).
 */
int dbw_received_grads_update(int num_layers, const int32_t* widths, int prec,
                              float* w, int64_t d,
                              const float* pool, int64_t S, const int32_t* labels,
                              const int32_t* idx, int n, int B,
                              const uint8_t* mask, float lr, float* gbar, float* loss,
                              double* partials, size_t partials_bytes,
                              void* ws, size_t ws_bytes, void* stream);

/* Initialise a device dbw_state for n workers and window D (k_0 = n). */
int dbw_state_init(dbw_state* state, int n, int D, void* stream);

/*
 * End-of-iteration statistics (Sect. 3.1) and time bookkeeping (Sect. 3.2):
 *   V^+ = SS / (k-1)                         Eq. (10)
 *   ||grad F||^2^+ = max(||g_t||^2 - V^+/k, 0) Eq. (11)
 *   F^_t = mean of loss[j] over received j    (summed in increasing j)
 *   L^+_t from Eq. (12) with iteration t-1's estimates and F^_{t-1} - F^_t
 * recorded into the state's rings (k = 1 and invalid Eq. (12) values are not
 * recorded), S[r] += tsorted[r] for all r, c += 1, vclock += tsorted[k-1].
 *
 *  partials    the buffer the preceding dbw_aggregate_update (or
 *              dbw_received_grads_update) of this iteration wrote.
 *  mask, loss  [n] this iteration's selection and per-worker losses.
 *  tsorted     [n] from dbw_select_fastest.
 *  lr          the learning rate eta used by the update.
 *  stats_out   [DBW_STATS_LEN] fp64 out (nullable), see DBW_STAT_*.
 *  row_sqnorm  [n] fp64 out (nullable): ||g_j||^2 for received rows, NaN for the
 *              others -- unless the aggregation ran with DBW_ALL_ROW_NORMS, then
 *              ||g_j||^2 of every row.
 */
int dbw_grad_stats(const double* partials, int n, const uint8_t* mask,
                   const float* loss, const double* tsorted, double lr,
                   dbw_state* state, double* stats_out, double* row_sqnorm,
                   void* stream);

/*
 * Eqs. (16), (18), (19): choose k_t for the iteration about to start and write
 * b_t = n - k_t to ``b_out`` (device int32 scalar) and to state->k_next.
 *   G^_k  = (eta - q) N^ - q V^ / k,  q = L^ eta^2 / 2, with N^, V^, L^ the
 *           window means of Eqs. (13)-(15) over the last min(D, recorded) values;
 *   T^_k  = S[k-1] / c;
 *   k_t   = argmax_{k: G^_k > 0} G^_k / T^_k (ties -> larger k), k_t = n if no
 *           G^_k > 0 or any window is still empty (k_0 = k_1 = n);
 *   Eq. (19): if t >= 2, F^_{t-1} > beta F^_{t-2} and k_{t-1} < n, then
 *           k_t = max(k_t, k_{t-1} + 1).
 * All fp64 operations are performed one at a time in this order (no fused
 * multiply-add), so equal states give bit-identical b_t.
 *
 *  flags      0 or DBW_CHOOSE_BLIND (gain of k := k, Sect. 4's B-DBW).
 *  ratio_out  [n] fp64 out (nullable): G^_k / T^_k for k = 1..n (NaN while a
 *             window is empty).
 */
int dbw_choose_b(dbw_state* state, double lr, double beta, int flags,
                 int32_t* b_out, double* ratio_out, void* stream);

/* ------------------------------------------------------------------------
 * Push-and-wait (PsW, Sect. 2): after an update the PS pushes the new vector; a
 * busy worker first completes its current computation, then takes the most
 * recent vector.  The k_{t-1} workers received last time are idle when
 * iteration t starts, the others are still busy for a residual time r_j.
 * Sect. 3.2: t_{h,i,t} = time, from the start of iteration t, at which the i-th
 * gradient of w_t arrives given k_{t-1} = h; late workers still report, so
 * every worker that computes on w_t yields a sample (when it arrives).
 * Eq. (17): x_{h,k} = least squares fit to the samples of cell (h, k), increasing
 * in k, decreasing in h, increasing along the diagonal; T^_k = x*_{k,k}.
 *
 * Readings (the paper leaves these open):
 *  - worker j's round trip time on w_t is omega_j of iteration t (one
 *    computation per worker per iteration); it computes on w_t iff r_j < T_t,
 *    where T_t is the k_t-th arrival; its gradient then arrives at r_j + omega_j.
 *  - Eq. (17) does not fix cells without samples.  The rows whose diagonal cell
 *    has samples are fitted on their observed cells, weighted by sample counts.
 *    A row's observed ranks are a prefix, so chains over observed cells generate
 *    the order among them.  Every other diagonal cell is the pooled mean of its
 *    column, made nondecreasing over such cells and clipped to the bounds the
 *    order places on it.  No such row yet: T^ is NaN.
 *  - the fit is Dykstra's alternating projections with weighted
 *    pool-adjacent-violators on each chain, in fp32 (sample counts and sums are
 *    exact; fp64 would cost ~14x in the sequential chains), warm-started from the
 *    previous estimate's dual variables, stopped when a sweep moves no cell by
 *    more than tol x the largest cell mean.  The solution is constant on blocks of
 *    cells, each at the count-weighted mean of its samples: one more sweep records
 *    which cells the projections pool, and every block's value is then its mean
 *    in fp64 from the exact cell sums (blocks that still break the order are
 *    merged, in at most 32 rounds; if that does not settle, the fp32 values stand
 *    and DBW_PSW_UNPOLISHED is raised).  The pooled column means and their PAVA
 *    are fp64 too.
 *
 * The state is one opaque device buffer of dbw_psw_bytes(n) bytes that starts
 * with this header (the offsets locate its arrays, for inspection):
 */
typedef struct {
    int32_t n;          /* workers */
    int32_t h;          /* k_{t-1} (n before the first iteration) */
    int32_t sweeps;     /* Dykstra sweeps of the last dbw_psw_estimate (the recording sweep not counted) */
    int32_t flags;      /* DBW_PSW_* bits, sticky */
    double vclock;      /* tau_t, the push-and-wait virtual clock */
    double unit;        /* value of one unit of the int64 cell sums (2^-32) */
    int64_t iterations; /* iterations recorded */
    int64_t off_r;      /* double  r[n]        residual busy time of each worker */
    int64_t off_pend;   /* int32   pend[2n]    (h, i) of worker j's sample still on its way, h = 0: none */
    int64_t off_pendv;  /* double  pendv[n]    its value */
    int64_t off_sum;    /* int64   sum[n*n]    cell (h, i) at (h-1)*n + (i-1), in units */
    int64_t off_cnt;    /* int32   cnt[n*n]    samples of each cell */
    int64_t off_x;      /* float   x[n*n]      fitted cells of the group rows (fp32 fit) */
    int64_t reserved[6];
} dbw_psw_header;

#define DBW_PSW_NOT_CONVERGED 1 /* the last estimate stopped at max_sweeps */
#define DBW_PSW_RANGE 2         /* a sample outside [0, 2^31) was clamped in the cell sums */
#define DBW_PSW_UNPOLISHED 4    /* the exact block means did not settle: T^ is the fp32 fit */

/* Bytes of the push-and-wait state for n workers (grows as n^2: 6.0 MB at n = 256, 76 MB at n = 1024). */
size_t dbw_psw_bytes(int n);

/* All workers idle, no sample, tau = 0, h = n.  psw: 256-byte aligned device buffer. */
int dbw_psw_init(void* psw, int n, void* stream);

/*
 * arrivals[j] = r_j + omega[j]: when worker j's gradient of w_t reaches the PS,
 * counted from the start of iteration t.  Pass ``arrivals`` to
 * dbw_select_fastest as the times: its first k_t are the received workers.
 *  omega  [n] fp64 this iteration's round trip times (device).
 */
int dbw_psw_arrivals(const void* psw, int n, const double* omega, double* arrivals, void* stream);

/*
 * End of iteration t: with T_t = tsorted[k-1], records every sample that has
 * reached the PS (the arrivals up to T_t, and earlier late samples whose worker
 * became free), keeps the later ones pending, advances the residuals, the clock
 * (tau += T_t) and h = k_t.
 *  order, tsorted, k   from the dbw_select_fastest call on dbw_psw_arrivals' output.
 */
int dbw_psw_record(void* psw, int n, const int32_t* order, const double* tsorted, const int32_t* k,
                   void* stream);

/*
 * Eq. (17): T_hat[k-1] = T^_k for k = 1..n (NaN before any sample).
 *  tol         stop when a Dykstra sweep moves no cell by more than tol x the
 *              largest cell mean; > 0, values below 1e-6 (the fp32 fit's
 *              resolution) act as 1e-6.  The returned values are the exact block
 *              means once the sweeps have found the blocks, so they need not be
 *              tight: measured, tol from 1e-6 to 1e-3 gives the same T^ (within
 *              1e-10 of the fp64 oracle) in 2.5x fewer sweeps at 1e-3.  A partition
 *              the sweeps have not settled would be off by up to tol; 1e-4 is the
 *              pipeline's choice.
 *  max_sweeps  cap (>= 1); reaching it raises DBW_PSW_NOT_CONVERGED.
 */
int dbw_psw_estimate(void* psw, int n, double tol, int max_sweeps, double* T_hat, void* stream);

/*
 * dbw_choose_b with given time estimates: T^_k = T_hat[k-1] in Eqs. (18)-(19)
 * instead of the push-and-interrupt S[k-1] / c (e.g. dbw_psw_estimate's output).
 * NaN in T_hat[0] means "no estimate yet": k_t = n.
 */
int dbw_choose_b_times(dbw_state* state, const double* T_hat, double lr, double beta, int flags, int32_t* b_out,
                       double* ratio_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DBW_H */
