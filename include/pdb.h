/*
 * pdb.h -- C ABI of libpdb: serially-equivalent sparse SGD on one GPU.
 *
 * The method is data-centric synchronization (Parameter Database): each
 * training example's sparse SGD update is a transaction whose read and write
 * set is the example's nonzero features.  Examples that share no feature run
 * concurrently; examples that share one run in data order, so the trained
 * weights equal those of sequential SGD over the data in its given order.
 *
 * Paper anchors (the paper's own section, definition and algorithm labels):
 *   Definition 1   parameter database M(Theta, D): D immutable, Theta mutable
 *   Definition 2   chunks (here: single features)
 *   Definition 3   an iteration reads its chunks, then writes them
 *   Algorithm 1,   the sequential computation every result must equal
 *   Definition 4
 *   Algorithm 2a   BSP: read barrier, reads, compute, write barrier, writes
 *   Algorithm 2b   relaxed: per-chunk Read and Write Constraints (Sec. 4.4)
 *   Theorem 2      RC + WC give the sequential result
 *   Theorem 3      BSP executions are a subset of RC/WC executions
 *   Section 5      read protocol: a per-chunk iteration number gates reads
 *   Section 7      admissible delay: reads and writes within delta iterations
 *
 * Conventions for every call:
 *   - Pointers named as device pointers must be device memory of the current
 *     CUDA device; the caller owns them and keeps them alive until the work
 *     queued on `stream` has finished.
 *   - `stream` is a cudaStream_t passed as void*; NULL is the legacy default
 *     stream.  Every call only enqueues work on `stream` (asynchronous),
 *     except where a comment says it synchronizes.
 *   - Return value: PDB_OK or a negative PDB_E* code for errors found on the
 *     host (arguments, allocation, launch).  Errors found by the kernels
 *     (bad CSR contents, expired waits) are recorded in the conflicts
 *     handle's device status word; read it with pdb_status().  Once a handle
 *     holds an error, later kernels that use it return at once and the
 *     handle must be rebuilt.
 *   - Calls that share a handle must be ordered on one stream (the handles
 *     hold device-side counters that a concurrent call would clobber).
 *   - Limits: n_rows, n_cols and nnz below 2^31 (positions and ids are int32).
 *   - Memory: handles allocate stream-ordered from a memory pool the library
 *     creates for each device on first use.  That pool keeps freed blocks for
 *     reuse (its release threshold is raised) until the process exits; the
 *     device's default pool and every other process-wide CUDA setting are left
 *     as they are.
 *   - Host memory: a pinned, device-mapped slab of small words, one per
 *     process (grown in slabs of 64 slots), holds each conflicts handle's info
 *     words and stages pdb_status' read.  The library's kernels store those
 *     words into it directly: a device-to-host copy of a few bytes would queue
 *     behind the caller's large copies on the copy engine.
 *   - Diagnostics: every call opens an NVTX range named after it (seen by
 *     profilers); with the environment variable PDB_LOG set to anything but
 *     "" or "0" each call (but pdb_sgd_epoch_ready_noalloc) prints one line
 *     of pdb_get_stats on stderr afterwards, which synchronizes the device.
 *     PDB_NEAR (pdb_build_conflicts) and PDB_LEVELS (pdb_schedule_build)
 *     are described where they apply.
 */
#ifndef PDB_H
#define PDB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------- errors */
#define PDB_OK 0
#define PDB_EINVAL (-1)   /* null pointer, negative size, row_ptr not nondecreasing from 0 to nnz, size mismatch */
#define PDB_ERANGE (-2)   /* a feature id outside [0, n_cols) */
#define PDB_EDUP (-3)     /* a feature id repeated inside one example (read/write sets are sets, Def. 3) */
#define PDB_ENOMEM (-4)   /* device allocation failed */
#define PDB_ECUDA (-5)    /* a CUDA runtime call or launch failed */
#define PDB_ETIMEOUT (-6) /* a bounded device-side wait expired (the kernel stopped, the GPU stays usable) */
#define PDB_EFAULT (-7)   /* an internal invariant failed on the device */
#define PDB_ESTATE (-8)   /* wrong handle for this call (e.g. a READY schedule where levels are needed) */
#define PDB_ETOOBIG (-9)  /* beyond a fixed limit: the scratch of pdb_sgd_epoch_ready_noalloc, CHAIN's
                             row length, or a feature occurring 2^29 times or more */

/* ---------------------------------------------------------------- types */

/* The data D of the parameter database M(Theta, D) (Definition 1): n_rows
 * examples in CSR form over n_cols features.  Example t holds the features
 * col[row_ptr[t] .. row_ptr[t+1]) with values val[...] (val == NULL means
 * every value is 1.0, binary features).  Device pointers, caller-owned,
 * never written by the library.  Example order is the data order that the
 * result must reproduce.  Rows may be empty; ids in a row must be distinct
 * (any order). */
typedef struct {
    int64_t n_rows, n_cols, nnz;
    const int64_t *row_ptr; /* [n_rows + 1] */
    const int32_t *col;     /* [nnz] */
    const float *val;       /* [nnz] or NULL */
} pdb_csr;

/* Loss term f_t of example t as a function of its margin m = w . x_t
 * (Eq. 2's data terms; the regularizer g is not supported).
 *   LOGISTIC  f = log(1 + exp(-y m)),  y in {-1, +1}
 *   SQUARED   f = (m - y)^2 / 2
 *   HINGE     f = max(0, 1 - y m), subgradient 0 at y m = 1 */
typedef enum { PDB_LOSS_LOGISTIC = 0, PDB_LOSS_SQUARED = 1, PDB_LOSS_HINGE = 2 } pdb_loss;

/* How pdb_sgd_epoch keeps conflicting examples in data order.
 *   LEVELS  dependency levels: level-synchronous execution, one grid barrier
 *           per level (each level is one BSP step over disjoint examples,
 *           Theorem 3)
 *   READY   per-feature ready counters: an occurrence of feature j with rank
 *           r reads w_j once the iteration number of j equals r and
 *           publishes r + 1 with its write (the read protocol of Section 5
 *           with the iteration number counted per feature); no barrier at
 *           all.  The number lives in the same 64-bit word as the weight,
 *           with an epoch stamp: all epochs run in one pipelined launch,
 *           each feature's next-epoch occurrences starting as soon as its
 *           last occurrence of the epoch has written.
 *   CHAIN   for conflict graphs that are close to one chain (a feature in
 *           most examples): one thread block runs the examples strictly in
 *           data order (Algorithm 1 itself), prefetching ids, values and
 *           weights ahead and forwarding each new weight whose next
 *           occurrence is among the next 16 examples through shared memory,
 *           so a dependency hop costs a few hundred cycles (examples of at
 *           most 256 ids).  Longer examples run with all n_cols weights
 *           resident in shared memory instead, when they fit (about 55,000
 *           features; dense examples of ~1000 features); else PDB_ETOOBIG.
 *   WINDOW  for conflict graphs whose consecutive occurrences of a feature
 *           mostly lie far apart: w stays a plain float array.  A position
 *           whose previous occurrence lies at least `near` positions back
 *           (a distance fixed by the build, >= 2^22) reads w_j once the
 *           completion watermark -- every example before it finished --
 *           has passed that occurrence; a nearer one takes the weight from
 *           its previous occurrence through feature j's 64-bit record,
 *           bits(w_j) | tag << 32, written only by positions whose next
 *           occurrence is near, the tag being the reader's occurrence rank
 *           with an epoch stamp (the read protocol of Section 5 on the near
 *           pairs only).
 *   AUTO    CHAIN when the longest per-feature chain exceeds n_rows / 20 and
 *           CHAIN takes the rows (see above); else WINDOW when at most 1/8
 *           of the positions have a near next occurrence; else READY (waits
 *           on the host for the conflict build to read those numbers). */
typedef enum {
    PDB_SCHED_LEVELS = 0,
    PDB_SCHED_READY = 1,
    PDB_SCHED_CHAIN = 2,
    PDB_SCHED_AUTO = 3,
    PDB_SCHED_WINDOW = 4
} pdb_sched_mode;

/* Gates of pdb_ssp_epoch (Section 7; iterations counted per feature, the
 * occurrence of feature j with rank r being iteration r of j). */
typedef enum {
    PDB_SSP_COUNT = 1,  /* counters: rank r reads once r - delay writes of j are done and writes once
                         * r - delay + 1 occurrences of j have read (the default) */
    PDB_SSP_PREFIX = 2  /* prefixes: rank r reads once every rank <= r - 1 - delay has written and writes
                         * once every rank <= r - delay has read (the Write Protocol's slowest reader) */
} pdb_ssp_gates;

/* Launch and wait options; a zeroed struct (or NULL) selects the defaults. */
typedef struct {
    int32_t blocks_per_sm;     /* persistent grid = blocks_per_sm x #SM (at most the occupancy
                                  maximum); 0 = that maximum, for WINDOW 3 */
    int32_t ticket_chunk;      /* READY: consecutive examples a warp takes per ticket; 0 = 2 */
    double wait_timeout_s;     /* limit of every device-side wait; 0 = 2 seconds; at most 10^6 seconds */
    uint64_t *trace;           /* optional (NULL = off), pdb_sgd_epoch and pdb_ssp_epoch: device array of
                                * n_epochs * n_rows * 2 words; per example (epoch-major) the %globaltimer
                                * value (ns) once all its reads are done, then once its update is computed
                                * and before any of its writes is issued, so a caller can check an
                                * execution against the Read and Write Constraints (Section 4.4) or the
                                * asynchronous ones (Section 7).  Costs two stores per example. */
    int32_t ssp_gates;         /* pdb_ssp_epoch: a pdb_ssp_gates value; 0 = PDB_SSP_COUNT */
} pdb_opts;

/* Sizes and timings; timings are CUDA-event milliseconds of the last call of
 * each kind on the given handles (0 when not run). */
typedef struct {
    int64_t n_rows, n_cols, nnz;
    int64_t n_levels;        /* LEVELS schedule: number of levels L; else -1 */
    int64_t max_level_width; /* LEVELS schedule: largest level; else -1 */
    int64_t max_chain;       /* most occurrences of one feature (longest per-feature chain) */
    double ms_build, ms_schedule, ms_sgd, ms_bsp;
    double ms_sgd_kernels;   /* pdb_sgd_epoch's update kernels alone (no record packing) */
    int64_t sched_mode;      /* mode the schedule runs (AUTO resolved); -1 without a schedule */
} pdb_stats;

typedef struct pdb_conflicts pdb_conflicts; /* opaque, library-owned device arrays */
typedef struct pdb_schedule pdb_schedule;   /* opaque, library-owned device arrays */
typedef struct pdb_bsp_plan pdb_bsp_plan;   /* opaque, library-owned device arrays */

/* ---------------------------------------------------------------- calls */

/* Conflict structure of D (Definitions 2-3; read protocol of Section 5).
 * Validates X on the device (row_ptr, id range, no repeated id in a row),
 * stable-sorts the (feature, position) pairs by feature and links
 * consecutive occurrences of each feature into a chain:
 *   csc_pos[nnz]    positions grouped by feature, data order inside a feature
 *   feat_ptr[F+1]   feature j occupies csc_pos[feat_ptr[j] .. feat_ptr[j+1])
 *   prev[p], next[p] previous / next position holding col[p], -1 if none
 *   rank[p]         number of earlier positions holding col[p]
 * It also marks, per position, whether the previous and the next
 * occurrence lie within a distance `near` (the WINDOW schedule's input; see
 * pdb_schedule_ready) and counts those pairs: near = 2^22 positions, or
 * k * 2^15 rounded up to a power of two for a mean example length k > 128,
 * or the value of the environment variable PDB_NEAR (>= 1) when set at
 * this call.  Any near >= 1 gives the same SGD result; it only decides which
 * positions wait on the watermark.
 * A feature occurring 2^29 times or more is reported as PDB_ETOOBIG.
 * Above 2^22 positions the position-order gate array is built on first use
 * (a READY, CHAIN or LEVELS schedule, or pdb_conflicts_arrays), enqueued on
 * that call's stream; the WINDOW schedule needs only the near pairs' words,
 * which the build writes directly.
 * *out receives a new handle (free with pdb_conflicts_free) even when the
 * device later reports a CSR error through pdb_status.  The handle keeps
 * referring to X's arrays (D is immutable, Definition 1): they must stay
 * valid and unchanged while the handle is in use.  Allocates its arrays
 * stream-ordered on `stream`. */
int pdb_build_conflicts(const pdb_csr *X, pdb_conflicts **out, void *stream);

/* Borrowed device pointers into the handle (valid until it is freed): the
 * per-feature occurrence chains of Section 5's read protocol.  Any output
 * pointer may be NULL.  prev/next/rank are derived from the CSC
 * order (rank = slot - feat_ptr[j], neighbours in the slot order) and are
 * materialized by a kernel enqueued on `stream` the first time one of them
 * is requested; read them after that work has completed. */
int pdb_conflicts_arrays(const pdb_conflicts *c, const int32_t **csc_pos, const int64_t **feat_ptr,
                         const int32_t **prev, const int32_t **next, const int32_t **rank, void *stream);

/* Schedule for pdb_sgd_epoch (each mode keeps the Read and Write
 * Constraints of Section 4.4 per feature, so every mode gives the sequential
 * result, Theorem 2).
 *   LEVELS (Theorem 3): level[t] = 1 + max over features j of t with an
 *     earlier occurrence of level[row of that occurrence], 0 if none
 *     (longest conflict path), computed by dataflow (examples in data order, each
 *     waiting, bounded, for its predecessors' levels) or, with the
 *     environment variable PDB_LEVELS=kahn, by a Kahn-style frontier sweep
 *     (one grid barrier per level); both give the same levels.  order[N]
 *     lists the examples by level, ascending id inside a level; level_ptr[L+1]
 *     delimits the levels.
 *   READY (Section 5, read protocol): one 64-bit record per feature,
 *     bits(w_j) | version_j << 32, filled from w by pdb_sgd_epoch; each
 *     position waits for the version equal to its occurrence rank (the
 *     conflicts' gate array).
 *   CHAIN (Algorithm 1 in data order on one SM): per position, whether an
 *     example among the 16 before it writes its feature last (its weight is
 *     then forwarded on chip) and where the next occurrence sits if within
 *     the 16 examples after; nothing when the
 *     longest example has more than 256 ids and the weights fit in shared
 *     memory (resident); PDB_ETOOBIG when they do not.
 *   WINDOW: per feature a 64-bit hand-off record for near pairs, one
 *     progress word per worker warp, a ticket and the completion watermark;
 *     the positions' near flags are in the gate.
 *   AUTO: CHAIN, WINDOW or READY (see pdb_sched_mode).
 * Allocates stream-ordered on `stream`. */
int pdb_schedule_build(const pdb_conflicts *c, pdb_sched_mode mode, pdb_schedule **out, void *stream);

/* LEVELS schedule arrays (borrowed device pointers, any may be NULL) and the
 * level count (Theorem 3's levels).  SYNCHRONIZES `stream` to read L from the device.
 * PDB_ESTATE for a READY schedule. */
int pdb_schedule_levels(const pdb_schedule *s, const int32_t **level, const int32_t **order,
                        const int64_t **level_ptr, int64_t *n_levels, void *stream);

/* READY and WINDOW schedule arrays (borrowed device pointers, any may be
 * NULL; Section 5's read protocol per feature): gate[nnz], per position bits
 * 0..28 the version it waits for (its occurrence rank), bit 29 set when the next occurrence of its feature lies
 * within the build's `near` distance, bit 30 when the previous one does,
 * bit 31 on the last occurrence of its feature (under WINDOW with more than
 * 2^22 positions: the WINDOW engine's copy, which holds only the words of
 * positions with a near pair and 0 elsewhere); and, READY only,
 * records[n_cols] (weight bits | version << 32, the version being the rank
 * waited for in bits 0..28 and an epoch stamp 1..7 in bits 29..31;
 * meaningful while pdb_sgd_epoch runs; NULL under WINDOW).  PDB_ESTATE for LEVELS and CHAIN
 * schedules. */
int pdb_schedule_ready(const pdb_schedule *s, const uint32_t **gate, const uint64_t **records);

/* n_epochs passes of SGD over X in data order (Algorithm 1 with one
 * iteration per example), run concurrently under the schedule's constraint.
 * w (device, n_cols floats, caller-owned) is read and updated in place; y
 * (device, n_rows floats) are the labels.  For every example t:
 *   m = w . x_t         32 partial sums: element i of the row adds into
 *                       partial i mod 32 with a fused multiply-add, then
 *                       the partials combine pairwise (xor 16, 8, 4, 2, 1)
 *   g = dloss/dm (m, y) fp32; logistic uses exp by Cody-Waite reduction and
 *                       a degree-7 Taylor polynomial
 *   w_j = w_j - (eta*g) * x_tj  for the features of t
 * Each fp32 operation is rounded once, so the result is bitwise the same for
 * every schedule and equals the sequential run (Theorem 2).
 * X and c must be the same data the schedule was built from.  The host
 * waits for c's build to complete if it has not (the kernel variant depends
 * on the longest example, which the build records). */
int pdb_sgd_epoch(const pdb_csr *X, const float *y, const pdb_conflicts *c, const pdb_schedule *s, float *w,
                  pdb_loss loss, float eta, int n_epochs, const pdb_opts *opts, void *stream);

/* SGD with admissible delay (Section 7): like pdb_sgd_epoch under a READY
 * schedule, with the asynchronous Read and Write Constraints per feature
 * (iterations counted per feature: the occurrence of j with rank r is
 * iteration r of j), in the form opts->ssp_gates selects:
 *   PDB_SSP_COUNT   (default) rank r reads w_j once at least r - delay
 *                   writes of j are done, and writes once at least
 *                   r - delay + 1 occurrences of j have read;
 *   PDB_SSP_PREFIX  rank r reads once every rank <= r - 1 - delay of j has
 *                   written, and writes once every rank <= r - delay has
 *                   read (the paper's Write Protocol: a writer waits for
 *                   the slowest reader).  Keeps a done-bitmap per direction
 *                   over the CSC slots: nnz / 4 bytes in all, allocated on
 *                   first use and kept with the schedule.
 * Either way a write applies its step to the current w_j (an atomic fp32
 * add of -(eta*g)*x_j), so every example's update is applied exactly once;
 * w is updated in place.
 *   delay = 0    the sequential result, bitwise equal to pdb_sgd_epoch
 *                (both forms)
 *   delay > 0    the result depends on timing and is not deterministic.  A
 *                read of rank r sees at least r - delay writes of its
 *                feature.  Under PDB_SSP_PREFIX it sees every write of rank
 *                <= r - 1 - delay and none of rank >= r + delay; under
 *                PDB_SSP_COUNT a slow reader holds no writer back, so its
 *                read may also see writes of later occurrences
 *   delay >= the longest chain  no waits at all (Hogwild with atomic updates)
 *   coef         optional device array of n_epochs * n_rows floats (NULL for
 *                none): the step eta*g each example applied, epoch-major,
 *                for auditing a delayed run
 * s must be a READY schedule of c (PDB_ESTATE otherwise); delay < 0 or an
 * unknown opts->ssp_gates is PDB_EINVAL; under PDB_SSP_PREFIX a gate word
 * whose rank lies past its feature's occurrences is PDB_EFAULT (reported
 * through pdb_status).  Every wait is bounded (pdb_opts.wait_timeout_s). */
int pdb_ssp_epoch(const pdb_csr *X, const float *y, const pdb_conflicts *c, const pdb_schedule *s, float *w,
                  pdb_loss loss, float eta, int n_epochs, int64_t delay, float *coef, const pdb_opts *opts,
                  void *stream);

/* BSP comparison (Algorithm 2a with `batch` examples between barriers):
 * per batch [b*B, min((b+1)*B, N)) every example computes c_i = eta *
 * dloss/dm at the weights of the batch start (read barrier), then each
 * feature j takes delta_j = sum over the batch's examples, ascending, of
 * c_i * x_ij and w_j = w_j - delta_j (write barrier).  batch = 1 equals
 * sequential SGD (Theorem 1).  Allocates per-call scratch stream-ordered;
 * sizing it waits (host) for the conflict build of c to finish. */
int pdb_bsp_epoch(const pdb_csr *X, const float *y, const pdb_conflicts *c, float *w, pdb_loss loss, float eta,
                  int64_t batch, int n_epochs, const pdb_opts *opts, void *stream);

/* Algorithm 2a split over data-parallel ranks.  Every rank holds the whole
 * data and a replica of w.  Per batch b (rows [b*B, min((b+1)*B, N))) each
 * rank computes the coefficients c_i = eta * dloss/dm of its slice of the
 * batch's rows at the batch-start weights (the reads), the ranks gather the
 * batch's coefficients in row order (a collective of the caller's choice),
 * and every rank applies delta_j = sum over the batch's examples, ascending,
 * of c_i * x_ij, w_j = w_j - delta_j (the writes).  The arithmetic and its
 * order are pdb_bsp_epoch's, so any split gives that call's result bit for
 * bit.
 *
 * pdb_bsp_plan_build: sorts c's pairs by (batch, feature, example) once for
 *   batch size `batch` (>= 1; above N it is N) into a plan handle (device
 *   arrays, library-owned; the plan borrows c, which must outlive it).
 *   SYNCHRONIZES `stream` (the batch bounds are copied to the host).
 *   PDB_EINVAL for a NULL argument or batch < 1.
 * pdb_bsp_plan_batches: number of batches, or -1 for NULL.
 * pdb_bsp_coef: coef[i - row_begin] = c_i for rows [row_begin, row_end),
 *   which must lie inside one batch (PDB_EINVAL otherwise); w = the batch's
 *   start weights (device, n_cols floats); coef device, caller-owned.
 *   X, y, loss as for pdb_sgd_epoch.  Asynchronous.
 * pdb_bsp_apply: the write half of batch `batch_index` with coef = all of
 *   the batch's coefficients in row order (device, rows of the batch
 *   floats); w updated in place.  Asynchronous.  An inconsistent plan is
 *   PDB_EFAULT in c's status word.
 * pdb_bsp_plan_free: waits for the work enqueued on the plan, frees its arrays. */
int pdb_bsp_plan_build(const pdb_conflicts *c, int64_t batch, pdb_bsp_plan **out, void *stream);
int64_t pdb_bsp_plan_batches(const pdb_bsp_plan *p);
int pdb_bsp_coef(const pdb_bsp_plan *p, const pdb_csr *X, const float *y, const float *w, pdb_loss loss, float eta,
                 int64_t row_begin, int64_t row_end, float *coef, void *stream);
int pdb_bsp_apply(const pdb_bsp_plan *p, float *w, int64_t batch_index, const float *coef, void *stream);
void pdb_bsp_plan_free(pdb_bsp_plan *p);

/* SYNCHRONIZES `stream` and returns the device status of handle c: PDB_OK
 * or the first error a kernel recorded (PDB_EINVAL, PDB_ERANGE, PDB_EDUP,
 * PDB_ETIMEOUT, PDB_EFAULT); PDB_ECUDA if the synchronization itself fails. */
int pdb_status(const pdb_conflicts *c, void *stream);

/* Sizes and timings; waits (host) for the work enqueued on c and s to read
 * the event timers and L, not for the device's other streams.  s may be
 * NULL. */
int pdb_get_stats(const pdb_conflicts *c, const pdb_schedule *s, pdb_stats *out);

/* Release a handle: waits for the work enqueued on this handle by earlier
 * calls (not for the rest of the device, whose other streams keep running),
 * then returns its arrays to the library's memory pool. */
void pdb_conflicts_free(pdb_conflicts *c);
void pdb_schedule_free(pdb_schedule *s);

/* Text of an error code. */
const char *pdb_strerror(int code);

/* Allocation-free variant of pdb_sgd_epoch with a READY schedule
 * (Algorithm 1 under Section 5's read protocol).  The paper has no
 * counterpart of the allocation-free form.  It is for callers that cannot
 * let a library allocate device memory while they train: a server that has
 * handed all device memory to its own pool and must not see it grow or
 * fragment, or a host runtime that accounts for every device allocation
 * itself.  It calls no cudaMalloc, cudaFree or allocating library routine:
 * its scratch (one 64-bit (weight, version) record per feature, a ticket
 * counter and a status word) is one fixed array inside the library of 2^20
 * records, about 8 MiB, that every GPU loading the library holds until the
 * process exits.
 *   X, y, w     as for pdb_sgd_epoch; X->n_cols must be <= 2^20, else
 *               PDB_ETOOBIG and nothing runs.
 *   gate[nnz]   per position, the gate word (occurrence rank of its feature
 *               in bits 0..28, bit 31 on the feature's last occurrence,
 *               bits 29-30 ignored here) -- the array that
 *               pdb_schedule_ready returns for a READY schedule of X (device,
 *               caller-owned here).
 * Same arithmetic and result as pdb_sgd_epoch.  Set-up: the first call on
 * each device (and again after that device's context is reset) looks up
 * the array's device address with cudaGetSymbolAddress.  The call cannot be
 * recorded into a CUDA graph (it synchronizes).  All calls on a device share the array,
 * which keeps the last call's contents (each call clears what must start at
 * zero): calls whose GPU work overlaps race, so order them on one stream.
 * SYNCHRONIZES `stream` (the status word is copied to the host) and returns
 * PDB_OK, a kernel-recorded error (PDB_ETIMEOUT, PDB_EFAULT), or a host
 * error. */
int pdb_sgd_epoch_ready_noalloc(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, pdb_loss loss,
                                float eta, int n_epochs, void *stream);

/* ---------------------------------------------------------------- utilities */

/* cudaMemcpyAsync with the kind inferred from the pointers (for bindings that
 * need to read the borrowed arrays). */
int pdb_memcpy(void *dst, const void *src, size_t bytes, void *stream);

/* Number of CUDA kernels this library has launched in this process so far
 * (every launch site counts once per launch). */
int64_t pdb_launch_count(void);

/* out[i] = the library's device exp of x[i] (device arrays of n floats), the
 * same function the logistic gradient uses.  The paper fixes no exponential;
 * this one is Cody-Waite range reduction (Cody and Waite 1980) with a
 * degree-7 Taylor polynomial, within 2 ulp of exp on [-87, 88.5] and exact
 * at 0, so the oracle can restate it bit for bit.  n < 0, or a NULL array
 * with n > 0, is PDB_EINVAL. */
int pdb_eval_expf(const float *x, float *out, int64_t n, void *stream);

/* out[i] = eta-free loss derivative dloss/dm at margin m[i] and label y[i]
 * (device arrays of n floats), the same function every engine applies
 * (Section 6.3's SGD step, gradient of Eq. 2 without a regulariser):
 * logistic -y / (1 + exp(y m)) with the exp above, squared m - y, hinge
 * (y m < 1 ? -y : 0).  For the logistic loss with y = +1 or -1 and
 * 1 <= 1 + exp(y m) < 2^126 the quotient is formed as a reciprocal, equal
 * bit for bit to the IEEE division.  n < 0, an unknown loss, or a NULL array
 * with n > 0 is PDB_EINVAL. */
int pdb_eval_grad(const float *m, const float *y, float *out, int64_t n, pdb_loss loss, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* PDB_H */
