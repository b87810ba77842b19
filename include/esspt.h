/* esspt: a stale-synchronous parameter table on one GPU (sm_103a).
 *
 * One process, one GPU.  P simulated workers share a table of n_rows rows of
 * K fp32 values.  Time advances in clocks (Sec. 2.2): during clock c every
 * worker p reads the table at its read version v_p(c) and adds updates; the
 * Clock() step then makes version c = version c-1 + the sum of every
 * worker's updates of clock c (additive updates, Sec. 2.1; updates coalesced
 * per clock, Sec. 4 "Communication Protocol").  The consistency model picks
 * v_p(c) inside the SSP bound (Sec. 3 "SSP Bounded-Staleness"; Sec. 4 READ
 * guarantee):   max(0, c-1-s) <= v_p(c) <= c-1,   s = 0 being BSP.
 *
 * Versions live in a ring of s+2 table slots in HBM: s+1 readable versions
 * plus the version being written.  Version v sits in slot v mod (s+2).
 *
 * Conventions for every entry point:
 *  - Device pointers are caller-owned (e.g. torch tensors); the library never
 *    allocates device memory and never frees caller memory.  The caller
 *    allocates the workspace whose size the *_workspace_bytes queries return.
 *  - Pointers marked "device or host" may be either (CUDA unified addressing).
 *  - Work is enqueued on the stream given in esspt_config.stream and is
 *    asynchronous unless the entry point says it synchronises.
 *  - Every call returns an esspt_status; errors never abort or trap; the text
 *    of the last error is available from esspt_last_error().
 *  - A context is not thread-safe; use one host thread per context.
 *
 * Row ids are global: for matrix factorisation (Sec. 3.1) rows 0..N-1 hold
 * the user factors L_i and rows N..N+M-1 the item factors R_j (one row per
 * item, the transpose of the paper's column R_{*j}).
 */
#ifndef ESSPT_H
#define ESSPT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ESSPT_OK = 0,
  ESSPT_EINVAL = 1, /* bad argument (null pointer, size, index, version outside the live window) */
  ESSPT_ESTATE = 2, /* call made in the wrong state (e.g. before esspt_table_init) */
  ESSPT_ENOSPC = 3, /* workspace smaller than the size query returned */
  ESSPT_ESTALE = 4, /* a read version broke the staleness bound (schedule rejected) */
  ESSPT_ECUDA = 5,  /* a CUDA runtime call failed; see esspt_last_error() */
} esspt_status;

typedef enum {
  /* SSP with lazy pull (Sec. 2.2; SSPTable of Sec. 4): a worker refreshes its
   * cached table only when it would otherwise break the bound, so its
   * staleness (c-1) - v_p(c) cycles through 0..s.  With `phased` set each
   * worker starts at a seeded phase in [0, s]. */
  ESSPT_SSP_LAZY = 0,
  /* ESSP with eager push (Sec. 2.2, Sec. 4): the server pushes version c-1
   * as soon as every worker has clocked; the push reaches worker p after a
   * seeded delay d ~ Geometric(essp_p) (failures before the first success),
   * clamped to [0, min(essp_max_delay, s)]; v_p(c) = max(v_p(c-1), c-1-d). */
  ESSPT_ESSP_EAGER = 1,
  /* The caller supplies every v_p(c) with esspt_set_schedule(). */
  ESSPT_EXTERNAL = 2,
  /* VAP, the value-bounded model (Sec. 2.1): a worker that reads version v
   * at clock c has the updates X[c-1] - X[v] in transit.  Every worker reads
   * the stalest v in [max(0, c-1-s), c-1] whose in-transit max-norm
   * |X[c-1] - X[v]|_inf (over the whole table, fp32) is at most
   * vap_v0 / sqrt(c), the shrinking bound v_t = v0 / sqrt(t) of the
   * SGD-under-VAP theorem (Sec. 3).  Version c-1 always qualifies; a NaN
   * norm never does.  Each clock reads the s+1 candidate versions once more
   * to compute the norms (the cost the paper names for VAP). */
  ESSPT_VAP = 3,
  /* SSP with a row-granular cache (Sec. 4 "Ensuring Consistency
   * Guarantees": each cached row carries its own clock c_param, and the
   * SSPTable client asks the server for a row only when its copy is too
   * stale).  Worker p holds row r at its own version V[p][r], none before
   * the first read.  At clock c a read of row r is served by the cached copy
   * while V[p][r] >= c-1-s; otherwise (or if r is not cached) the row is
   * first fetched at version c-1.  All reads of a row in one clock see the
   * same version.  For esspt_mf_sgd_clock the rows a worker reads are the
   * user and item rows of its entries in the clock's minibatch.  The cache
   * never evicts: the workspace holds P * n_rows int32 versions.  The ring
   * must hold fewer than 2^31 float4 ((s+2) * n_rows * K/4).
   * v_p(c) as reported by esspt_read_schedule is c-1. */
  ESSPT_SSP_ROW = 4,
} esspt_model;

typedef struct {
  int64_t n_rows;         /* rows of the table, > 0 */
  int32_t row_width;      /* K: values per row, a multiple of 4, 4..512 */
  int32_t num_workers;    /* P, 1..65536 */
  int32_t staleness;      /* s >= 0 */
  int32_t model;          /* esspt_model */
  int32_t phased;         /* ESSPT_SSP_LAZY: 1 = seeded per-worker phase */
  int32_t essp_max_delay; /* ESSPT_ESSP_EAGER: delay clamp (>= 0) */
  double essp_p;          /* ESSPT_ESSP_EAGER: success probability in (0, 1] */
  uint64_t seed;          /* seed of the schedule's counter generator (SplitMix64) */
  void* stream;           /* cudaStream_t; NULL = legacy default stream */
  double vap_v0;          /* ESSPT_VAP: initial value bound v0 >= 0 */
} esspt_config;

typedef struct esspt_ctx esspt_ctx;

/* Bytes of device workspace a table with this configuration needs: the
 * (s+2)-slot version ring plus the schedule state.  0 on invalid config. */
size_t esspt_workspace_bytes(const esspt_config* cfg);

/* Create a context over caller-allocated device workspace `d_workspace`
 * (256-byte aligned, `bytes` >= esspt_workspace_bytes(cfg)).  The workspace
 * must stay allocated until esspt_destroy().  *out receives the context.
 * ESSPT_EINVAL on a bad config, ESSPT_ENOSPC on a short workspace. */
esspt_status esspt_create(const esspt_config* cfg, void* d_workspace, size_t bytes, esspt_ctx** out);

/* Release the host-side context (not the caller's workspace).  Synchronises
 * the stream first.  NULL is accepted. */
esspt_status esspt_destroy(esspt_ctx* ctx);

/* Set version 0 from n_rows*K fp32 values (device or host, row-major) and
 * start clock 1: computes the read versions v_p(1) = 0.  May be called again
 * to restart from a new version 0. */
esspt_status esspt_table_init(esspt_ctx* ctx, const float* rows);

/* GET (Sec. 4 "PS Interface"): copy rows `d_row_ids[0..n)` (device int32,
 * each in [0, n_rows)) of worker `worker`'s read version v_p(c) into
 * `d_out` (device, n*K fp32, row-major).  If `h_version_out` is non-NULL the
 * call synchronises and stores v_p(c) there.  Out-of-range row ids are
 * skipped on the device and reported as ESSPT_EINVAL by esspt_poll().
 * ESSPT_SSP_ROW: each row is read at the worker's cached version of that
 * row, refreshed first as the model says, and `h_version_out` receives the
 * oldest version read (c-1 if no row was read). */
esspt_status esspt_get(esspt_ctx* ctx, int32_t worker, const int32_t* d_row_ids, int64_t n,
                       float* d_out, int32_t* h_version_out);

/* INC (Sec. 4 "PS Interface"): add `d_deltas` (device, n*K fp32) to rows
 * `d_row_ids[0..n)` of the version being written in clock c.  Updates are
 * additive and commutative (Sec. 2.1, Sec. 4), so repeated rows accumulate;
 * fp32 atomic accumulation makes their order, and so the last bits,
 * unspecified.  Out-of-range row ids are skipped and reported by esspt_poll(). */
esspt_status esspt_inc(esspt_ctx* ctx, int32_t worker, const int32_t* d_row_ids, const float* d_deltas,
                       int64_t n);

/* CLOCK (Sec. 4): every worker ticks.  Version c becomes final (version c-1
 * plus all INCs of clock c), the clock advances to c+1 and the read versions
 * v_p(c+1) are computed on the device under the configured model.  A read
 * version outside the bound is latched on the device and returned as
 * ESSPT_ESTALE by esspt_poll(). */
esspt_status esspt_clock(esspt_ctx* ctx);

/* ESSPT_EXTERNAL only: set the read versions v_p(c) of the current clock
 * from `h_v` (host, P int32).  Checked on the host against the bound:
 * ESSPT_ESTALE (and nothing changes) if any v_p(c) is outside
 * [max(0, c-1-s), c-1].  Must be called before the clock's first GET. */
esspt_status esspt_set_schedule(esspt_ctx* ctx, const int32_t* h_v);

/* Synchronise the stream and report, then clear, any error latched on the
 * device (ESSPT_ESTALE: a read version broke the bound; ESSPT_EINVAL: a GET
 * or INC row id was out of range). */
esspt_status esspt_poll(esspt_ctx* ctx);

/* Current clock c (the clock in progress; versions 0..c-1 are final) and,
 * if h_v is non-NULL, the read versions v_p(c) (host, P int32).  Synchronises. */
esspt_status esspt_read_schedule(esspt_ctx* ctx, int32_t* h_v, int32_t* h_clock);

/* Copy table version `version` (n_rows*K fp32) to `out` (device or host).
 * `version` must be final and still in the ring: c-1-s <= version <= c-1,
 * version >= 0.  Synchronises when `out` is host memory. */
esspt_status esspt_read_table(esspt_ctx* ctx, int32_t version, float* out);

/* Text of the last error on this context ("" if none).  Valid until the next
 * call on the context.  NULL ctx gives the last esspt_create() error. */
const char* esspt_last_error(const esspt_ctx* ctx);

/* ---- Matrix factorisation by SGD on the table (Sec. 3.1, Sec. 5) ---------- */

/* Bytes of device workspace esspt_mf_load() needs for n_obs observed entries
 * of an n_users x (n_rows - n_users) matrix split into F minibatches; the
 * workspace holds the re-laid-out entries for the life of the context. */
size_t esspt_mf_workspace_bytes(const esspt_ctx* ctx, int64_t n_obs, int64_t n_users, int32_t F);

/* Bytes of temporary device scratch esspt_mf_load() needs (sort buffers);
 * the scratch may be freed once esspt_mf_load() returns. */
size_t esspt_mf_scratch_bytes(const esspt_ctx* ctx, int64_t n_obs, int64_t n_users, int32_t F);

/* Load the observed entries D_obs (Sec. 3.1) and their partition:
 *   d_i, d_j   device int32[n_obs]: user in [0, n_users), item in [0, M);
 *   d_D        device fp32[n_obs]: observed value D_ij;
 *   d_mb       device uint8[n_obs]: minibatch of each entry, in [0, F); clock
 *              c processes minibatch (c-1) mod F (Sec. 5: a fixed fraction
 *              of the data per Clock());
 *   d_worker   device int32[n_users]: worker owning each user's entries
 *              (Sec. 3.1: D_obs is partitioned over the workers), in [0, P).
 * The entries are re-laid out in `d_mf_workspace` (caller-allocated, 256-byte
 * aligned, esspt_mf_workspace_bytes() long, kept until esspt_destroy()),
 * using `d_scratch` (256-byte aligned, esspt_mf_scratch_bytes() long) during
 * the call; the input arrays and the scratch may be freed after the call
 * returns.  Synchronises.  Requires 1 <= F <= 255, n_obs < 2^31 and
 * F * n_users < 2^31.  ESSPT_EINVAL if an index is out of range (nothing is
 * loaded), ESSPT_ENOSPC if a buffer is short. */
esspt_status esspt_mf_load(esspt_ctx* ctx, const int32_t* d_i, const int32_t* d_j, const float* d_D,
                           const uint8_t* d_mb, int64_t n_obs, const int32_t* d_worker, int64_t n_users,
                           int32_t F, void* d_mf_workspace, size_t bytes, void* d_scratch,
                           size_t scratch_bytes);

/* One whole clock of stale-synchronous MF-SGD (the fused hot path):
 * for every entry (i, j) of minibatch b = (c-1) mod F owned by worker
 * p = w(i), with L_i and R_j read at version v_p(c):
 *     e = D_ij - L_i . R_j,
 *     L_i += eta (e R_j - lambda L_i),   R_j += eta (e L_i - lambda R_j)
 * (Sec. 3.1, both updates from the same read version), summed into version c
 * on top of version c-1 together with any INCs already made this clock; then
 * CLOCK as esspt_clock().  If cap > 0, the summed update of a row with n > cap
 * entries in this minibatch is scaled by cap/n (hot-row step cap; cap = 0
 * disables it).  If d_sq_loss is non-NULL (device fp64) the squared
 * residuals sum e^2 of the clock's entries, at their read versions, are
 * added to *d_sq_loss.  ESSPT_ESTATE before esspt_mf_load(). */
esspt_status esspt_mf_sgd_clock(esspt_ctx* ctx, float eta, float lambda, int32_t cap, double* d_sq_loss);

/* Bytes of the work buffer esspt_mf_sgd_clock_sequential() needs:
 * P * (n_rows - n_users) * K fp32.  0 before esspt_mf_load(). */
size_t esspt_mf_sequential_work_bytes(const esspt_ctx* ctx);

/* One clock of MF-SGD with read-my-writes inside each worker, the per-entry
 * SGD of Sec. 3.1 as each worker runs it (Sec. 5): worker p walks its
 * entries of minibatch b (its users in ascending id, a user's entries in
 * input order) and reads L_i and R_j from version v_p(c) plus its own
 * updates of this clock so far; the summed changes of all workers then make
 * version c as in esspt_mf_sgd_clock() (same cap rule, same loss output,
 * then CLOCK).  The entries of one worker form one dependent chain, so this
 * runs one warp per worker: a semantic variant, far slower than the
 * minibatch clock.  `d_work` (device, 16-byte aligned, caller-owned) must
 * hold esspt_mf_sequential_work_bytes() bytes; it is cleared by the call.
 * ESSPT_EINVAL under the row-granular model ESSPT_SSP_ROW. */
esspt_status esspt_mf_sgd_clock_sequential(esspt_ctx* ctx, float eta, float lambda, int32_t cap,
                                           double* d_sq_loss, void* d_work, size_t work_bytes);

/* Objective of Sec. 3.1 / Sec. 5 at table version `version` over ALL loaded
 * entries: *h_sq = sum e^2 (squared loss) and
 * *h_pen = sum [e^2 + lambda (|L_i|^2 + |R_j|^2)] (l2-penalised, per entry).
 * fp32 residuals, fp64 sums.  Uses `d_scratch` (device, 2 doubles).
 * Synchronises. */
esspt_status esspt_mf_objective(esspt_ctx* ctx, int32_t version, float lambda, double* d_scratch,
                                double* h_sq, double* h_pen);

/* Number of entries of minibatch b (0 <= b < F) after esspt_mf_load(). */
esspt_status esspt_mf_minibatch_size(esspt_ctx* ctx, int32_t b, int64_t* n_b);

/* Copy minibatch b as laid out on the device (entries sorted by user) to host
 * memory: h_u, h_j (int32) and h_D (fp32) hold its n_b entries, h_uoff
 * (int32, n_users+1) the offset of each user's entries.  Synchronises.
 * Together with esspt_mf_stage_minibatch() this keeps the observed entries
 * resident on the host, as each worker of Sec. 3.1 stores its own partition. */
esspt_status esspt_mf_export_minibatch(esspt_ctx* ctx, int32_t b, int32_t* h_u, int32_t* h_j, float* h_D,
                                       int32_t* h_uoff);

/* Bytes of the device staging buffer esspt_mf_stage_minibatch() needs: the
 * user and item ids of the largest minibatch plus one set of user offsets.
 * 0 before esspt_mf_load(). */
size_t esspt_mf_stage_bytes(const esspt_ctx* ctx);

/* Copy minibatch b from host memory (the arrays esspt_mf_export_minibatch()
 * produced, possibly with new values h_D) to the device, asynchronously on
 * `stream` (cudaStream_t; NULL = the context's stream; pinned host memory
 * gives a true async copy).  Together with esspt_mf_export_minibatch() this
 * keeps the observed entries resident on the host, as each worker of
 * Sec. 3.1 stores its own partition of D_obs.
 *   h_D    replaces the values of minibatch b;
 *   h_u, h_j, h_uoff  must be the loaded structure of minibatch b: they are
 *          copied into `d_stage` (device, 256-byte aligned, caller-owned,
 *          esspt_mf_stage_bytes() long) and compared on the device with the
 *          loaded layout; any difference is latched and reported by
 *          esspt_poll() as ESSPT_EINVAL.  The clock kernels never read the
 *          staged structure, so a changed one cannot make them read outside
 *          the table; only the new values take effect.
 * The caller orders the call after the last clock that read minibatch b and
 * before the next clock that reads it (e.g. with events when `stream` is not
 * the context's stream).  Calls that overlap on the GPU must use different
 * staging buffers.  The host arrays must stay valid until the stream reaches
 * the copy.  ESSPT_ENOSPC if `stage_bytes` is short. */
esspt_status esspt_mf_stage_minibatch(esspt_ctx* ctx, int32_t b, const int32_t* h_u, const int32_t* h_j,
                                      const float* h_D, const int32_t* h_uoff, void* d_stage, size_t stage_bytes,
                                      void* stream);

/* Profiling hook: when `before` and `after` (cudaEvent_t) are non-NULL,
 * every following esspt_mf_sgd_clock() records `before` on the stream just
 * before its SGD kernels (gather, residual, user-row merge) and `after` just
 * after them; the item-row Clock() merge and the next clock's schedule come
 * after `after`.  NULL, NULL turns it off. */
esspt_status esspt_set_profile_events(esspt_ctx* ctx, void* before, void* after);

/* The objective of esspt_mf_objective() split by worker, for callers that
 * cannot allocate device memory (a pool owned by another framework, a hook
 * inside a hot loop, a fixed memory budget).  It needs neither the caller's
 * scratch nor any allocation: its accumulators are a 32 KB array built into
 * the library, held by every GPU that loads it until the process exits.
 * The paper has no counterpart to this entry point.
 *   version  a final version in the live window (as esspt_mf_objective);
 *   h_sq, h_pen  host, P doubles each: per worker p, sum e^2 and
 *            sum [e^2 + lambda(|L_i|^2 + |R_j|^2)] over the entries of the
 *            users p owns.
 * At most 2048 workers; more gives ESSPT_EINVAL and queues no work.  The first
 * call on a device looks up the array's address with that device current;
 * make it before any stream capture.  Every call clears the shared array
 * first and synchronises the stream; calls that overlap on the GPU (other
 * streams, no ordering between them) race on the array. */
esspt_status esspt_mf_worker_objective_noalloc(esspt_ctx* ctx, int32_t version, float lambda, double* h_sq,
                                               double* h_pen);

#ifdef __cplusplus
}
#endif
#endif /* ESSPT_H */
