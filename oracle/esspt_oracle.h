/* Reference oracle for one clock of stale-synchronous MF-SGD.
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, single-threaded fp64 CPU
 * restatement of the paper's per-clock semantics.  It exists to check the
 * CUDA library; only the test suite, the smoke check and the benchmark's CPU
 * baseline may load it.  It shares no code, header or constant with the CUDA
 * library.
 *
 * What one clock c (1-based) computes, producing table version c:
 *   1. the read version v_p(c) of every worker p (Sec. 2.2 SSP condition;
 *      Sec. 3 formal SSP bound; Sec. 4 READ guarantee and server push; or
 *      the value bound of Sec. 2.1 VAP, see ORC_VAP), checked against
 *      max(0, c-1-s) <= v_p(c) <= c-1;
 *   2. for every observed entry (i, j) of minibatch b = (c-1) mod F, owned by
 *      worker p = w(i): e = D_ij - L_i . R_j at version v_p(c), and the
 *      Sec. 3.1 updates  dL_i += eta (e R_j - lambda L_i),
 *                         dR_j += eta (e L_i - lambda R_j),
 *      both from the same read version (no read-my-writes, Sec. 3 footnote);
 *      with `sequential` set, each worker instead walks its entries (users in
 *      ascending id, a user's entries in input order) and reads L_i and R_j
 *      from its read version plus its own updates of this clock so far;
 *   3. the Clock() merge X[c] = X[c-1] + scale (.) sum of deltas (additive
 *      updates, Sec. 2.1; coalesced per clock, Sec. 4), where scale is 1
 *      unless the hot-row step cap C is on: then row r's summed delta is
 *      scaled by min(1, C / n_r), n_r = entries of row r in this clock.
 *
 * Tables are (n_users + n_items) rows of K doubles: user rows 0..N-1 are L,
 * item rows N..N+M-1 are R (one row per item, the transpose of the paper's
 * column R_{*j}).
 */
#ifndef ESSPT_ORACLE_H
#define ESSPT_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ORC_VAP: every worker reads the stalest version v in [max(0, c-1-s), c-1]
 * whose in-transit updates X[c-1] - X[v] have max-norm at most
 * v_c = vap_v0 / sqrt(c) (Sec. 2.1 VAP condition, with the shrinking bound
 * v_t = v0 / sqrt(t) of the SGD-under-VAP theorem of Sec. 3); version c-1
 * always qualifies. */
/* ORC_SSP_ROW: SSP with row-granular lazy refresh (Sec. 4 client cache: each
 * cached row has its own clock c_param).  Worker p holds row r at version
 * V[p][r], none before its first read.  At clock c every row the worker
 * reads (the rows of its entries in this clock's minibatch) is refreshed to
 * version c-1 if it is not held or V[p][r] < c-1-s, and read at V[p][r];
 * all reads of a row in one clock see the same version. */
enum { ORC_SSP_LAZY = 0, ORC_ESSP_EAGER = 1, ORC_EXTERNAL = 2, ORC_VAP = 3, ORC_SSP_ROW = 4 };

typedef struct {
  int64_t n_users;     /* N */
  int64_t n_items;     /* M */
  int32_t K;           /* rank */
  int32_t P;           /* workers */
  int32_t s;           /* staleness bound */
  int32_t F;           /* minibatches per pass; clock c uses b = (c-1) mod F */
  int32_t model;       /* ORC_SSP_LAZY / ORC_ESSP_EAGER / ORC_EXTERNAL / ORC_VAP / ORC_SSP_ROW */
  int32_t phased;      /* SSP: 1 = seeded per-worker refresh phase, 0 = none */
  uint64_t seed;       /* schedule seed */
  double essp_p;       /* ESSP delay ~ Geometric(essp_p), failures before success */
  int32_t essp_max_delay;
  int32_t cap;         /* hot-row step cap C; 0 = off */
  double eta;          /* step size */
  double lambda;       /* l2 penalty, per observation */
  int32_t keep_all;    /* 1 = keep every version (unbounded history) */
  double vap_v0;       /* ORC_VAP: initial value bound v0 */
  int32_t eta_decay;   /* 1 = clock c uses eta / sqrt(c) (the step-size schedule of the Sec. 3 theorems) */
  int32_t sequential;  /* 1 = each worker runs sequential SGD over its entries, seeing its own
                          updates within the clock (read-my-writes; Sec. 3.1 as run in Sec. 5) */
} orc_config;

typedef struct orc_state orc_state;

/* Input arrays are borrowed, not copied, and must outlive the state.
 * Returns NULL on invalid arguments or allocation failure. */
orc_state* orc_create(const orc_config* cfg, int64_t n_obs, const int32_t* i, const int32_t* j,
                      const float* D, const uint8_t* minibatch, const int32_t* user_worker,
                      const float* L0, const float* R0);
void orc_destroy(orc_state* st);

/* Run one clock.  v_ext (P entries) is read only for ORC_EXTERNAL.
 * Returns 0, or -1 on a staleness-bound violation (state unchanged). */
int orc_clock(orc_state* st, const int32_t* v_ext);

/* Completed clocks (= newest version). */
int32_t orc_version(const orc_state* st);

/* Read versions used by the last clock, P entries.  Returns -1 before clock 1.
 * ORC_SSP_ROW reports c-1 for every worker (its reads are per row). */
int orc_schedule(const orc_state* st, int32_t* v_out);

/* Copy table version `version` ((N+M)*K doubles).  Returns -1 if not held. */
int orc_table(const orc_state* st, int32_t version, double* out);

/* Objective at `version` over ALL observed entries:
 * sq = sum e^2 (Sec. 5 squared loss), pen = sum [e^2 + lambda(|L_i|^2+|R_j|^2)]. */
int orc_objective(const orc_state* st, int32_t version, double* sq, double* pen);

/* ORC_ESSP_EAGER delay thresholds: thr[k-1] = floor((1-essp_p)^k 2^32) for
 * k = 1..essp_max_delay (a delay is >= k iff the draw's top 32 bits are below
 * thr[k-1]).  Returns essp_max_delay. */
int orc_essp_thresholds(const orc_config* cfg, uint32_t* thr);

/* Squared loss of the last clock: sum of e^2 over the entries of its
 * minibatch, each e taken where its update was computed (at the worker's
 * read version; in the sequential variant, at the worker's view just before
 * the entry).  Returns -1 before clock 1. */
int orc_clock_loss(const orc_state* st, double* out);

/* ORC_VAP: the in-transit max-norms the last clock c compared against its
 * bound: out[k] = |X[c-1] - X[c-1-k]|_inf for k = 0..s (0 where c-1-k < 0),
 * and *bound = vap_v0 / sqrt(c).  Returns -1 for other models or before
 * clock 1. */
int orc_vap_norms(const orc_state* st, double* out, double* bound);

/* ORC_SSP_ROW: the version worker p holds row r at (after the last clock's
 * refreshes), -1 if it has never read it.  Returns -1 for other models. */
int orc_row_version(const orc_state* st, int32_t p, int64_t r, int32_t* out);

/* The schedule rule alone, for clock c, given the previous read versions.
 * Used by the schedule tests; orc_clock calls the same function. */
int orc_schedule_rule(const orc_config* cfg, int32_t c, const int32_t* v_prev, int32_t* v_out);

/* The counter generator (SplitMix64) draw `index` of `stream` under `seed`. */
uint64_t orc_ctr_u64(uint64_t seed, uint64_t stream, uint64_t index);

#ifdef __cplusplus
}
#endif
#endif
