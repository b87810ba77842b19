/* Reference oracle for stale-synchronous MF-SGD: plain fp64 C, single thread.
 *
 * TEST INFRASTRUCTURE ONLY (tests, smoke check, CPU baseline of the bench).
 * See esspt_oracle.h for the per-clock semantics and the paper passages they
 * follow.  Readings of passages the paper leaves open:
 *   - clocks are 1-based; version v is the table after clocks 1..v; a read at
 *     clock c must see every update of clocks 1..c-1-s, so
 *     max(0, c-1-s) <= v_p(c) <= c-1, and s = 0 gives v = c-1: the BSP
 *     clock differential v - c = -1 of Fig. 1;
 *   - SSP lazy pull refreshes a worker's whole cached table only when it
 *     would otherwise break the bound (the SSP worker of Sec. 2.2 defers its
 *     refresh as long as the bound allows), at a seeded per-worker phase phi_p
 *     in [0, s];
 *   - ESSP eager push: the server's push of version c-1 reaches worker p
 *     after a delay of delta_{p,c} ~ Geometric(p) clocks clamped to
 *     [0, min(max_delay, s)]; the read version never goes backwards;
 *   - all entries of a worker in one clock read the same version and both
 *     updates use the old L_i and R_j (no read-my-writes, Sec. 3 footnote);
 *   - VAP (Sec. 2.1): a worker reading version v at clock c has the updates
 *     X[c-1] - X[v] in transit; in this lockstep simulation every worker
 *     refreshes as lazily as the value bound allows, i.e. reads the stalest
 *     version inside the staleness window whose in-transit max-norm is at
 *     most v0 / sqrt(c) (the shrinking bound v_t = v0 / sqrt(t) of the
 *     SGD-under-VAP theorem, Sec. 3, with t = c); a NaN norm never qualifies;
 *   - row-granular SSP (Sec. 4 client cache, one c_param per row): a row not
 *     in the cache is fetched at the server's newest version, c-1 (the first
 *     read registers the row); a cached row at version v serves a read at
 *     clock c while v >= c-1-s (the same bound as above) and is otherwise
 *     refreshed to c-1.  The cache never evicts;
 *   - sequential (read-my-writes) SGD: the order of a worker's entries in a
 *     clock is not given; users are taken in ascending id and a user's
 *     entries in input order.  The worker's summed change joins the Clock()
 *     merge like any other delta.
 */
#include "esspt_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#define ORC_STREAM_PHASE 101u
#define ORC_STREAM_DELAY 102u

/* SplitMix64 (Steele, Lea and Flood, OOPSLA 2014): output n of a sequence
 * with initial state s0 is mix(s0 + n * 0x9E3779B97F4A7C15). */
static uint64_t orc_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

uint64_t orc_ctr_u64(uint64_t seed, uint64_t stream, uint64_t index) {
  uint64_t s0 = orc_mix64(seed) ^ orc_mix64(stream);
  return orc_mix64(s0 + (index + 1u) * 0x9E3779B97F4A7C15ull);
}

/* Map a draw to [0, n) by the multiply-high of its top 32 bits. */
static uint32_t orc_below(uint64_t h, uint32_t n) {
  return (uint32_t)(((h >> 32) * (uint64_t)n) >> 32);
}

struct orc_state {
  orc_config cfg;
  int64_t n_obs;
  const int32_t* i;
  const int32_t* j;
  const float* D;
  const uint8_t* mb;
  const int32_t* w;
  int64_t rows;     /* N + M */
  int32_t nslots;   /* versions held */
  double* tables;   /* nslots * rows * K */
  int32_t version;  /* newest complete version */
  int32_t* v_prev;  /* read versions of the last clock (P) */
  double* delta;    /* rows * K */
  int64_t* count;   /* rows, entries per row in this clock */
  double* vap_norm; /* s+1, ORC_VAP norms of the last clock */
  int32_t* rowver;  /* ORC_SSP_ROW: P * rows cached versions, -1 = not held */
  double vap_bound; /* ORC_VAP bound of the last clock */
  double clock_sq;  /* sum of e^2 over the last clock's entries */
};

static double* orc_slot(const orc_state* st, int32_t version) {
  int64_t slot = st->cfg.keep_all ? version : version % st->nslots;
  return st->tables + slot * st->rows * st->cfg.K;
}

static int orc_holds(const orc_state* st, int32_t version) {
  if (version < 0 || version > st->version) return 0;
  if (st->cfg.keep_all) return 1;
  return version > st->version - st->nslots;
}

/* P(delay >= k) = (1-p)^k for a delay counted in failures before the first
 * success; as a 32-bit threshold, floor((1-p)^k 2^32).  *q holds (1-p)^(k-1)
 * on entry and (1-p)^k on return. */
static uint32_t orc_threshold_next(double* q, double fail) {
  *q *= fail;
  return (uint32_t)floor(*q * 4294967296.0);
}

int orc_essp_thresholds(const orc_config* cfg, uint32_t* thr) {
  double q = 1.0;
  for (int32_t k = 1; k <= cfg->essp_max_delay; ++k) thr[k - 1] = orc_threshold_next(&q, 1.0 - cfg->essp_p);
  return cfg->essp_max_delay;
}

int orc_schedule_rule(const orc_config* cfg, int32_t c, const int32_t* v_prev, int32_t* v_out) {
  int32_t lo = c - 1 - cfg->s;
  if (lo < 0) lo = 0;
  for (int32_t p = 0; p < cfg->P; ++p) {
    int32_t v;
    if (cfg->model == ORC_SSP_LAZY) {
      /* Lazy pull: staleness (c-1) - v cycles 0, 1, ..., s with phase phi_p. */
      int32_t phi = 0;
      if (cfg->phased) phi = (int32_t)orc_below(orc_ctr_u64(cfg->seed, ORC_STREAM_PHASE, (uint64_t)p), (uint32_t)(cfg->s + 1));
      v = (c - 1) - ((c - 1 + phi) % (cfg->s + 1));
      if (v < 0) v = 0;
    } else if (cfg->model == ORC_ESSP_EAGER) {
      /* Eager push: delay = number of failures before the first success of a
       * Bernoulli(essp_p) sequence, by inverse CDF on a 32-bit uniform u:
       * delay >= k  iff  u < floor((1-essp_p)^k * 2^32). */
      int32_t dmax = cfg->essp_max_delay < cfg->s ? cfg->essp_max_delay : cfg->s;
      uint32_t u = (uint32_t)(orc_ctr_u64(cfg->seed, ORC_STREAM_DELAY, ((uint64_t)(uint32_t)c << 32) | (uint32_t)p) >> 32);
      double q = 1.0;
      int32_t delay = 0;
      for (int32_t k = 1; k <= dmax; ++k)
        if (u < orc_threshold_next(&q, 1.0 - cfg->essp_p)) delay = k;
      v = c - 1 - delay;
      if (v_prev != NULL && v_prev[p] > v) v = v_prev[p];
      if (v < 0) v = 0;
    } else {
      return -1;
    }
    v_out[p] = v;
  }
  for (int32_t p = 0; p < cfg->P; ++p)
    if (v_out[p] < lo || v_out[p] > c - 1) return -1;
  return 0;
}

/* ORC_VAP read version of clock c: the stalest v in the window whose
 * in-transit max-norm |X[c-1] - X[v]|_inf is at most v0 / sqrt(c). */
static int32_t orc_vap_version(orc_state* st, int32_t c) {
  const orc_config* cfg = &st->cfg;
  const int64_t n = st->rows * cfg->K;
  const double* cur = orc_slot(st, c - 1);
  const double bound = cfg->vap_v0 / sqrt((double)c);
  int32_t v = c - 1;
  for (int32_t k = 0; k <= cfg->s; ++k) st->vap_norm[k] = 0.0;
  st->vap_bound = bound;
  for (int32_t k = cfg->s; k >= 1; --k) {
    if (c - 1 - k < 0) continue;
    const double* old = orc_slot(st, c - 1 - k);
    double m = 0.0;
    for (int64_t x = 0; x < n; ++x) {
      double d = fabs(cur[x] - old[x]);
      if (d != d) {
        m = d;
        break;
      }
      if (d > m) m = d;
    }
    st->vap_norm[k] = m;
  }
  for (int32_t k = cfg->s; k >= 1; --k) {
    if (c - 1 - k < 0) continue;
    if (st->vap_norm[k] <= bound) {
      v = c - 1 - k;
      break;
    }
  }
  return v;
}

int orc_vap_norms(const orc_state* st, double* out, double* bound) {
  if (st->cfg.model != ORC_VAP || st->version < 1) return -1;
  memcpy(out, st->vap_norm, (size_t)(st->cfg.s + 1) * sizeof(double));
  *bound = st->vap_bound;
  return 0;
}

orc_state* orc_create(const orc_config* cfg, int64_t n_obs, const int32_t* i, const int32_t* j,
                      const float* D, const uint8_t* minibatch, const int32_t* user_worker,
                      const float* L0, const float* R0) {
  if (!cfg || cfg->n_users <= 0 || cfg->n_items <= 0 || cfg->K <= 0 || cfg->P <= 0 || cfg->s < 0 ||
      cfg->F <= 0 || n_obs < 0 || cfg->model < 0 || cfg->model > ORC_SSP_ROW ||
      (cfg->model == ORC_VAP && !(cfg->vap_v0 >= 0.0)) || (cfg->sequential && cfg->model == ORC_SSP_ROW))
    return NULL;
  orc_state* st = (orc_state*)calloc(1, sizeof(orc_state));
  if (!st) return NULL;
  st->cfg = *cfg;
  st->n_obs = n_obs;
  st->i = i;
  st->j = j;
  st->D = D;
  st->mb = minibatch;
  st->w = user_worker;
  st->rows = cfg->n_users + cfg->n_items;
  /* s+1 readable versions plus the one being written. */
  st->nslots = cfg->keep_all ? 1 : cfg->s + 2;
  int64_t K = cfg->K;
  st->tables = (double*)calloc((size_t)(st->nslots * st->rows * K), sizeof(double));
  st->v_prev = (int32_t*)calloc((size_t)cfg->P, sizeof(int32_t));
  st->delta = (double*)calloc((size_t)(st->rows * K), sizeof(double));
  st->count = (int64_t*)calloc((size_t)st->rows, sizeof(int64_t));
  st->vap_norm = (double*)calloc((size_t)cfg->s + 1, sizeof(double));
  if (cfg->model == ORC_SSP_ROW) {
    st->rowver = (int32_t*)malloc((size_t)cfg->P * (size_t)st->rows * sizeof(int32_t));
    if (st->rowver)
      for (int64_t x = 0; x < (int64_t)cfg->P * st->rows; ++x) st->rowver[x] = -1;
  }
  if (!st->tables || !st->v_prev || !st->delta || !st->count || !st->vap_norm ||
      (cfg->model == ORC_SSP_ROW && !st->rowver)) {
    orc_destroy(st);
    return NULL;
  }
  double* x0 = st->tables;
  for (int64_t r = 0; r < cfg->n_users; ++r)
    for (int64_t q = 0; q < K; ++q) x0[r * K + q] = (double)L0[r * K + q];
  for (int64_t r = 0; r < cfg->n_items; ++r)
    for (int64_t q = 0; q < K; ++q) x0[(cfg->n_users + r) * K + q] = (double)R0[r * K + q];
  st->version = 0;
  return st;
}

void orc_destroy(orc_state* st) {
  if (!st) return;
  free(st->tables);
  free(st->v_prev);
  free(st->delta);
  free(st->count);
  free(st->vap_norm);
  free(st->rowver);
  free(st);
}

static int orc_grow(orc_state* st) {
  /* keep_all: one more version slot. */
  size_t per = (size_t)(st->rows * st->cfg.K);
  double* t = (double*)realloc(st->tables, (size_t)(st->nslots + 1) * per * sizeof(double));
  if (!t) return -1;
  st->tables = t;
  st->nslots += 1;
  return 0;
}

static int orc_sequential_deltas(orc_state* st, const int32_t* v, uint8_t b, double eta);

int orc_clock(orc_state* st, const int32_t* v_ext) {
  const orc_config* cfg = &st->cfg;
  const int64_t K = cfg->K, N = cfg->n_users;
  int32_t c = st->version + 1;
  int32_t* v = (int32_t*)malloc((size_t)cfg->P * sizeof(int32_t));
  if (!v) return -2;

  /* 1. Read versions. */
  if (cfg->model == ORC_EXTERNAL) {
    int32_t lo = c - 1 - cfg->s < 0 ? 0 : c - 1 - cfg->s;
    for (int32_t p = 0; p < cfg->P; ++p) {
      v[p] = v_ext[p];
      if (v[p] < lo || v[p] > c - 1) {
        free(v);
        return -1;
      }
    }
  } else if (cfg->model == ORC_VAP) {
    const int32_t vv = orc_vap_version(st, c);
    for (int32_t p = 0; p < cfg->P; ++p) v[p] = vv;
  } else if (cfg->model == ORC_SSP_ROW) {
    for (int32_t p = 0; p < cfg->P; ++p) v[p] = c - 1;
  } else if (orc_schedule_rule(cfg, c, st->v_prev, v) != 0) {
    free(v);
    return -1;
  }
  if (cfg->keep_all && orc_grow(st) != 0) {
    free(v);
    return -2;
  }

  /* 2. Deltas of every entry of minibatch b, each at its worker's version. */
  memset(st->delta, 0, (size_t)(st->rows * K) * sizeof(double));
  memset(st->count, 0, (size_t)st->rows * sizeof(int64_t));
  st->clock_sq = 0.0;
  const uint8_t b = (uint8_t)((c - 1) % cfg->F);
  const double eta = cfg->eta_decay ? cfg->eta / sqrt((double)c) : cfg->eta;
  if (cfg->sequential) {
    if (orc_sequential_deltas(st, v, b, eta) != 0) {
      free(v);
      return -2;
    }
  } else if (cfg->model == ORC_SSP_ROW) {
    /* Refresh every row a worker reads this clock, before any read. */
    const int32_t lo = c - 1 - cfg->s;
    for (int64_t k = 0; k < st->n_obs; ++k) {
      if (st->mb[k] != b) continue;
      int64_t ui = st->i[k], ij = st->j[k];
      int32_t* V = st->rowver + (int64_t)st->w[ui] * st->rows;
      if (V[ui] < 0 || V[ui] < lo) V[ui] = c - 1;
      if (V[N + ij] < 0 || V[N + ij] < lo) V[N + ij] = c - 1;
    }
  }
  for (int64_t k = 0; k < st->n_obs && !cfg->sequential; ++k) {
    if (st->mb[k] != b) continue;
    int64_t ui = st->i[k], ij = st->j[k];
    int32_t p = st->w[ui];
    const double* Li;
    const double* Rj;
    if (cfg->model == ORC_SSP_ROW) {
      const int32_t* V = st->rowver + (int64_t)p * st->rows;
      Li = orc_slot(st, V[ui]) + ui * K;
      Rj = orc_slot(st, V[N + ij]) + (N + ij) * K;
    } else {
      const double* x = orc_slot(st, v[p]);
      Li = x + ui * K;
      Rj = x + (N + ij) * K;
    }
    double dot = 0.0;
    for (int64_t q = 0; q < K; ++q) dot += Li[q] * Rj[q];
    double e = (double)st->D[k] - dot;
    st->clock_sq += e * e;
    double* dL = st->delta + ui * K;
    double* dR = st->delta + (N + ij) * K;
    for (int64_t q = 0; q < K; ++q) {
      dL[q] += eta * (e * Rj[q] - cfg->lambda * Li[q]);
      dR[q] += eta * (e * Li[q] - cfg->lambda * Rj[q]);
    }
    st->count[ui] += 1;
    st->count[N + ij] += 1;
  }

  /* 3. Clock() merge into version c. */
  const double* prev = orc_slot(st, c - 1);
  st->version = c; /* slot of c is now addressable */
  double* next = orc_slot(st, c);
  for (int64_t r = 0; r < st->rows; ++r) {
    double scale = 1.0;
    if (cfg->cap > 0 && st->count[r] > cfg->cap) scale = (double)cfg->cap / (double)st->count[r];
    for (int64_t q = 0; q < K; ++q) next[r * K + q] = prev[r * K + q] + scale * st->delta[r * K + q];
  }
  memcpy(st->v_prev, v, (size_t)cfg->P * sizeof(int32_t));
  free(v);
  return 0;
}

/* Sequential SGD of every worker over its entries of minibatch b at clock c:
 * worker p's view of row r is X[v_p(c)][r] + its own delta of this clock so
 * far.  Adds each worker's delta and the entry counts into st->delta and
 * st->count.  Returns -2 on allocation failure. */
static int orc_sequential_deltas(orc_state* st, const int32_t* v, uint8_t b, double eta) {
  const orc_config* cfg = &st->cfg;
  const int64_t K = cfg->K, N = cfg->n_users;
  /* Entries of minibatch b grouped by user, input order within a user. */
  int64_t* uoff = (int64_t*)calloc((size_t)N + 1, sizeof(int64_t));
  double* mine = (double*)calloc((size_t)(st->rows * K), sizeof(double));
  int32_t* stamp = (int32_t*)malloc((size_t)st->rows * sizeof(int32_t));
  int64_t* touched = (int64_t*)malloc((size_t)st->rows * sizeof(int64_t));
  if (!uoff || !mine || !stamp || !touched) {
    free(uoff), free(mine), free(stamp), free(touched);
    return -2;
  }
  int64_t nb = 0;
  for (int64_t k = 0; k < st->n_obs; ++k)
    if (st->mb[k] == b) uoff[st->i[k] + 1] += 1, ++nb;
  for (int64_t u = 0; u < N; ++u) uoff[u + 1] += uoff[u];
  int64_t* order = (int64_t*)malloc((size_t)(nb > 0 ? nb : 1) * sizeof(int64_t));
  int64_t* fill = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  if (!order || !fill) {
    free(uoff), free(mine), free(stamp), free(touched), free(order), free(fill);
    return -2;
  }
  memcpy(fill, uoff, (size_t)N * sizeof(int64_t));
  for (int64_t k = 0; k < st->n_obs; ++k)
    if (st->mb[k] == b) order[fill[st->i[k]]++] = k;
  for (int64_t r = 0; r < st->rows; ++r) stamp[r] = -1;

  for (int32_t p = 0; p < cfg->P; ++p) {
    const double* x = orc_slot(st, v[p]);
    int64_t nt = 0;
    for (int64_t u = 0; u < N; ++u) {
      if (st->w[u] != p) continue;
      for (int64_t t = uoff[u]; t < uoff[u + 1]; ++t) {
        const int64_t k = order[t], ij = st->j[k], rj = N + ij;
        const int64_t rows2[2] = {u, rj};
        for (int q2 = 0; q2 < 2; ++q2)
          if (stamp[rows2[q2]] != p) stamp[rows2[q2]] = p, touched[nt++] = rows2[q2];
        double* mL = mine + u * K;
        double* mR = mine + rj * K;
        double dot = 0.0;
        for (int64_t q = 0; q < K; ++q) dot += (x[u * K + q] + mL[q]) * (x[rj * K + q] + mR[q]);
        const double e = (double)st->D[k] - dot;
        st->clock_sq += e * e;
        for (int64_t q = 0; q < K; ++q) {
          const double Lq = x[u * K + q] + mL[q], Rq = x[rj * K + q] + mR[q];
          mL[q] += eta * (e * Rq - cfg->lambda * Lq);
          mR[q] += eta * (e * Lq - cfg->lambda * Rq);
        }
        st->count[u] += 1;
        st->count[rj] += 1;
      }
    }
    for (int64_t t = 0; t < nt; ++t) {
      const int64_t r = touched[t];
      for (int64_t q = 0; q < K; ++q) {
        st->delta[r * K + q] += mine[r * K + q];
        mine[r * K + q] = 0.0;
      }
    }
  }
  free(uoff), free(mine), free(stamp), free(touched), free(order), free(fill);
  return 0;
}

int32_t orc_version(const orc_state* st) { return st->version; }

int orc_row_version(const orc_state* st, int32_t p, int64_t r, int32_t* out) {
  if (st->cfg.model != ORC_SSP_ROW || p < 0 || p >= st->cfg.P || r < 0 || r >= st->rows) return -1;
  *out = st->rowver[(int64_t)p * st->rows + r];
  return 0;
}

int orc_clock_loss(const orc_state* st, double* out) {
  if (st->version < 1) return -1;
  *out = st->clock_sq;
  return 0;
}

int orc_schedule(const orc_state* st, int32_t* v_out) {
  if (st->version < 1) return -1;
  memcpy(v_out, st->v_prev, (size_t)st->cfg.P * sizeof(int32_t));
  return 0;
}

int orc_table(const orc_state* st, int32_t version, double* out) {
  if (!orc_holds(st, version)) return -1;
  memcpy(out, orc_slot(st, version), (size_t)(st->rows * st->cfg.K) * sizeof(double));
  return 0;
}

int orc_objective(const orc_state* st, int32_t version, double* sq, double* pen) {
  if (!orc_holds(st, version)) return -1;
  const int64_t K = st->cfg.K, N = st->cfg.n_users;
  const double* x = orc_slot(st, version);
  double s1 = 0.0, s2 = 0.0;
  for (int64_t k = 0; k < st->n_obs; ++k) {
    const double* Li = x + (int64_t)st->i[k] * K;
    const double* Rj = x + (N + st->j[k]) * K;
    double dot = 0.0, nl = 0.0, nr = 0.0;
    for (int64_t q = 0; q < K; ++q) {
      dot += Li[q] * Rj[q];
      nl += Li[q] * Li[q];
      nr += Rj[q] * Rj[q];
    }
    double e = (double)st->D[k] - dot;
    s1 += e * e;
    s2 += e * e + st->cfg.lambda * (nl + nr);
  }
  *sq = s1;
  *pen = s2;
  return 0;
}
