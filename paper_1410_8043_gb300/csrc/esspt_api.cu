// The esspt C-ABI: context, version-ring state machine and launches.
// Every entry point returns a status; no exception crosses the ABI.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

using namespace esspt;

struct esspt_ctx {
  esspt_config cfg{};
  cudaStream_t st = nullptr;
  int64_t n_rows = 0;
  int32_t K = 0, P = 0, s = 0, nslots = 0, dmax = 0;
  float* ring = nullptr;
  int32_t* v = nullptr;
  uint32_t* status = nullptr;
  uint32_t* thr = nullptr;
  uint32_t* vap_norm = nullptr;  // [s+1] VAP in-transit norms of the current clock
  int32_t clock = 0;      // clock in progress (0 = table not initialised)
  bool acc_ready = false; // slot of version `clock` holds version clock-1 + INCs so far
  bool sched_set = false; // ESSPT_EXTERNAL: v_p(clock) supplied
  std::string err;
  // matrix factorisation
  bool mf = false;
  int64_t n_users = 0, n_items = 0, n_obs = 0;
  int32_t F = 0;
  int32_t *rec_u = nullptr, *rec_j = nullptr, *uoff = nullptr, *item_cnt = nullptr, *worker = nullptr;
  int32_t *item_rep = nullptr, *rec_dst = nullptr;
  float *rec_D = nullptr, *dR = nullptr, *dL = nullptr;
  int32_t* rowver = nullptr;     // row-granular SSP: [P][n_rows] cached versions, -1 = never read
  int32_t* user_slot = nullptr;  // row-granular SSP: [n_users] per-clock ring slot of each user row
  int32_t* rec_row = nullptr;    // row-granular SSP: per-clock ring row of each entry's item row
  int4 *chunk = nullptr, *heavy = nullptr;
  std::vector<int64_t> mb_base, chunk_base, heavy_base;
  cudaEvent_t ev_before = nullptr, ev_after = nullptr;
  // Work-list path: last clock that changed each user row, and the last clock
  // at which every idle row is still copied forward (after an INC or a
  // sequential clock, whose writes are not tracked per row).
  int32_t* chg = nullptr;
  int32_t copy_all_until = 0;
  int32_t* hot_item = nullptr;   // work-list path: [F][kHot] hot items of each minibatch
};

namespace {

thread_local std::string g_create_err;

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

esspt_status fail(esspt_ctx* c, esspt_status code, const std::string& msg) {
  if (c) c->err = msg;
  return code;
}

esspt_status cuda_fail(esspt_ctx* c, cudaError_t e, const char* where) {
  return fail(c, ESSPT_ECUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

#define ESSPT_CUDA(ctx, call)                                        \
  do {                                                               \
    cudaError_t e_ = (call);                                         \
    if (e_ != cudaSuccess) return cuda_fail((ctx), e_, #call);       \
  } while (0)

bool config_ok(const esspt_config* c, std::string* why) {
  if (!c) return *why = "null config", false;
  if (c->n_rows <= 0) return *why = "n_rows must be > 0", false;
  if (c->row_width < 4 || c->row_width > 512 || c->row_width % 4 != 0)
    return *why = "row_width must be a multiple of 4 in [4, 512]", false;
  if (c->num_workers < 1 || c->num_workers > 65536) return *why = "num_workers must be in [1, 65536]", false;
  if (c->staleness < 0 || c->staleness > (1 << 20)) return *why = "staleness must be in [0, 2^20]", false;
  if (c->model < ESSPT_SSP_LAZY || c->model > ESSPT_SSP_ROW) return *why = "unknown model", false;
  // The SGD kernels index item rows with 32-bit float4 offsets; in row mode
  // the offset spans the whole ring.
  if (c->model == ESSPT_SSP_ROW &&
      (double)(c->staleness + 2) * (double)c->n_rows * (double)(c->row_width / 4) >= 2147483647.0)
    return *why = "row-granular model: the ring must hold fewer than 2^31 float4", false;
  if (c->model == ESSPT_VAP && !(c->vap_v0 >= 0.0)) return *why = "vap_v0 must be >= 0", false;
  if (c->model == ESSPT_ESSP_EAGER) {
    if (!(c->essp_p > 0.0 && c->essp_p <= 1.0)) return *why = "essp_p must be in (0, 1]", false;
    if (c->essp_max_delay < 0) return *why = "essp_max_delay must be >= 0", false;
  }
  const double ring = (double)(c->staleness + 2) * (double)c->n_rows * (double)c->row_width * 4.0;
  if (ring > 9.0e18) return *why = "table too large", false;
  return true;
}

int32_t delay_max(const esspt_config* c) {
  if (c->model != ESSPT_ESSP_EAGER) return 0;
  return c->essp_max_delay < c->staleness ? c->essp_max_delay : c->staleness;
}

struct Carve {
  size_t ring, v, status, thr, vap, rowver, total;
};

Carve carve(const esspt_config* c) {
  Carve k{};
  size_t o = 0;
  k.ring = o;
  o += align256((size_t)(c->staleness + 2) * (size_t)c->n_rows * (size_t)c->row_width * sizeof(float));
  k.v = o;
  o += align256(sizeof(int32_t) * (size_t)c->num_workers);
  k.status = o;
  o += 256;
  k.thr = o;
  o += align256(sizeof(uint32_t) * (size_t)(delay_max(c) + 1));
  k.vap = o;
  o += c->model == ESSPT_VAP ? align256(sizeof(uint32_t) * (size_t)(c->staleness + 1)) : 0;
  k.rowver = o;
  o += c->model == ESSPT_SSP_ROW ? align256(sizeof(int32_t) * (size_t)c->num_workers * (size_t)c->n_rows) : 0;
  k.total = o;
  return k;
}

float* slot_ptr(const esspt_ctx* c, int64_t version) {
  return c->ring + (version % c->nslots) * c->n_rows * c->K;
}

esspt_status need_init(esspt_ctx* c) {
  if (!c) return ESSPT_EINVAL;
  if (c->clock < 1) return fail(c, ESSPT_ESTATE, "table not initialised (call esspt_table_init)");
  return ESSPT_OK;
}

esspt_status need_schedule(esspt_ctx* c) {
  if (c->cfg.model == ESSPT_EXTERNAL && !c->sched_set)
    return fail(c, ESSPT_ESTATE, "external model: call esspt_set_schedule for this clock first");
  return ESSPT_OK;
}

// Compute v_p(clock) on the device (or only check it, for ESSPT_EXTERNAL).
ScheduleArgs schedule_args(const esspt_ctx* c, int32_t clock);

esspt_status run_schedule(esspt_ctx* c) {
  if (c->cfg.model == ESSPT_VAP) {
    // In-transit norms of the candidate versions against version clock-1.
    const int32_t kmax = std::min(c->s, c->clock - 1);
    ESSPT_CUDA(c, cudaMemsetAsync(c->vap_norm, 0, sizeof(uint32_t) * (size_t)(c->s + 1), c->st));
    if (kmax > 0)
      ESSPT_CUDA(c, launch_vap_norms(c->ring, c->n_rows * c->K, c->nslots, c->clock, kmax, c->vap_norm, c->st));
  }
  ESSPT_CUDA(c, launch_schedule(schedule_args(c, c->clock), c->st));
  return ESSPT_OK;
}

// Make the slot of version `clock` hold version clock-1 (before any delta).
esspt_status ensure_acc(esspt_ctx* c) {
  if (c->acc_ready) return ESSPT_OK;
  ESSPT_CUDA(c, launch_copy_rows(slot_ptr(c, c->clock), slot_ptr(c, c->clock - 1), c->n_rows * c->K, c->st));
  c->acc_ready = true;
  return ESSPT_OK;
}

// Version `clock` is final: advance and schedule the next clock (unless a
// kernel of the clock already did, `scheduled`).
esspt_status advance(esspt_ctx* c, bool scheduled = false) {
  c->clock += 1;
  c->acc_ready = false;
  c->sched_set = false;
  if (c->cfg.model == ESSPT_EXTERNAL || scheduled) return ESSPT_OK;
  return run_schedule(c);
}

ScheduleArgs schedule_args(const esspt_ctx* c, int32_t clock) {
  ScheduleArgs a{};
  a.v = c->v;
  a.status = c->status;
  a.thr = c->thr;
  a.P = c->P;
  a.c = clock;
  a.s = c->s;
  a.model = c->cfg.model;
  a.phased = c->cfg.phased;
  a.dmax = c->dmax;
  a.seed = c->cfg.seed;
  a.vap_norm = c->vap_norm;
  a.vap_bound = c->cfg.model == ESSPT_VAP ? c->cfg.vap_v0 / std::sqrt((double)clock) : 0.0;
  return a;
}

bool is_host_ptr(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return true;
  }
  return at.type == cudaMemoryTypeHost || at.type == cudaMemoryTypeUnregistered;
}

struct MfCarve {
  size_t rec_u, rec_j, rec_D, rec_dst, uoff, mb_base, item_cnt, item_rep, dR, worker, chunk, chunk_base, heavy, heavy_base, dL,
      user_slot, rec_row, chg, hot_item, total;
  int64_t max_chunks, max_heavy, dR_rows, dL_rows;
};

// Persistent MF workspace: entries laid out by (minibatch, user), per-minibatch
// user offsets and item counts, item replica rows, heavy-user lists and the
// zero-initialised delta replicas dR (items) and dL (heavy users).
MfCarve mf_carve(int64_t n_obs, int64_t n_users, int64_t n_items, int32_t F, int32_t K, bool row_mode) {
  MfCarve k{};
  k.max_chunks = layout_max_chunks(n_obs, F, n_users, uses_work16(K));
  k.max_heavy = layout_max_heavy(n_obs, F);
  k.dR_rows = layout_max_item_reps(n_obs, n_items);
  k.dL_rows = n_users + layout_max_user_reps(n_obs);
  size_t o = 0;
  auto take = [&o](size_t bytes) {
    const size_t at = o;
    o += align256(bytes);
    return at;
  };
  // 16 bytes of slack past the entry arrays for vector-aligned staging.
  k.rec_u = take(sizeof(int32_t) * (n_obs + 4));
  k.rec_j = take(sizeof(int32_t) * (n_obs + 4));
  k.rec_D = take(sizeof(float) * (n_obs + 4));
  k.rec_dst = take(sizeof(int32_t) * (n_obs + 4));
  k.uoff = take(sizeof(int32_t) * (size_t)F * (n_users + 1));
  k.mb_base = take(sizeof(int64_t) * (F + 1));
  k.item_cnt = take(sizeof(int32_t) * (size_t)F * n_items);
  k.item_rep = take(sizeof(int32_t) * (n_items + 1));
  k.dR = take(sizeof(float4) * (size_t)k.dR_rows * dR_stride4(K));
  k.worker = take(sizeof(int32_t) * n_users);
  k.chunk = take(sizeof(int4) * k.max_chunks);
  k.chunk_base = take(sizeof(int64_t) * (F + 1));
  k.heavy = take(sizeof(int4) * k.max_heavy);
  k.heavy_base = take(sizeof(int64_t) * (F + 1));
  k.dL = take(sizeof(float) * (size_t)k.dL_rows * K);
  // Row-granular SSP: per-clock user slots and entry ring rows (a minibatch
  // holds at most n_obs entries).
  k.user_slot = row_mode ? take(sizeof(int32_t) * n_users) : o;
  k.rec_row = row_mode ? take(sizeof(int32_t) * (n_obs + 4)) : o;
  // Work-list path: the clock that last changed each user row.
  k.chg = uses_work16(K) ? take(sizeof(int32_t) * n_users) : o;
  k.hot_item = uses_hot(K) ? take(sizeof(int32_t) * (size_t)F * kHot) : o;
  k.total = o;
  return k;
}

bool mf_sizes_ok(const esspt_ctx* c, int64_t n_obs, int64_t n_users, int32_t F) {
  if (!(c && n_obs >= 0 && n_obs < (int64_t)INT32_MAX && n_users > 0 && n_users < c->n_rows && F >= 1 && F <= 255 &&
        (int64_t)F * n_users < (int64_t)INT32_MAX))
    return false;
  // The SGD kernels offset item rows and item replica rows by 32-bit float4
  // products (item * K/4, replica row * row stride).
  const int64_t n_items = c->n_rows - n_users;
  return n_items * (c->K / 4) < (int64_t)INT32_MAX &&
         layout_max_item_reps(n_obs, n_items) * dR_stride4(c->K) < (int64_t)INT32_MAX;
}

}  // namespace

namespace esspt {

esspt_status mf_view(esspt_ctx* c, int32_t version, const float** slot, int64_t* n_users, int32_t* K,
                     const int32_t** rec_u, const int32_t** rec_j, const float** rec_D, const int32_t** worker,
                     int64_t* n_obs, int32_t* P, cudaStream_t* st) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (!c->mf) return fail(c, ESSPT_ESTATE, "no MF data loaded (call esspt_mf_load)");
  const int32_t lo = c->clock - 1 - c->s > 0 ? c->clock - 1 - c->s : 0;
  if (version < lo || version > c->clock - 1) return fail(c, ESSPT_EINVAL, "version outside the live window");
  *slot = slot_ptr(c, version);
  *n_users = c->n_users;
  *K = c->K;
  *rec_u = c->rec_u;
  *rec_j = c->rec_j;
  *rec_D = c->rec_D;
  *worker = c->worker;
  *n_obs = c->n_obs;
  *P = c->P;
  *st = c->st;
  return ESSPT_OK;
}

esspt_status mf_fail(esspt_ctx* c, esspt_status code, const char* msg) { return fail(c, code, msg); }

}  // namespace esspt

extern "C" {

size_t esspt_workspace_bytes(const esspt_config* cfg) {
  std::string why;
  if (!config_ok(cfg, &why)) return 0;
  return carve(cfg).total;
}

esspt_status esspt_create(const esspt_config* cfg, void* d_workspace, size_t bytes, esspt_ctx** out) {
  g_create_err.clear();
  if (!out) return g_create_err = "null output pointer", ESSPT_EINVAL;
  *out = nullptr;
  std::string why;
  if (!config_ok(cfg, &why)) return g_create_err = why, ESSPT_EINVAL;
  if (!d_workspace || (reinterpret_cast<uintptr_t>(d_workspace) & 255u) != 0)
    return g_create_err = "workspace must be a 256-byte aligned device pointer", ESSPT_EINVAL;
  const Carve k = carve(cfg);
  if (bytes < k.total) return g_create_err = "workspace too small", ESSPT_ENOSPC;
  esspt_ctx* c = new (std::nothrow) esspt_ctx();
  if (!c) return g_create_err = "out of host memory", ESSPT_ECUDA;
  c->cfg = *cfg;
  c->st = static_cast<cudaStream_t>(cfg->stream);
  c->n_rows = cfg->n_rows;
  c->K = cfg->row_width;
  c->P = cfg->num_workers;
  c->s = cfg->staleness;
  c->nslots = cfg->staleness + 2;
  c->dmax = delay_max(cfg);
  char* w = static_cast<char*>(d_workspace);
  c->ring = reinterpret_cast<float*>(w + k.ring);
  c->v = reinterpret_cast<int32_t*>(w + k.v);
  c->status = reinterpret_cast<uint32_t*>(w + k.status);
  c->thr = reinterpret_cast<uint32_t*>(w + k.thr);
  if (cfg->model == ESSPT_VAP) c->vap_norm = reinterpret_cast<uint32_t*>(w + k.vap);
  if (cfg->model == ESSPT_SSP_ROW) c->rowver = reinterpret_cast<int32_t*>(w + k.rowver);
  // ESSP delay thresholds thr[k] = floor((1-p)^k * 2^32): P(delay >= k) = (1-p)^k.
  std::vector<uint32_t> thr((size_t)c->dmax + 1, 0u);
  double q = 1.0;
  const double fail_p = 1.0 - cfg->essp_p;
  for (int32_t i = 1; i <= c->dmax; ++i) {
    q *= fail_p;
    thr[i] = (uint32_t)std::floor(q * 4294967296.0);
  }
  cudaError_t e = cudaMemcpyAsync(c->thr, thr.data(), thr.size() * sizeof(uint32_t), cudaMemcpyHostToDevice, c->st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->status, 0, sizeof(uint32_t), c->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->st);
  if (e != cudaSuccess) {
    g_create_err = std::string("esspt_create: ") + cudaGetErrorString(e);
    delete c;
    return ESSPT_ECUDA;
  }
  *out = c;
  return ESSPT_OK;
}

esspt_status esspt_destroy(esspt_ctx* c) {
  if (!c) return ESSPT_OK;
  cudaError_t e = cudaStreamSynchronize(c->st);
  delete c;
  return e == cudaSuccess ? ESSPT_OK : ESSPT_ECUDA;
}

const char* esspt_last_error(const esspt_ctx* c) { return c ? c->err.c_str() : g_create_err.c_str(); }

esspt_status esspt_table_init(esspt_ctx* c, const float* rows) {
  if (!c) return ESSPT_EINVAL;
  if (!rows) return fail(c, ESSPT_EINVAL, "null rows");
  ESSPT_CUDA(c, cudaMemcpyAsync(c->ring, rows, (size_t)c->n_rows * c->K * sizeof(float), cudaMemcpyDefault, c->st));
  ESSPT_CUDA(c, cudaMemsetAsync(c->v, 0, sizeof(int32_t) * c->P, c->st));
  if (c->rowver)  // no row cached: every byte 0xff is version -1
    ESSPT_CUDA(c, cudaMemsetAsync(c->rowver, 0xff, sizeof(int32_t) * (size_t)c->P * (size_t)c->n_rows, c->st));
  c->clock = 1;
  c->acc_ready = false;
  c->sched_set = false;
  if (c->chg) {  // every row is version 0's: unchanged since clock 0
    ESSPT_CUDA(c, cudaMemsetAsync(c->chg, 0, sizeof(int32_t) * (size_t)c->n_users, c->st));
    c->copy_all_until = 0;
  }
  if (c->cfg.model != ESSPT_EXTERNAL) return run_schedule(c);
  return ESSPT_OK;
}

esspt_status esspt_set_schedule(esspt_ctx* c, const int32_t* h_v) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (c->cfg.model != ESSPT_EXTERNAL) return fail(c, ESSPT_ESTATE, "set_schedule needs the external model");
  if (!h_v) return fail(c, ESSPT_EINVAL, "null schedule");
  const int32_t lo = c->clock - 1 - c->s > 0 ? c->clock - 1 - c->s : 0;
  for (int32_t p = 0; p < c->P; ++p)
    if (h_v[p] < lo || h_v[p] > c->clock - 1) {
      char buf[160];
      std::snprintf(buf, sizeof buf, "read version %d of worker %d outside [%d, %d] at clock %d", h_v[p], p, lo,
                    c->clock - 1, c->clock);
      return fail(c, ESSPT_ESTALE, buf);
    }
  ESSPT_CUDA(c, cudaMemcpyAsync(c->v, h_v, sizeof(int32_t) * c->P, cudaMemcpyHostToDevice, c->st));
  c->sched_set = true;
  return run_schedule(c);  // device-side check of the same bound
}

esspt_status esspt_get(esspt_ctx* c, int32_t worker, const int32_t* d_row_ids, int64_t n, float* d_out,
                       int32_t* h_version_out) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if ((s = need_schedule(c)) != ESSPT_OK) return s;
  if (worker < 0 || worker >= c->P) return fail(c, ESSPT_EINVAL, "worker out of range");
  if (n < 0 || (n > 0 && (!d_row_ids || !d_out))) return fail(c, ESSPT_EINVAL, "bad row list");
  int32_t* vmin = reinterpret_cast<int32_t*>(c->status) + kGetMinWord;
  if (c->rowver) ESSPT_CUDA(c, cudaMemsetAsync(vmin, 0x7f, sizeof(int32_t), c->st));
  ESSPT_CUDA(c, launch_get(c->ring, c->n_rows, c->K, c->nslots, c->v, worker, d_row_ids, n, d_out, c->status,
                           c->rowver, c->clock, c->s, vmin, c->st));
  if (h_version_out) {
    const int32_t* src = c->rowver ? vmin : c->v + worker;
    ESSPT_CUDA(c, cudaMemcpyAsync(h_version_out, src, sizeof(int32_t), cudaMemcpyDeviceToHost, c->st));
    ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
    if (c->rowver && *h_version_out == 0x7f7f7f7f) *h_version_out = c->clock - 1;  // no row read
  }
  return ESSPT_OK;
}

esspt_status esspt_inc(esspt_ctx* c, int32_t worker, const int32_t* d_row_ids, const float* d_deltas, int64_t n) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (worker < 0 || worker >= c->P) return fail(c, ESSPT_EINVAL, "worker out of range");
  if (n < 0 || (n > 0 && (!d_row_ids || !d_deltas))) return fail(c, ESSPT_EINVAL, "bad row list");
  if ((s = ensure_acc(c)) != ESSPT_OK) return s;
  ESSPT_CUDA(c, launch_inc(slot_ptr(c, c->clock), c->n_rows, c->K, d_row_ids, d_deltas, n, c->status, c->st));
  // INC changes rows the work-list path does not track: copy every idle row
  // until the changed version has gone round the ring.
  c->copy_all_until = std::max(c->copy_all_until, c->clock + c->s + 1);
  return ESSPT_OK;
}

esspt_status esspt_clock(esspt_ctx* c) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if ((s = ensure_acc(c)) != ESSPT_OK) return s;
  return advance(c);
}

esspt_status esspt_poll(esspt_ctx* c) {
  if (!c) return ESSPT_EINVAL;
  uint32_t bits = 0;
  ESSPT_CUDA(c, cudaMemcpyAsync(&bits, c->status, sizeof bits, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  ESSPT_CUDA(c, cudaMemsetAsync(c->status, 0, sizeof(uint32_t), c->st));
  if (bits & kErrStale) return fail(c, ESSPT_ESTALE, "a read version broke the staleness bound");
  if (bits & (kErrRowRange | kErrInput)) return fail(c, ESSPT_EINVAL, "a row id was out of range");
  return ESSPT_OK;
}

esspt_status esspt_read_schedule(esspt_ctx* c, int32_t* h_v, int32_t* h_clock) {
  if (!c) return ESSPT_EINVAL;
  if (h_v) {
    esspt_status s = need_init(c);
    if (s != ESSPT_OK) return s;
    ESSPT_CUDA(c, cudaMemcpyAsync(h_v, c->v, sizeof(int32_t) * c->P, cudaMemcpyDeviceToHost, c->st));
  }
  ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  if (h_clock) *h_clock = c->clock;
  return ESSPT_OK;
}

esspt_status esspt_read_table(esspt_ctx* c, int32_t version, float* out) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (!out) return fail(c, ESSPT_EINVAL, "null output");
  const int32_t lo = c->clock - 1 - c->s > 0 ? c->clock - 1 - c->s : 0;
  if (version < lo || version > c->clock - 1) return fail(c, ESSPT_EINVAL, "version outside the live window");
  ESSPT_CUDA(c, cudaMemcpyAsync(out, slot_ptr(c, version), (size_t)c->n_rows * c->K * sizeof(float),
                                cudaMemcpyDefault, c->st));
  if (is_host_ptr(out)) ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  return ESSPT_OK;
}

size_t esspt_mf_workspace_bytes(const esspt_ctx* c, int64_t n_obs, int64_t n_users, int32_t F) {
  if (!mf_sizes_ok(c, n_obs, n_users, F)) return 0;
  return mf_carve(n_obs, n_users, c->n_rows - n_users, F, c->K, c->rowver != nullptr).total;
}

size_t esspt_mf_scratch_bytes(const esspt_ctx* c, int64_t n_obs, int64_t n_users, int32_t F) {
  if (!mf_sizes_ok(c, n_obs, n_users, F)) return 0;
  return layout_scratch_bytes(n_obs, n_users, c->n_rows - n_users, F);
}

esspt_status esspt_mf_load(esspt_ctx* c, const int32_t* d_i, const int32_t* d_j, const float* d_D,
                           const uint8_t* d_mb, int64_t n_obs, const int32_t* d_worker, int64_t n_users, int32_t F,
                           void* d_ws, size_t bytes, void* d_scratch, size_t scratch_bytes) {
  if (!c) return ESSPT_EINVAL;
  if (!mf_sizes_ok(c, n_obs, n_users, F)) return fail(c, ESSPT_EINVAL, "bad MF sizes");
  if (!d_worker || !d_ws || !d_scratch || (n_obs > 0 && (!d_i || !d_j || !d_D || !d_mb)))
    return fail(c, ESSPT_EINVAL, "null MF pointer");
  if ((reinterpret_cast<uintptr_t>(d_ws) & 255u) || (reinterpret_cast<uintptr_t>(d_scratch) & 255u))
    return fail(c, ESSPT_EINVAL, "MF buffers must be 256-byte aligned");
  const int64_t n_items = c->n_rows - n_users;
  const MfCarve k = mf_carve(n_obs, n_users, n_items, F, c->K, c->rowver != nullptr);
  if (bytes < k.total) return fail(c, ESSPT_ENOSPC, "MF workspace too small");
  if (scratch_bytes < layout_scratch_bytes(n_obs, n_users, n_items, F))
    return fail(c, ESSPT_ENOSPC, "MF scratch too small");
  c->mf = false;
  char* w = static_cast<char*>(d_ws);
  LayoutBuild b{};
  b.i = d_i;
  b.j = d_j;
  b.D = d_D;
  b.mb = d_mb;
  b.worker = d_worker;
  b.n_obs = n_obs;
  b.n_users = n_users;
  b.n_items = n_items;
  b.F = F;
  b.P = c->P;
  b.rec_u = reinterpret_cast<int32_t*>(w + k.rec_u);
  b.rec_j = reinterpret_cast<int32_t*>(w + k.rec_j);
  b.rec_D = reinterpret_cast<float*>(w + k.rec_D);
  b.uoff = reinterpret_cast<int32_t*>(w + k.uoff);
  b.mb_base = reinterpret_cast<int64_t*>(w + k.mb_base);
  b.item_cnt = reinterpret_cast<int32_t*>(w + k.item_cnt);
  b.item_rep = reinterpret_cast<int32_t*>(w + k.item_rep);
  b.rec_dst = reinterpret_cast<int32_t*>(w + k.rec_dst);
  b.chunk = reinterpret_cast<int4*>(w + k.chunk);
  b.chunk_base = reinterpret_cast<int64_t*>(w + k.chunk_base);
  b.heavy = reinterpret_cast<int4*>(w + k.heavy);
  b.heavy_base = reinterpret_cast<int64_t*>(w + k.heavy_base);
  b.max_chunks = k.max_chunks;
  b.light_items = uses_work16(c->K);
  b.hot_item = uses_hot(c->K) ? reinterpret_cast<int32_t*>(w + k.hot_item) : nullptr;
  b.max_heavy = k.max_heavy;
  b.scratch = d_scratch;
  b.scratch_bytes = scratch_bytes;
  b.status = c->status;
  // Validate every index first; nothing is loaded on a bad input.
  uint32_t bits = 0;
  ESSPT_CUDA(c, cudaMemsetAsync(c->status, 0, sizeof(uint32_t), c->st));
  ESSPT_CUDA(c, launch_validate(b, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(&bits, c->status, sizeof bits, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  if (bits & kErrInput) {
    ESSPT_CUDA(c, cudaMemsetAsync(c->status, 0, sizeof(uint32_t), c->st));
    return fail(c, ESSPT_EINVAL, "an MF input index is out of range");
  }
  int32_t* worker = reinterpret_cast<int32_t*>(w + k.worker);
  ESSPT_CUDA(c, cudaMemcpyAsync(worker, d_worker, sizeof(int32_t) * n_users, cudaMemcpyDeviceToDevice, c->st));
  float* dR = reinterpret_cast<float*>(w + k.dR);
  float* dL = reinterpret_cast<float*>(w + k.dL);
  ESSPT_CUDA(c, cudaMemsetAsync(dR, 0, sizeof(float4) * (size_t)k.dR_rows * dR_stride4(c->K), c->st));
  ESSPT_CUDA(c, cudaMemsetAsync(dL, 0, sizeof(float) * (size_t)k.dL_rows * c->K, c->st));
  ESSPT_CUDA(c, cudaMemsetAsync(b.rec_u + n_obs, 0, 16, c->st));
  ESSPT_CUDA(c, cudaMemsetAsync(b.rec_j + n_obs, 0, 16, c->st));
  ESSPT_CUDA(c, cudaMemsetAsync(b.rec_D + n_obs, 0, 16, c->st));
  ESSPT_CUDA(c, build_layout(b, c->st));
  std::vector<int64_t> mbb((size_t)F + 1), chb((size_t)F + 1), hvb((size_t)F + 1);
  ESSPT_CUDA(c, cudaMemcpyAsync(mbb.data(), b.mb_base, sizeof(int64_t) * (F + 1), cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(chb.data(), b.chunk_base, sizeof(int64_t) * (F + 1), cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(hvb.data(), b.heavy_base, sizeof(int64_t) * (F + 1), cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(&bits, c->status, sizeof bits, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  if (chb[F] > k.max_chunks || hvb[F] > k.max_heavy || (bits & kErrInput)) {
    ESSPT_CUDA(c, cudaMemsetAsync(c->status, 0, sizeof(uint32_t), c->st));
    return fail(c, ESSPT_ECUDA, "internal: chunk list overflow");
  }
  c->n_users = n_users;
  c->n_items = n_items;
  c->n_obs = n_obs;
  c->F = F;
  c->rec_u = b.rec_u;
  c->rec_j = b.rec_j;
  c->rec_D = b.rec_D;
  c->uoff = b.uoff;
  if (c->rowver) {
    c->user_slot = reinterpret_cast<int32_t*>(w + k.user_slot);
    c->rec_row = reinterpret_cast<int32_t*>(w + k.rec_row);
  }
  c->item_cnt = b.item_cnt;
  c->worker = worker;
  c->item_rep = b.item_rep;
  c->rec_dst = b.rec_dst;
  c->dR = dR;
  c->dL = dL;
  c->chunk = b.chunk;
  c->heavy = b.heavy;
  c->chg = nullptr;
  c->hot_item = b.hot_item;
  if (uses_work16(c->K)) {
    c->chg = reinterpret_cast<int32_t*>(w + k.chg);
    ESSPT_CUDA(c, cudaMemsetAsync(c->chg, 0, sizeof(int32_t) * (size_t)n_users, c->st));
    // rows changed before this load are not tracked
    c->copy_all_until = c->clock + c->s + 1;
  }
  c->mb_base = mbb;
  c->chunk_base = chb;
  c->heavy_base = hvb;
  c->mf = true;
  return ESSPT_OK;
}

esspt_status esspt_mf_sgd_clock(esspt_ctx* c, float eta, float lambda, int32_t cap, double* d_sq_loss) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (!c->mf) return fail(c, ESSPT_ESTATE, "no MF data loaded (call esspt_mf_load)");
  if ((s = need_schedule(c)) != ESSPT_OK) return s;
  if (cap < 0) return fail(c, ESSPT_EINVAL, "cap must be >= 0");
  const int32_t b = (c->clock - 1) % c->F;
  // Version c is merged from version c-1, or in place when INCs already
  // initialised it during this clock.
  const int32_t slot_out = c->clock % c->nslots;
  const int32_t slot_base = c->acc_ready ? slot_out : (c->clock - 1) % c->nslots;
  SgdArgs a{};
  a.ring = c->ring;
  a.n_rows = c->n_rows;
  a.K = c->K;
  a.n_users = (int32_t)c->n_users;
  a.nslots = c->nslots;
  a.slot_base = slot_base;
  a.slot_out = slot_out;
  a.n_b = (int32_t)(c->mb_base[b + 1] - c->mb_base[b]);
  a.v = c->v;
  a.worker = c->worker;
  a.uoff = c->uoff + (int64_t)b * (c->n_users + 1);
  a.rec_j = c->rec_j + c->mb_base[b];
  a.rec_D = c->rec_D + c->mb_base[b];
  a.rec_dst = c->rec_dst + c->mb_base[b];
  a.item_rep = c->item_rep;
  a.dR = c->dR;
  a.dR_ld = dR_stride4(c->K);
  a.eta = eta;
  a.lambda = lambda;
  a.cap = cap;
  a.sq_loss = d_sq_loss;
  a.chg = c->chg;
  a.clock = c->clock;
  a.hot_item = c->hot_item ? c->hot_item + (int64_t)b * kHot : nullptr;
  a.copy_all_until = c->copy_all_until;
  if (c->rowver) {
    // Row-granular SSP: refresh the rows read this clock; the kernels then
    // take each user's slot and each entry's item ring row from the refresh.
    RowRefreshArgs r{};
    r.rowver = c->rowver;
    r.worker = c->worker;
    r.uoff = a.uoff;
    r.rec_u = c->rec_u + c->mb_base[b];
    r.rec_j = a.rec_j;
    r.n_rows = c->n_rows;
    r.n_users = a.n_users;
    r.n_b = a.n_b;
    r.c = c->clock;
    r.s = c->s;
    r.nslots = c->nslots;
    r.user_slot = c->user_slot;
    r.rec_row = c->rec_row;
    ESSPT_CUDA(c, launch_row_refresh(r, c->st));
    a.row_mode = 1;
    a.user_slot = c->user_slot;
    a.rec_j = c->rec_row;
  }
  const int64_t nch = c->chunk_base[b + 1] - c->chunk_base[b];
  const int64_t nhv = c->heavy_base[b + 1] - c->heavy_base[b];
  if (c->ev_before) ESSPT_CUDA(c, cudaEventRecord(c->ev_before, c->st));
  ChunkArgs ch{};
  ch.a = a;
  ch.chunk = c->chunk + c->chunk_base[b];
  ch.n_chunks = nch;
  ch.dL = c->dL;
  if (uses_work16(c->K)) {
    // Work-list path: users without entries are copied forward; every other
    // user (and every chunk of a heavy user) is one item of the work kernel.
    ESSPT_CUDA(c, launch_user_copy(a, c->st));
    ESSPT_CUDA(c, launch_sgd_work16(ch, c->st));
  } else {
    if (nch > 0) ESSPT_CUDA(c, launch_sgd_chunks(ch, c->st));
    ESSPT_CUDA(c, launch_sgd_users(a, c->st));
  }
  if (nhv > 0) {
    HeavyMergeArgs h{};
    h.ring = c->ring;
    h.n_rows = c->n_rows;
    h.K = c->K;
    h.nslots = c->nslots;
    h.slot_base = slot_base;
    h.slot_out = slot_out;
    h.heavy = c->heavy + c->heavy_base[b];
    h.n_heavy = nhv;
    h.dL = c->dL;
    h.eta = eta;
    h.cap = cap;
    h.chg = c->chg;
    h.clock = c->clock;
    ESSPT_CUDA(c, launch_heavy_merge(h, c->st));
  }
  if (c->ev_after) ESSPT_CUDA(c, cudaEventRecord(c->ev_after, c->st));
  ItemMergeArgs m{};
  m.ring = c->ring;
  m.n_rows = c->n_rows;
  m.K = c->K;
  m.n_users = (int32_t)c->n_users;
  m.n_items = (int32_t)c->n_items;
  m.slot_base = slot_base;
  m.slot_out = slot_out;
  m.item_rep = c->item_rep;
  m.dR = c->dR;
  m.dR_ld = dR_stride4(c->K);
  m.item_cnt = c->item_cnt + (int64_t)b * c->n_items;
  m.eta = eta;
  m.cap = cap;
  // SSP and ESSP schedules need only the previous read versions, so the merge
  // computes them; VAP needs version c complete, so it runs after the merge.
  m.do_schedule = c->cfg.model == ESSPT_SSP_LAZY || c->cfg.model == ESSPT_ESSP_EAGER || c->cfg.model == ESSPT_SSP_ROW;
  m.sched = schedule_args(c, c->clock + 1);
  ESSPT_CUDA(c, launch_item_merge(m, c->st));
  c->acc_ready = true;
  return advance(c, m.do_schedule != 0);
}

size_t esspt_mf_sequential_work_bytes(const esspt_ctx* c) {
  if (!c || !c->mf) return 0;
  return sizeof(float) * (size_t)c->P * (size_t)c->n_items * (size_t)c->K;
}

esspt_status esspt_mf_sgd_clock_sequential(esspt_ctx* c, float eta, float lambda, int32_t cap, double* d_sq_loss,
                                           void* d_work, size_t work_bytes) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (!c->mf) return fail(c, ESSPT_ESTATE, "no MF data loaded (call esspt_mf_load)");
  if ((s = need_schedule(c)) != ESSPT_OK) return s;
  if (cap < 0) return fail(c, ESSPT_EINVAL, "cap must be >= 0");
  if (c->rowver) return fail(c, ESSPT_EINVAL, "the sequential clock reads whole-table versions; not ESSPT_SSP_ROW");
  const size_t need = esspt_mf_sequential_work_bytes(c);
  if (!d_work || (reinterpret_cast<uintptr_t>(d_work) & 15u)) return fail(c, ESSPT_EINVAL, "work must be 16-byte aligned");
  if (work_bytes < need) return fail(c, ESSPT_ENOSPC, "sequential work buffer too small");
  const int32_t b = (c->clock - 1) % c->F;
  SeqArgs a{};
  a.ring = c->ring;
  a.n_rows = c->n_rows;
  a.K = c->K;
  a.n_users = (int32_t)c->n_users;
  a.n_items = (int32_t)c->n_items;
  a.nslots = c->nslots;
  a.slot_out = c->clock % c->nslots;
  a.slot_base = c->acc_ready ? a.slot_out : (c->clock - 1) % c->nslots;
  a.P = c->P;
  a.v = c->v;
  a.worker = c->worker;
  a.uoff = c->uoff + (int64_t)b * (c->n_users + 1);
  a.rec_j = c->rec_j + c->mb_base[b];
  a.rec_D = c->rec_D + c->mb_base[b];
  a.item_cnt = c->item_cnt + (int64_t)b * c->n_items;
  a.mine = static_cast<float*>(d_work);
  a.eta = eta;
  a.lambda = lambda;
  a.cap = cap;
  a.sq_loss = d_sq_loss;
  ESSPT_CUDA(c, cudaMemsetAsync(d_work, 0, need, c->st));
  if (c->ev_before) ESSPT_CUDA(c, cudaEventRecord(c->ev_before, c->st));
  ESSPT_CUDA(c, launch_seq_clock(a, c->st));
  if (c->ev_after) ESSPT_CUDA(c, cudaEventRecord(c->ev_after, c->st));
  // the sequential kernels' row writes are not tracked per row
  c->copy_all_until = std::max(c->copy_all_until, c->clock + c->s + 1);
  c->acc_ready = true;
  return advance(c);
}

esspt_status esspt_mf_objective(esspt_ctx* c, int32_t version, float lambda, double* d_scratch, double* h_sq,
                                double* h_pen) {
  esspt_status s = need_init(c);
  if (s != ESSPT_OK) return s;
  if (!c->mf) return fail(c, ESSPT_ESTATE, "no MF data loaded (call esspt_mf_load)");
  if (!d_scratch || !h_sq || !h_pen) return fail(c, ESSPT_EINVAL, "null pointer");
  const int32_t lo = c->clock - 1 - c->s > 0 ? c->clock - 1 - c->s : 0;
  if (version < lo || version > c->clock - 1) return fail(c, ESSPT_EINVAL, "version outside the live window");
  ESSPT_CUDA(c, launch_objective(slot_ptr(c, version), c->n_users, c->K, c->rec_u, c->rec_j, c->rec_D, c->n_obs,
                                 lambda, d_scratch, c->st));
  double out[2] = {0.0, 0.0};
  ESSPT_CUDA(c, cudaMemcpyAsync(out, d_scratch, sizeof out, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  *h_sq = out[0];
  *h_pen = out[1];
  return ESSPT_OK;
}

esspt_status esspt_mf_minibatch_size(esspt_ctx* c, int32_t b, int64_t* n_b) {
  if (!c) return ESSPT_EINVAL;
  if (!c->mf) return fail(c, ESSPT_ESTATE, "no MF data loaded (call esspt_mf_load)");
  if (b < 0 || b >= c->F || !n_b) return fail(c, ESSPT_EINVAL, "bad minibatch");
  *n_b = c->mb_base[b + 1] - c->mb_base[b];
  return ESSPT_OK;
}

esspt_status esspt_mf_export_minibatch(esspt_ctx* c, int32_t b, int32_t* h_u, int32_t* h_j, float* h_D,
                                       int32_t* h_uoff) {
  int64_t n = 0;
  esspt_status s = esspt_mf_minibatch_size(c, b, &n);
  if (s != ESSPT_OK) return s;
  if (!h_u || !h_j || !h_D || !h_uoff) return fail(c, ESSPT_EINVAL, "null host buffer");
  const int64_t base = c->mb_base[b];
  ESSPT_CUDA(c, cudaMemcpyAsync(h_u, c->rec_u + base, sizeof(int32_t) * n, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(h_j, c->rec_j + base, sizeof(int32_t) * n, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(h_D, c->rec_D + base, sizeof(float) * n, cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaMemcpyAsync(h_uoff, c->uoff + (int64_t)b * (c->n_users + 1), sizeof(int32_t) * (c->n_users + 1),
                                cudaMemcpyDeviceToHost, c->st));
  ESSPT_CUDA(c, cudaStreamSynchronize(c->st));
  return ESSPT_OK;
}

size_t esspt_mf_stage_bytes(const esspt_ctx* c) {
  if (!c || !c->mf) return 0;
  int64_t mx = 0;
  for (int32_t b = 0; b < c->F; ++b) mx = std::max(mx, c->mb_base[b + 1] - c->mb_base[b]);
  return 2 * align256(sizeof(int32_t) * (size_t)mx) + align256(sizeof(int32_t) * (size_t)(c->n_users + 1));
}

esspt_status esspt_mf_stage_minibatch(esspt_ctx* c, int32_t b, const int32_t* h_u, const int32_t* h_j,
                                      const float* h_D, const int32_t* h_uoff, void* d_stage, size_t stage_bytes,
                                      void* stream) {
  int64_t n = 0;
  esspt_status s = esspt_mf_minibatch_size(c, b, &n);
  if (s != ESSPT_OK) return s;
  if (!h_u || !h_j || !h_D || !h_uoff) return fail(c, ESSPT_EINVAL, "null host buffer");
  if (!d_stage || (reinterpret_cast<uintptr_t>(d_stage) & 255u)) return fail(c, ESSPT_EINVAL, "stage must be 256-byte aligned");
  if (stage_bytes < esspt_mf_stage_bytes(c)) return fail(c, ESSPT_ENOSPC, "staging buffer too small");
  cudaStream_t st = stream ? static_cast<cudaStream_t>(stream) : c->st;
  const int64_t base = c->mb_base[b];
  // The values go straight into the layout; the structure only into the
  // staging buffer, where it is compared with the loaded one.
  char* w = static_cast<char*>(d_stage);
  int32_t* su = reinterpret_cast<int32_t*>(w);
  int32_t* sj = reinterpret_cast<int32_t*>(w + align256(sizeof(int32_t) * (size_t)n));
  int32_t* suoff = reinterpret_cast<int32_t*>(w + 2 * align256(sizeof(int32_t) * (size_t)n));
  int32_t* ruoff = c->uoff + (int64_t)b * (c->n_users + 1);
  ESSPT_CUDA(c, cudaMemcpyAsync(c->rec_D + base, h_D, sizeof(float) * n, cudaMemcpyHostToDevice, st));
  ESSPT_CUDA(c, cudaMemcpyAsync(su, h_u, sizeof(int32_t) * n, cudaMemcpyHostToDevice, st));
  ESSPT_CUDA(c, cudaMemcpyAsync(sj, h_j, sizeof(int32_t) * n, cudaMemcpyHostToDevice, st));
  ESSPT_CUDA(c, cudaMemcpyAsync(suoff, h_uoff, sizeof(int32_t) * (c->n_users + 1), cudaMemcpyHostToDevice, st));
  ESSPT_CUDA(c, launch_stage_check(su, sj, suoff, c->rec_u + base, c->rec_j + base, ruoff, n, c->n_users + 1,
                                   c->status, st));
  return ESSPT_OK;
}

esspt_status esspt_set_profile_events(esspt_ctx* c, void* before, void* after) {
  if (!c) return ESSPT_EINVAL;
  if ((before == nullptr) != (after == nullptr)) return fail(c, ESSPT_EINVAL, "give both events or neither");
  c->ev_before = static_cast<cudaEvent_t>(before);
  c->ev_after = static_cast<cudaEvent_t>(after);
  return ESSPT_OK;
}

}  // extern "C"
