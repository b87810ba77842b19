// Library-internal declarations shared by the esspt .cu translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "esspt.h"

namespace esspt {

// Latched device error bits (status word in the workspace).
enum : uint32_t {
  kErrStale = 1u,     // a read version broke the staleness bound
  kErrRowRange = 2u,  // a GET/INC row id outside [0, n_rows)
  kErrInput = 4u,     // an MF input index outside its range
};

// Word of the context's status block (after the error bits) that receives
// the oldest row version a row-granular GET read.
constexpr int kGetMinWord = 16;

// Counter-generator stream ids of the schedule.
constexpr uint64_t kStreamPhase = 101u;
constexpr uint64_t kStreamDelay = 102u;

// Users with more than kHeavy entries in a minibatch are split in chunks of
// kChunk entries, processed apart from the per-user kernel.
constexpr int32_t kHeavy = 96;
constexpr int32_t kChunk = 64;
// Replica accumulators: an item gets one delta row per kItemRep entries
// (largest minibatch count, rounded up to a power of two); a heavy user one
// per kUserRep chunks.  Replicas spread the fp32 reductions of popular rows
// over many L2 addresses and keep each partial sum short.
#ifndef ESSPT_ITEM_REP
#define ESSPT_ITEM_REP 2048
#endif
constexpr int32_t kItemRep = ESSPT_ITEM_REP;
constexpr int32_t kUserRep = 64;
#ifndef ESSPT_MAX_REP
#define ESSPT_MAX_REP 64
#endif
constexpr int32_t kMaxRep = ESSPT_MAX_REP;

// Rows of 36..64 values (9..16 float4 slices) take the work-list path: every
// user with 1..kHeavy entries in a minibatch is one work item beside the
// chunks of the heavy users, processed by one kernel, and the users without
// entries are copied forward by a streaming kernel.
inline bool uses_work16(int32_t K) { return K > 32 && K <= 64; }
// Work-list path: the kHot items with the most entries of each minibatch have
// their updates summed per warp in shared memory and added to the replica
// rows once per warp instead of once per entry (0 = off).  An entry of hot
// slot h carries rec_dst = -1 - h.
#ifndef ESSPT_W16_HOT
#define ESSPT_W16_HOT 2
#endif
constexpr int kHot = ESSPT_W16_HOT;
inline bool uses_hot(int32_t K) { return kHot > 0 && uses_work16(K); }
// Resident blocks per SM that the launches of the forward copy and of the
// work kernel ask for (the occupancy limit caps the second).
constexpr int kCopyBlocksPerSm = 8;
constexpr int kWorkBlocksPerSm = 8;

// Row stride (in float4) of the item delta replicas: K rounded up to a whole
// number of 32-byte sectors, so that a row's reductions touch the fewest sectors.
inline int32_t dR_stride4(int32_t K) { return ((K + 7) / 8) * 2; }

struct ScheduleArgs {
  int32_t* v;              // [P] read versions (in: v(c-1), out: v(c))
  uint32_t* status;        // latched error bits
  const uint32_t* thr;     // [dmax+1] ESSP delay thresholds, thr[k] = floor((1-p)^k 2^32)
  const uint32_t* vap_norm;  // [s+1] VAP: bits of |X[c-1] - X[c-1-k]|_inf (fp32, >= 0)
  double vap_bound;        // VAP: v0 / sqrt(c)
  int32_t P, c, s, model, phased, dmax;
  uint64_t seed;
};

// One clock of MF-SGD over the users of minibatch b.
struct SgdArgs {
  float* ring;              // (s+2) * n_rows * K
  int64_t n_rows;
  int32_t K;
  int32_t n_users;
  int32_t nslots;           // s + 2
  int32_t slot_base;        // slot merged from (c-1, or c if INCs already landed there)
  int32_t slot_out;         // slot of version c
  int32_t n_b;              // entries of minibatch b
  const int32_t* v;         // [P] read versions
  const int32_t* worker;    // [n_users]
  const int32_t* uoff;      // [n_users+1] entry offsets of minibatch b (relative)
  const int32_t* rec_j;     // item of each entry of minibatch b; in row mode the ring row
                            // (slot * n_rows + N + item) of the item's cached version
  const float* rec_D;       // value of each entry of minibatch b
  const int32_t* rec_dst;   // replica row in dR that each entry's item update adds into
  const int32_t* item_rep;  // [M+1] prefix of extra replicas: replica 0 of item j is row j of dR,
                            // replica r > 0 row M + item_rep[j] + r - 1
  float* dR;                // item delta replicas (all zero between clocks)
  int32_t dR_ld;            // float4 per dR row (K rounded up to whole 32-byte sectors)
  float eta, lambda;
  int32_t cap;
  double* sq_loss;          // optional
  int32_t row_mode;         // row-granular SSP: per-user slots and per-entry ring rows
  const int32_t* user_slot; // [n_users] row mode: ring slot of each user's cached row
  // Work-list path: chg[u] = last clock that changed user row u (written with
  // every user row that changes); an idle row whose slot already holds its
  // current value is not copied forward: clock > copy_all_until and
  // clock - chg[u] >= nslots (unchanged over the whole ring).
  int32_t* chg;
  int32_t clock, copy_all_until;
  const int32_t* hot_item;  // [kHot] work-list path: item of each hot slot of minibatch b, -1 if unused
};

// Chunks of heavy users: x = user, y = begin, z = end (relative), w = replica row in dL.
// On the work-list path a user with 1..kHeavy entries is one item with w = -1
// (its row of version c is written directly).
struct ChunkArgs {
  SgdArgs a;
  const int4* chunk;
  int64_t n_chunks;
  float* dL;                // heavy-user delta replicas (all zero between clocks)
};

// Merge of heavy user rows: x = user, y = first replica row, z = replicas, w = entries.
struct HeavyMergeArgs {
  float* ring;
  int64_t n_rows;
  int32_t K, nslots, slot_base, slot_out;
  const int4* heavy;
  int64_t n_heavy;
  float* dL;
  float eta;
  int32_t cap;
  int32_t* chg;             // work-list path: set chg[user] = clock (see SgdArgs)
  int32_t clock;
};

// Clock() merge of the item rows: R^c_j = R^base_j + eta s_j sum of replicas.
struct ItemMergeArgs {
  float* ring;
  int64_t n_rows;
  int32_t K, n_users, n_items, slot_base, slot_out;
  const int32_t* item_rep;
  float* dR;
  int32_t dR_ld;
  const int32_t* item_cnt;  // [M] entries per item in minibatch b
  float eta;
  int32_t cap;
  int32_t do_schedule;      // also compute the next clock's read versions
  ScheduleArgs sched;
};

// Launchers (return the launch error, if any).
cudaError_t launch_schedule(const ScheduleArgs& a, cudaStream_t st);
// VAP: norm[k] = bits of max |X[c-1] - X[c-1-k]| over the table, k = 1..kmax
// (norm must be zero on entry; a NaN difference gives +inf).
cudaError_t launch_vap_norms(const float* ring, int64_t slot_floats, int32_t nslots, int32_t c, int32_t kmax,
                             uint32_t* norm, cudaStream_t st);
cudaError_t launch_copy_rows(float* dst, const float* src, int64_t n_floats, cudaStream_t st);
// GET; with rowver non-null (row-granular SSP at clock c) each row is read at
// the worker's cached version, refreshed to c-1 first where it is missing or
// older than c-1-s, and *vmin receives the oldest version read.
cudaError_t launch_get(const float* ring, int64_t n_rows, int32_t K, int32_t nslots, const int32_t* v,
                       int32_t worker, const int32_t* ids, int64_t n, float* out, uint32_t* status,
                       int32_t* rowver, int32_t c, int32_t s, int32_t* vmin, cudaStream_t st);
cudaError_t launch_inc(float* slot, int64_t n_rows, int32_t K, const int32_t* ids, const float* d, int64_t n,
                       uint32_t* status, cudaStream_t st);
cudaError_t launch_sgd_users(const SgdArgs& a, cudaStream_t st);
// Row-granular SSP, before the SGD kernels of clock c: refresh the cached
// version of every row a worker reads (rowver[p * n_rows + r], -1 = never
// read) to c-1 where it is missing or older than c-1-s, and write the ring
// slot of each user's row and the ring row of each entry's item row.
struct RowRefreshArgs {
  int32_t* rowver;
  const int32_t* worker;   // [n_users]
  const int32_t* uoff;     // [n_users+1] of minibatch b
  const int32_t* rec_u;    // [n_b] user of each entry
  const int32_t* rec_j;    // [n_b] item of each entry
  int64_t n_rows;
  int32_t n_users, n_b, c, s, nslots;
  int32_t* user_slot;      // out [n_users]
  int32_t* rec_row;        // out [n_b]
};
cudaError_t launch_row_refresh(const RowRefreshArgs& a, cudaStream_t st);

// Sequential (read-my-writes) SGD of one clock over minibatch b: the users
// kernel writes every user row of version c, the item merge every item row.
struct SeqArgs {
  float* ring;
  int64_t n_rows;
  int32_t K, n_users, n_items, nslots, slot_base, slot_out, P;
  const int32_t* v;         // [P] read versions
  const int32_t* worker;    // [n_users]
  const int32_t* uoff;      // [n_users+1] entry offsets of minibatch b
  const int32_t* rec_j;     // item of each entry of minibatch b
  const float* rec_D;
  const int32_t* item_cnt;  // [n_items] entries per item in minibatch b (hot-row cap)
  float* mine;              // [P][n_items][K] each worker's item changes this clock (zero on entry)
  float eta, lambda;
  int32_t cap;
  double* sq_loss;          // optional
};
cudaError_t launch_seq_clock(const SeqArgs& a, cudaStream_t st);
cudaError_t launch_sgd_chunks(const ChunkArgs& a, cudaStream_t st);
// Work-list path (uses_work16): the items of minibatch b (light users and
// heavy-user chunks) and the forward copy of the users without entries.
cudaError_t launch_sgd_work16(const ChunkArgs& a, cudaStream_t st);
cudaError_t launch_user_copy(const SgdArgs& a, cudaStream_t st);
cudaError_t launch_heavy_merge(const HeavyMergeArgs& a, cudaStream_t st);
cudaError_t launch_item_merge(const ItemMergeArgs& a, cudaStream_t st);
cudaError_t launch_objective(const float* slot, int64_t n_users, int32_t K, const int32_t* rec_u,
                             const int32_t* rec_j, const float* rec_D, int64_t n_obs, float lambda,
                             double* out2, cudaStream_t st);

// MF layout build (setup, not per clock).
struct LayoutBuild {
  const int32_t* i;
  const int32_t* j;
  const float* D;
  const uint8_t* mb;
  const int32_t* worker;
  int64_t n_obs, n_users, n_items;
  int32_t F, P;
  // outputs (persistent)
  int32_t* rec_u;
  int32_t* rec_j;
  float* rec_D;
  int32_t* rec_dst;     // replica row of each entry's item update
  int32_t* uoff;        // [F][n_users+1]
  int64_t* mb_base;     // [F+1]
  int32_t* item_cnt;    // [F][n_items]
  int32_t* item_rep;    // [n_items+1]
  int4* chunk;          // [max_chunks]
  int64_t* chunk_base;  // [F+1]
  int4* heavy;          // [max_heavy]
  int64_t* heavy_base;  // [F+1]
  int64_t max_chunks, max_heavy;
  bool light_items;     // also list every user with 1..kHeavy entries (work-list path)
  int32_t* hot_item;    // [F][kHot] work-list path with kHot > 0: the hot items of each minibatch
  // scratch
  void* scratch;
  size_t scratch_bytes;
  uint32_t* status;
};

size_t layout_scratch_bytes(int64_t n_obs, int64_t n_users, int64_t n_items, int32_t F);
int64_t layout_max_chunks(int64_t n_obs, int32_t F, int64_t n_users, bool light_items);
int64_t layout_max_heavy(int64_t n_obs, int32_t F);
int64_t layout_max_item_reps(int64_t n_obs, int64_t n_items);
int64_t layout_max_user_reps(int64_t n_obs);
cudaError_t build_layout(const LayoutBuild& b, cudaStream_t st);
cudaError_t launch_validate(const LayoutBuild& b, cudaStream_t st);
// Staged minibatch check: su/sj (n entries) and suoff (n_off offsets) against
// the resident ru/rj/ruoff; a difference latches kErrInput.
cudaError_t launch_stage_check(const int32_t* su, const int32_t* sj, const int32_t* suoff, const int32_t* ru,
                               const int32_t* rj, const int32_t* ruoff, int64_t n, int64_t n_off, uint32_t* status,
                               cudaStream_t st);

// Read-only view of a context's loaded MF entries and of table version
// `version` (checked against the live window), for entry points defined in
// other translation units; and the context's error setter.
esspt_status mf_view(esspt_ctx* ctx, int32_t version, const float** slot, int64_t* n_users, int32_t* K,
                     const int32_t** rec_u, const int32_t** rec_j, const float** rec_D, const int32_t** worker,
                     int64_t* n_obs, int32_t* P, cudaStream_t* st);
esspt_status mf_fail(esspt_ctx* ctx, esspt_status code, const char* msg);

}  // namespace esspt
