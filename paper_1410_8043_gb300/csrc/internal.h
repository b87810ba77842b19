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

// Counter-generator stream ids of the schedule.
constexpr uint64_t kStreamPhase = 101u;
constexpr uint64_t kStreamDelay = 102u;

// Entries per chunk for users whose clock segment exceeds kHeavy entries.
constexpr int32_t kHeavy = 96;
constexpr int32_t kChunk = 64;

struct ScheduleArgs {
  int32_t* v;              // [P] read versions (in: v(c-1), out: v(c))
  uint32_t* status;        // latched error bits
  const uint32_t* thr;     // [dmax+1] ESSP delay thresholds, thr[k] = floor((1-p)^k 2^32)
  int32_t P, c, s, model, phased, dmax;
  uint64_t seed;
};

// Fused MF-SGD clock over the users of one minibatch.
struct SgdArgs {
  float* ring;             // (s+2) * n_rows * K
  int64_t n_rows;
  int32_t K;
  int32_t n_users;
  int32_t nslots;          // s + 2
  int32_t slot_base;       // slot the L rows are merged from (c-1, or c if INCs happened)
  int32_t slot_out;        // slot of version c
  const int32_t* v;        // [P] read versions
  const int32_t* worker;   // [n_users]
  const int32_t* uoff;     // [n_users+1] entry offsets of minibatch b, relative to its base
  const int32_t* rec_j;    // item of each entry (minibatch base applied)
  const float* rec_D;      // value of each entry
  const int32_t* item_cnt; // [M] entries per item in minibatch b
  float eta, lambda;
  int32_t cap;
  double* sq_loss;         // optional
};

struct ChunkArgs {
  SgdArgs a;
  const int32_t* chunk_user;   // [n_chunks]
  const int32_t* chunk_begin;  // relative to the minibatch base
  const int32_t* chunk_end;
  int64_t n_chunks;
};

// Launchers (return the launch error, if any).
cudaError_t launch_schedule(const ScheduleArgs& a, cudaStream_t st);
cudaError_t launch_copy_rows(float* dst, const float* src, int64_t n_floats, cudaStream_t st);
cudaError_t launch_get(const float* ring, int64_t n_rows, int32_t K, int32_t nslots, const int32_t* v,
                       int32_t worker, const int32_t* ids, int64_t n, float* out, uint32_t* status,
                       cudaStream_t st);
cudaError_t launch_inc(float* slot, int64_t n_rows, int32_t K, const int32_t* ids, const float* d, int64_t n,
                       uint32_t* status, cudaStream_t st);
cudaError_t launch_sgd_users(const SgdArgs& a, cudaStream_t st);
cudaError_t launch_sgd_chunks(const ChunkArgs& a, cudaStream_t st);
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
  int32_t* uoff;        // [F][n_users+1]
  int64_t* mb_base;     // [F+1]
  int32_t* item_cnt;    // [F][n_items]
  int32_t* chunk_user;  // [max_chunks]
  int32_t* chunk_begin;
  int32_t* chunk_end;
  int64_t* chunk_base;  // [F+1]
  int64_t max_chunks;
  // scratch
  void* scratch;
  size_t scratch_bytes;
  uint32_t* status;
};

size_t layout_scratch_bytes(int64_t n_obs, int64_t n_users, int32_t F);
int64_t layout_max_chunks(int64_t n_obs, int32_t F);
cudaError_t build_layout(const LayoutBuild& b, cudaStream_t st);
cudaError_t launch_validate(const LayoutBuild& b, cudaStream_t st);

}  // namespace esspt
