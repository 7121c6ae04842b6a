// Launch interface of the bandwidth-bound kernels (internal).
#pragma once

#include "meq_internal.cuh"

namespace meq {

constexpr int64_t kChunk = 4096;   // elements per momentum / apply block
constexpr int kCastTile = 64;      // X_0 cast tile (64 x 64 of W)
constexpr int kFinThreads = 1024;  // finalize block size
constexpr int kColSlab = 128;      // rows per block of the remaining-2D column pass

struct MatStats {
  double gamma_r;
  double gamma_c;
  int32_t direction;  // 0 = row (N_r), 1 = column (N_c), 2 = two-sided, 3 = vector, 4 = Eq. (6) shape factor
  int32_t pad;
};

// Device pointers and sizes the elementwise launchers need.
struct LaunchCtx {
  const MatInfo* mats;
  int nmat;
  const GroupInfo* groups;
  float* mom;
  const float* const* grads;
  float* const* params;
  const StepScalars* sc;
  float* partials;
  unsigned int* counters;
  float* x0scale;
  float* ginv;           // 1 / ||H||_F per hidden matrix, ordered group by group
  uint16_t* uslab;       // U of every hidden matrix, fp16, scaled by kUScale
  float* parts;          // NS-row and NS-column partial sums of squares
  float* rvec;
  float* cvec;
  float* svec;           // hidden: scale of the chosen side; others: 1 / row RMS
  float* tvec;           // remaining 2D: 1 / column RMS of the row-normalised momentum
  MatStats* stats;
  unsigned long long* dircount;  // per entry: Eq. (11) row choices, column choices
  int* nonfinite;                // 1 + index of the first entry whose momentum had a non-finite norm, or 0
  int64_t total_chunks, total_hchunks, total_tiles, total_rblks, total_slabs, total_xblks;
  int n_hidden;
};

constexpr int KIND_HIDDEN = 0, KIND_TWO_SIDED = 1, KIND_VECTOR = 2;

cudaError_t launch_momentum_norm(const LaunchCtx& L, cudaStream_t st);
cudaError_t launch_momentum_x0(const LaunchCtx& L, cudaStream_t st);  // fused momentum + bf16 X_0
cudaError_t launch_x0norm(const LaunchCtx& L, cudaStream_t st);       // 1 / ||H||_F from its partials
cudaError_t launch_rows(const LaunchCtx& L, cudaStream_t st);      // remaining 2D + vectors
cudaError_t launch_colpart(const LaunchCtx& L, cudaStream_t st);   // remaining 2D
cudaError_t launch_cast_x0(const LaunchCtx& L, bool fp16, cudaStream_t st);
cudaError_t launch_stats(const LaunchCtx& L, cudaStream_t st);  // finalize of the fused statistics
cudaError_t launch_apply(const LaunchCtx& L, cudaStream_t st);
// U~ of entry mi (the update apply_kernel applies) into dst (device, M.m x M.n fp32).
cudaError_t launch_update(const LaunchCtx& L, const MatInfo& M, int mi, float* dst, cudaStream_t st);
cudaError_t launch_wait_selftest(const int* flag, int* err, unsigned long long timeout_ns, cudaStream_t st);

}  // namespace meq
