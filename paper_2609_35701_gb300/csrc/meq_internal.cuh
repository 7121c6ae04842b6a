// Internal declarations shared by the MeqMuon CUDA sources (not part of the ABI).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <utility>

namespace meq {

// ------------------------------------------------------------ error codes
// Written (first writer wins) to the state's device error word.
enum DevErr : int {
  DEV_OK = 0,
  DEV_TIMEOUT_PRODUCER = 0x101,  // TMA warp waited too long for a free stage
  DEV_TIMEOUT_MMA_FULL = 0x102,  // MMA warp waited too long for a loaded stage
  DEV_TIMEOUT_MMA_TMEM = 0x103,  // MMA warp waited too long for a free accumulator
  DEV_TIMEOUT_EPI = 0x104,       // epilogue waited too long for an accumulator
  DEV_TIMEOUT_DRAIN = 0x105,     // waiting for in-flight copies / MMAs at exit
  DEV_TIMEOUT_SCHED_PUT = 0x106, // tile scheduler waited too long for a free slot of the tile ring
  DEV_TIMEOUT_SCHED_TAKE = 0x107,// a role waited too long for its next tile index
  DEV_TIMEOUT_TEST = 0x1FF,      // the wait-timeout self test
};

constexpr int kMaxGroups = 8;        // shape groups per GEMM launch
constexpr int kNsEpilogueWarps = 8;  // epilogue warps per CTA of the NS GEMM kernel

// U of the hidden weights is stored as fp16(kUScale * U). Every entry of U
// is bounded by its largest singular value, which the quintic keeps below
// about 1.25, so the scaled values stay far from fp16's overflow while
// entries down to 4e-9 keep fp16's full 11-bit precision.
constexpr float kUScale = 16384.0f;

// Per-matrix metadata (device copy built at init).
struct MatInfo {
  int64_t m, n;          // W layout: rows, cols
  int64_t s, l;          // oriented NS shape: s = min(m, n), l = max(m, n)
  int32_t trans;         // 1 when the NS layout is W^T (m > n)
  int32_t group;         // shape group (hidden weights)
  int32_t kind;          // 0 hidden, 1 remaining 2D (two-sided), 2 vector
  int32_t pad_;
  int64_t gidx;          // index inside its group
  int64_t mom_off;       // float offset of B in the momentum slab
  int64_t u_off;         // element offset of U in the fp16 U slab (row stride un)
  int64_t un;            // U row stride: cols rounded up to 8 (hidden), cols (others)
  int64_t vec_off;       // float offset of r (m), c (n) and scale (max(m, n))
  int64_t chunk_begin;   // first apply chunk (all kinds)
  int64_t hchunk_begin;  // first momentum-and-norm chunk (hidden weights only)
  int64_t rblk_begin;    // first 8-row block of the row pass (remaining 2D and vectors)
  int64_t slab_begin;    // first row slab of the column pass (remaining 2D only)
  int64_t tile_begin;    // first cast tile (hidden weights only)
  int64_t xblk_begin;    // first momentum-and-X_0 block (hidden weights only)
  int64_t rpart_off;     // float offset of NS-row partial sums of squares [2 * ceil(l/256)][s]
  int64_t cpart_off;     // float offset of column partial sums of squares: NS columns
                         // [ceil(s/32)][l] (hidden) or normalised columns [slabs][n] (remaining 2D)
};

// Per-group metadata for the elementwise kernels.
struct GroupInfo {
  int64_t s, l, lp, sp;  // shape and padded row strides (elements)
  int64_t count;
  void* x0;              // X-hat buffer 0: [count][s][lp] 16-bit
  float alpha0;          // power-of-two storage scale of X_0 (separate cast pass)
  int64_t mbase;         // offset of the group's matrices in the inverse-norm array
};

// Values that change per step (uploaded before each step).
struct StepScalars {
  float lr, mu, wd, eps;
  float rho, tie_atol;
  int32_t nesterov;
  int32_t rule;          // meq_update_rule
};

// --------------------------------------------------------------- GEMM side
enum GemmMode : int { MODE_GRAM = 0, MODE_POLY = 1, MODE_XUPD = 2, MODE_XLAST = 3 };

struct GemmGroup {
  CUtensorMap tmA;        // A operand (K-major), box {64, 128, 1}
  CUtensorMap tmB;        // B operand: K-major box {64, 256, 1} or MN-major box {64, 64, 1}
  CUtensorMap tmO;        // GRAM / POLY / XUPD: the 16-bit output (A, P or X next) for TMA stores,
                          // box {32, 32, 1}, 64-byte swizzle (the epilogue's staging layout)
  int32_t M, N, K;        // output rows, output cols, contraction
  int32_t count;          // matrices in the group
  int32_t tiles_m, tiles_n;
  int32_t tiles_per_mat;  // tiles_m * tiles_n, or the upper-triangle count when sym
  int32_t band;           // dense outputs: tile rows per band of the tile order
  int32_t tile_begin;     // first tile of this group in the launch
  int32_t sym;            // 1: symmetric s x s output (upper-triangle tiles, mirrored stores)
  int32_t trans;          // XLAST: 1 when the weight is the transpose of the NS layout
  float scale;            // GRAM: 1/alpha^2; XUPD: alpha_next/alpha; XLAST: 1/alpha
  const float* minv;      // iteration 0 with X_0 unnormalised: 1/||H||_F per matrix of the group
  int32_t minv_pow;       // epilogue scale *= minv^minv_pow (0, 1 or 2)
  int32_t out_fp16;       // 16-bit format of the output (1 = fp16, 0 = bf16)
  int32_t aux_fp16;       // POLY: 16-bit format of the A it reads in the epilogue
  void* out;              // XUPD: 16-bit X next; XLAST: fp16(kUScale U) in the weight's layout
  int64_t out_ld;         // XUPD / XLAST: output row stride in bytes
  int64_t out_mstride;    // XUPD / XLAST: output matrix stride in bytes
  const void* aux;        // POLY: 16-bit A
  int64_t aux_ld;         // bytes
  int64_t aux_mstride;    // bytes
  float* rpart;           // XLAST: NS-row partial sums of squares, [count][2 * tiles_n][M]
  float* cpart;           // XLAST: NS-column partial sums of squares, [count][ceil(M/32)][N]
  int32_t mode;           // GemmMode of the product
  uint32_t idesc;         // tcgen05 instruction descriptor
  int32_t b_mn_major;     // 1: B operand tile is MN-major (XUPD)
  int32_t tma_out;        // 1: the output leaves by TMA stores through tmO (else 16-byte thread stores)
};

// One GEMM launch: one product's shape groups, taken as one tile queue in
// group order.
struct GemmParams {
  GemmGroup g[kMaxGroups];
  int32_t ngroups;
  int32_t total_tiles;
  int32_t reverse;         // 1: tiles are taken in reverse order (alternates between launches)
  float ca, cb, cc;        // NS coefficients
  int* err;                // device error word
  int* sched;              // tile queue: [0] tiles handed out beyond the first wave, [1] units done;
                           // zero between launches (the last unit to finish resets both)
  int32_t debug_skip_load; // tests: the first pair's leader skips its first stage's loads
  unsigned long long timeout_ns;
};

// Programmatic dependent launch: a kernel lets the next one in the stream be
// scheduled as soon as it starts, and waits for its predecessor's results
// only where it first needs them.
__device__ __forceinline__ void pdl_allow_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait_predecessor() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Launch with the programmatic-serialization attribute (and a cluster shape
// when cluster_x > 1).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, int cluster_x,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  if (cluster_x > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = static_cast<unsigned>(cluster_x);
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Launchers (defined in the .cu files).
cudaError_t prepare_ns_gemm();  // sets the kernel's dynamic shared-memory limit (per device)
cudaError_t launch_ns_gemm(const GemmParams& p, int grid, int pair, cudaStream_t st);  // pair: 1 or 2 CTAs per tile
int ns_gemm_smem_bytes(int pair);

// Row / column statistics of one fp32 matrix (Eqs. (7), (8), (11)) with
// caller-given scratch of row_col_stats_scratch_floats(rows, cols) floats;
// frob = 1 describes U / ||U||_F instead of U. On failure *failed names the
// launch.
int64_t row_col_stats_scratch_floats(int64_t rows, int64_t cols);
cudaError_t launch_row_col_stats(const float* U, int64_t rows, int64_t cols, float eps, float tie_atol, int frob,
                                 float* scratch, float* r, float* c, double* gammas, int* direction, cudaStream_t st,
                                 const char** failed);

// Error text of the last failed call made without a state (meq_last_error(NULL)).
void set_global_error(const std::string& msg);

}  // namespace meq
