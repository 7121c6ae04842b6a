// Bandwidth-bound kernels of the MeqMuon step (everything except the NS GEMMs).
//
//   momentum_norm : B <- mu B + G (Eq. (10)) in place over every matrix, with
//                   deterministic per-chunk partial sums of the squared NS
//                   input; the last chunk of each matrix reduces them into the
//                   X_0 scale alpha0 / ||H||_F of Eq. (5).
//   cast_x0       : X-hat_0 = 16-bit(alpha0 H / ||H||_F) in the oriented NS
//                   layout (transposed through shared memory for tall W).
//   finalize      : r, c (Eq. (7)) from the partial sums of squares the last
//                   NS epilogue wrote, gamma_r, gamma_c (Eq. (8)), the
//                   direction (Eq. (11)) and the scale vector of Eq. (9).
//   rows, colpart : momentum, row and column statistics of the remaining 2D
//                   parameters and vectors (Eqs. (12), (13)).
//   apply         : W <- (1 - lr wd) W - rho lr U~ (Eq. (14)).
#include <algorithm>

#include "meq_elementwise.cuh"

namespace meq {
namespace {

constexpr int kThreads = 256;

// Largest i with begin(i) <= key; begin is nondecreasing in i. Entries that
// own no work of the enumeration share their begin with the next entry (or
// lie past the end), so they are never selected.
__device__ __forceinline__ int find_mat(const MatInfo* mats, int nmat, int64_t key, int which) {
  int lo = 0, hi = nmat - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    const int64_t b = which == 0   ? mats[mid].chunk_begin
                      : which == 1 ? mats[mid].tile_begin
                      : which == 2 ? mats[mid].hchunk_begin
                      : which == 3 ? mats[mid].rblk_begin
                      : which == 4 ? mats[mid].slab_begin
                                   : mats[mid].xblk_begin;
    if (b <= key) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Row i and column j of flat element e of a matrix with n columns. Every
// model weight has fewer than 2^32 elements, where a 32-bit division is
// several times cheaper than a 64-bit one (measured: about 0.5% of the
// Llama-130M and 350M steps); small32 is uniform over a block, so the
// branch does not diverge.
__device__ __forceinline__ void row_col(int64_t e, int64_t n, bool small32, int64_t& i, int64_t& j) {
  if (small32) {
    const uint32_t eu = static_cast<uint32_t>(e), nu = static_cast<uint32_t>(n);
    const uint32_t iu = eu / nu;
    i = iu;
    j = eu - iu * nu;
  } else {
    i = e / n;
    j = e - i * n;
  }
}

__device__ __forceinline__ float block_sum_f32(float v, float* sh) {
  const unsigned FULL = 0xffffffffu;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) sh[w] = v;
  __syncthreads();
  float r = 0.f;
  if (threadIdx.x == 0) {
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) r += sh[i];
    sh[0] = r;
  }
  __syncthreads();
  return sh[0];
}

// ------------------------------------------------------------- momentum + norm
__global__ void __launch_bounds__(kThreads) momentum_norm_kernel(const MatInfo* __restrict__ mats, int nmat,
                                                                 const GroupInfo* __restrict__ groups,
                                                                 float* __restrict__ mom,
                                                                 const float* const* __restrict__ grads,
                                                                 const StepScalars* __restrict__ sc,
                                                                 float* __restrict__ partials,
                                                                 unsigned int* __restrict__ counters,
                                                                 float* __restrict__ x0scale,
                                                                 int* __restrict__ nonfinite) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  __shared__ float shf[32];
  __shared__ int is_last;
  const int64_t chunk = blockIdx.x;
  const int mi = find_mat(mats, nmat, chunk, 2);
  const MatInfo& M = mats[mi];
  const int64_t numel = M.m * M.n;
  const int64_t e0 = (chunk - M.hchunk_begin) * kChunk;
  const int64_t e1 = min(e0 + kChunk, numel);
  const float mu = sc->mu;
  const int nesterov = sc->nesterov;
  float* B = mom + M.mom_off;
  const float* G = grads[mi];
  float ss = 0.f;
  // numel of a matrix need not be a multiple of 4: vector body + scalar tail.
  const int64_t vec_end = e0 + ((e1 - e0) & ~int64_t(3));
  for (int64_t e = e0 + 4 * threadIdx.x; e < vec_end; e += 4 * kThreads) {
    const float4 g = __ldcs(reinterpret_cast<const float4*>(G + e));
    float4 b = *reinterpret_cast<const float4*>(B + e);
    b.x = fmaf(mu, b.x, g.x);
    b.y = fmaf(mu, b.y, g.y);
    b.z = fmaf(mu, b.z, g.z);
    b.w = fmaf(mu, b.w, g.w);
    *reinterpret_cast<float4*>(B + e) = b;
    if (nesterov) {
      const float hx = fmaf(mu, b.x, g.x), hy = fmaf(mu, b.y, g.y), hz = fmaf(mu, b.z, g.z), hw = fmaf(mu, b.w, g.w);
      ss += hx * hx + hy * hy + hz * hz + hw * hw;
    } else {
      ss += b.x * b.x + b.y * b.y + b.z * b.z + b.w * b.w;
    }
  }
  for (int64_t e = vec_end + threadIdx.x; e < e1; e += kThreads) {
    const float g = G[e];
    const float b = fmaf(mu, B[e], g);
    B[e] = b;
    const float h = nesterov ? fmaf(mu, b, g) : b;
    ss += h * h;
  }
  const float part = block_sum_f32(ss, shf);
  if (threadIdx.x == 0) {
    partials[chunk] = part;
    __threadfence();
    const unsigned int nchunks = static_cast<unsigned int>((numel + kChunk - 1) / kChunk);
    const unsigned int prev = atomicAdd(&counters[mi], 1u);
    is_last = (prev + 1 == nchunks);
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  // Last chunk of this matrix: fixed-order fp32 reduction of its partials
  // (fp32 throughout: this GPU's fp64 rate is a small fraction of its fp32 rate).
  const int64_t nchunks = (numel + kChunk - 1) / kChunk;
  float acc = 0.f;
  for (int64_t c = threadIdx.x; c < nchunks; c += kThreads) acc += __ldcg(partials + M.hchunk_begin + c);
  const float total = block_sum_f32(acc, shf);
  if (threadIdx.x == 0) {
    const float nrm = sqrtf(total);
    if (!isfinite(total)) atomicCAS(nonfinite, 0, mi + 1);  // first non-finite entry, 1-based
    // Zero input: U = 0 (Eq. (5) is defined for a nonzero input only).
    x0scale[mi] = nrm > 0.f ? groups[M.group].alpha0 / nrm : 0.f;
    counters[mi] = 0u;
  }
}

__device__ __forceinline__ uint2 pack4_bf16(float a, float b, float c, float d) {
  uint2 w;
  __nv_bfloat162 x = __floats2bfloat162_rn(a, b), y = __floats2bfloat162_rn(c, d);
  w.x = *reinterpret_cast<uint32_t*>(&x);
  w.y = *reinterpret_cast<uint32_t*>(&y);
  return w;
}
__device__ __forceinline__ uint16_t bf16_bits(float v) {
  __nv_bfloat16 h = __float2bfloat16_rn(v);
  return *reinterpret_cast<uint16_t*>(&h);
}

// Hidden weights: B <- mu B + G (Eq. (10)) and X_0 = bf16(H) in the
// oriented NS layout, H being the NS input (B, or G + mu B for Nesterov).
// X_0 is left unnormalised: bf16 has the exponent range of fp32, and the
// first NS products apply 1 / ||H||_F (Eq. (5)) in their epilogues.
// Block t of the enumeration is a flat chunk of kChunk elements of W when
// X_0 has W's layout (B and G are contiguous, so they move as float4s
// whatever the row length), or a 64 x 64 tile of W transposed through shared
// memory when X_0 = W^T (tall W). Each block writes the fixed-order sum of
// squares of its part of H to partials[t]; x0norm_kernel reduces them.
__global__ void __launch_bounds__(kThreads, 8) momentum_x0_kernel(const MatInfo* __restrict__ mats, int nmat,
                                                                 const GroupInfo* __restrict__ groups,
                                                                 float* __restrict__ mom,
                                                                 const float* const* __restrict__ grads,
                                                                 const StepScalars* __restrict__ sc,
                                                                 float* __restrict__ partials) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  __shared__ float tile[kCastTile][kCastTile + 1];
  __shared__ float shf[32];
  const int64_t t = blockIdx.x;
  const int mi = find_mat(mats, nmat, t, 5);
  const MatInfo& M = mats[mi];
  const GroupInfo& Gi = groups[M.group];
  const int64_t lt = t - M.xblk_begin;
  const float mu = sc->mu;
  const int nesterov = sc->nesterov;
  float* B = mom + M.mom_off;
  const float* G = grads[mi];
  uint16_t* X = static_cast<uint16_t*>(Gi.x0) + M.gidx * Gi.s * Gi.lp;
  float ss = 0.f;
  if (!M.trans) {
    const int64_t e0 = lt * kChunk;
    const int64_t e1 = min(e0 + kChunk, M.m * M.n);
    const bool small32 = M.m * M.n <= static_cast<int64_t>(UINT32_MAX);
    for (int64_t e = e0 + 4 * threadIdx.x; e < e1; e += 4 * kThreads) {
      float h[4];
      if (e + 3 < e1) {
        const float4 g = __ldcs(reinterpret_cast<const float4*>(G + e));
        float4 b = *reinterpret_cast<const float4*>(B + e);
        b.x = fmaf(mu, b.x, g.x), b.y = fmaf(mu, b.y, g.y), b.z = fmaf(mu, b.z, g.z), b.w = fmaf(mu, b.w, g.w);
        *reinterpret_cast<float4*>(B + e) = b;
        if (nesterov) {
          h[0] = fmaf(mu, b.x, g.x), h[1] = fmaf(mu, b.y, g.y), h[2] = fmaf(mu, b.z, g.z), h[3] = fmaf(mu, b.w, g.w);
        } else {
          h[0] = b.x, h[1] = b.y, h[2] = b.z, h[3] = b.w;
        }
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          h[u] = 0.f;
          if (e + u < e1) {
            const float g = G[e + u];
            const float b = fmaf(mu, B[e + u], g);
            B[e + u] = b;
            h[u] = nesterov ? fmaf(mu, b, g) : b;
          }
        }
      }
      ss += h[0] * h[0] + h[1] * h[1] + h[2] * h[2] + h[3] * h[3];
      int64_t i, j;
      row_col(e, M.n, small32, i, j);
      if ((M.n & 3) == 0) {
        // four columns of one row (m n is then a multiple of 4, so e + 3 < e1)
        *reinterpret_cast<uint2*>(X + i * Gi.lp + j) = pack4_bf16(h[0], h[1], h[2], h[3]);
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (e + u < e1) X[i * Gi.lp + j] = bf16_bits(h[u]);
          if (++j == M.n) j = 0, ++i;
        }
      }
    }
  } else {
    const int64_t tiles_n = (M.n + kCastTile - 1) / kCastTile;
    const int64_t r0 = (lt / tiles_n) * kCastTile;
    const int64_t c0 = (lt % tiles_n) * kCastTile;
    const bool vec = (M.n & 3) == 0;
    const int cx = (threadIdx.x & 15) * 4;  // 4 columns
    const int ry = threadIdx.x >> 4;        // rows ry, ry + 16, ry + 32, ry + 48
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t row = r0 + ry + 16 * k, col = c0 + cx;
      float h[4] = {0.f, 0.f, 0.f, 0.f};
      if (row < M.m) {
        if (vec && col + 3 < M.n) {
          const float4 g = __ldcs(reinterpret_cast<const float4*>(G + row * M.n + col));
          float4 b = *reinterpret_cast<const float4*>(B + row * M.n + col);
          b.x = fmaf(mu, b.x, g.x), b.y = fmaf(mu, b.y, g.y), b.z = fmaf(mu, b.z, g.z), b.w = fmaf(mu, b.w, g.w);
          *reinterpret_cast<float4*>(B + row * M.n + col) = b;
          if (nesterov) {
            h[0] = fmaf(mu, b.x, g.x), h[1] = fmaf(mu, b.y, g.y), h[2] = fmaf(mu, b.z, g.z), h[3] = fmaf(mu, b.w, g.w);
          } else {
            h[0] = b.x, h[1] = b.y, h[2] = b.z, h[3] = b.w;
          }
        } else {
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (col + u < M.n) {
              const float g = G[row * M.n + col + u];
              const float b = fmaf(mu, B[row * M.n + col + u], g);
              B[row * M.n + col + u] = b;
              h[u] = nesterov ? fmaf(mu, b, g) : b;
            }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        ss += h[u] * h[u];
        tile[ry + 16 * k][cx + u] = h[u];
      }
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int xr = ry + 16 * k;
      const int64_t xrow = c0 + xr, xcol = r0 + cx;
      if (xrow >= M.n) continue;
      if (xcol + 3 < M.m) {
        *reinterpret_cast<uint2*>(X + xrow * Gi.lp + xcol) =
            pack4_bf16(tile[cx][xr], tile[cx + 1][xr], tile[cx + 2][xr], tile[cx + 3][xr]);
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (xcol + u < M.m) X[xrow * Gi.lp + xcol + u] = bf16_bits(tile[cx + u][xr]);
      }
    }
  }
  const float part = block_sum_f32(ss, shf);
  if (threadIdx.x == 0) partials[t] = part;
}

// 1 / ||H||_F of every hidden matrix (0 for a zero input, whose U is 0), one
// block per matrix: fixed-order fp32 reduction of the partials its momentum
// blocks wrote (fp32 throughout: this GPU's fp64 rate is a small fraction of
// its fp32 rate).
__global__ void __launch_bounds__(kThreads) x0norm_kernel(const MatInfo* __restrict__ mats,
                                                         const GroupInfo* __restrict__ groups,
                                                         const float* __restrict__ partials,
                                                         float* __restrict__ ginv, int* __restrict__ nonfinite) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  __shared__ float shf[32];
  const MatInfo& M = mats[blockIdx.x];
  if (M.kind != KIND_HIDDEN) return;
  const int64_t nblk = M.trans ? ((M.m + kCastTile - 1) / kCastTile) * ((M.n + kCastTile - 1) / kCastTile)
                               : (M.m * M.n + kChunk - 1) / kChunk;
  float acc = 0.f;
  for (int64_t c = threadIdx.x; c < nblk; c += kThreads) acc += partials[M.xblk_begin + c];
  const float total = block_sum_f32(acc, shf);
  if (threadIdx.x == 0) {
    const float nrm = sqrtf(total);
    if (!isfinite(total)) atomicCAS(nonfinite, 0, static_cast<int>(blockIdx.x) + 1);  // first non-finite entry, 1-based
    ginv[groups[M.group].mbase + M.gidx] = nrm > 0.f ? 1.0f / nrm : 0.f;
  }
}

// ------------------------------------------- remaining 2D parameters, vectors
// B <- mu B + G (Eq. (10)) and the row sums of squares of B, one warp per row
// (a vector is a single row). Row sums go to rvec.
__global__ void __launch_bounds__(kThreads) rows_kernel(const MatInfo* __restrict__ mats, int nmat,
                                                       float* __restrict__ mom, const float* const* __restrict__ grads,
                                                       const StepScalars* __restrict__ sc, float* __restrict__ rvec) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  const int64_t blk = blockIdx.x;
  const int mi = find_mat(mats, nmat, blk, 3);
  const MatInfo& M = mats[mi];
  const int lane = threadIdx.x & 31;
  const int64_t row = (blk - M.rblk_begin) * (kThreads / 32) + (threadIdx.x >> 5);
  if (row >= M.m) return;  // no block-wide synchronisation below
  const float mu = sc->mu;
  float* B = mom + M.mom_off + row * M.n;
  const float* G = grads[mi] + row * M.n;
  float ss = 0.f;
  if ((M.n & 3) == 0) {
    for (int64_t c = 4 * lane; c < M.n; c += 128) {
      const float4 g = __ldcs(reinterpret_cast<const float4*>(G + c));
      float4 b = *reinterpret_cast<const float4*>(B + c);
      b.x = fmaf(mu, b.x, g.x), b.y = fmaf(mu, b.y, g.y), b.z = fmaf(mu, b.z, g.z), b.w = fmaf(mu, b.w, g.w);
      *reinterpret_cast<float4*>(B + c) = b;
      ss += b.x * b.x + b.y * b.y + b.z * b.z + b.w * b.w;
    }
  } else {
    for (int64_t c = lane; c < M.n; c += 32) {
      const float b = fmaf(mu, B[c], G[c]);
      B[c] = b;
      ss += b * b;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (lane == 0) rvec[M.vec_off + row] = ss;
}

// Column sums of squares of N_r(B) (Eq. (12), inner operator): one block per
// kColSlab rows x 256 columns, deterministic; rows with RMS at or below eps
// contribute nothing.
__global__ void __launch_bounds__(kThreads) colpart_kernel(const MatInfo* __restrict__ mats, int nmat,
                                                          const float* __restrict__ mom, const float* __restrict__ rvec,
                                                          const StepScalars* __restrict__ sc, float* __restrict__ parts) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  __shared__ float rinv[kColSlab];
  const int64_t blk = blockIdx.x;
  const int mi = find_mat(mats, nmat, blk, 4);
  const MatInfo& M = mats[mi];
  const int64_t ncc = (M.n + kThreads - 1) / kThreads;  // column chunks
  const int64_t lb = blk - M.slab_begin;
  const int64_t ls = lb / ncc;
  const int64_t c = (lb - ls * ncc) * kThreads + threadIdx.x;
  const int64_t r0 = ls * kColSlab;
  const int nr = static_cast<int>(M.m - r0 < kColSlab ? M.m - r0 : kColSlab);
  for (int rr = threadIdx.x; rr < kColSlab; rr += kThreads) {
    float v = 0.f;
    if (rr < nr) {
      const float rms = sqrtf(rvec[M.vec_off + r0 + rr] / static_cast<float>(M.n));
      v = rms > sc->eps ? 1.0f / rms : 0.f;
    }
    rinv[rr] = v;
  }
  __syncthreads();
  if (c >= M.n) return;
  const float* B = mom + M.mom_off + r0 * M.n + c;
  float a4[4] = {0.f, 0.f, 0.f, 0.f};
  int r = 0;
  for (; r + 8 <= nr; r += 8) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float x = B[(r + u) * M.n] * rinv[r + u];
      a4[u & 3] += x * x;
    }
  }
  for (; r < nr; ++r) {
    const float x = B[r * M.n] * rinv[r];
    a4[r & 3] += x * x;
  }
  parts[M.cpart_off + ls * M.n + c] = (a4[0] + a4[1]) + (a4[2] + a4[3]);
}

// ------------------------------------------------------------------ X_0 cast
template <bool kFp16>
__device__ __forceinline__ uint16_t half_bits(float v) {
  if (kFp16) {
    __half h = __float2half_rn(v);
    return *reinterpret_cast<uint16_t*>(&h);
  }
  __nv_bfloat16 h = __float2bfloat16_rn(v);
  return *reinterpret_cast<uint16_t*>(&h);
}

__device__ __forceinline__ uint2 pack4(float a, float b, float c, float d, bool fp16) {
  uint2 w;
  if (fp16) {
    __half2 x = __floats2half2_rn(a, b), y = __floats2half2_rn(c, d);
    w.x = *reinterpret_cast<uint32_t*>(&x);
    w.y = *reinterpret_cast<uint32_t*>(&y);
  } else {
    __nv_bfloat162 x = __floats2bfloat162_rn(a, b), y = __floats2bfloat162_rn(c, d);
    w.x = *reinterpret_cast<uint32_t*>(&x);
    w.y = *reinterpret_cast<uint32_t*>(&y);
  }
  return w;
}

// One 64 x 64 tile of W per block. Threads read 4 consecutive columns
// (128-bit loads when the row length allows) and write 4 consecutive 16-bit
// values; tall matrices go through a shared-memory transpose.
template <bool kFp16>
__global__ void __launch_bounds__(kThreads) cast_x0_kernel(const MatInfo* __restrict__ mats, int nmat,
                                                           const GroupInfo* __restrict__ groups,
                                                           const float* __restrict__ mom,
                                                           const float* const* __restrict__ grads,
                                                           const StepScalars* __restrict__ sc,
                                                           const float* __restrict__ x0scale) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  __shared__ float tile[kCastTile][kCastTile + 1];
  const int64_t t = blockIdx.x;
  const int mi = find_mat(mats, nmat, t, 1);
  const MatInfo& M = mats[mi];
  const GroupInfo& Gi = groups[M.group];
  const int64_t tiles_n = (M.n + kCastTile - 1) / kCastTile;
  const int64_t lt = t - M.tile_begin;
  const int64_t r0 = (lt / tiles_n) * kCastTile;
  const int64_t c0 = (lt % tiles_n) * kCastTile;
  const float scale = x0scale[mi];
  const float mu = sc->mu;
  const int nesterov = sc->nesterov;
  const float* B = mom + M.mom_off;
  const float* G = grads[mi];
  uint16_t* X = static_cast<uint16_t*>(Gi.x0) + M.gidx * Gi.s * Gi.lp;
  const bool vec = (M.n & 3) == 0;
  const int cx = (threadIdx.x & 15) * 4;  // 4 columns
  const int ry = threadIdx.x >> 4;        // rows ry, ry + 16, ry + 32, ry + 48
  float h[4][4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int64_t row = r0 + ry + 16 * k, col = c0 + cx;
#pragma unroll
    for (int u = 0; u < 4; ++u) h[k][u] = 0.f;
    if (row >= M.m) continue;
    if (vec && col + 3 < M.n) {
      float4 b = *reinterpret_cast<const float4*>(B + row * M.n + col);
      if (nesterov) {
        const float4 g = *reinterpret_cast<const float4*>(G + row * M.n + col);
        b.x = fmaf(mu, b.x, g.x), b.y = fmaf(mu, b.y, g.y), b.z = fmaf(mu, b.z, g.z), b.w = fmaf(mu, b.w, g.w);
      }
      h[k][0] = b.x, h[k][1] = b.y, h[k][2] = b.z, h[k][3] = b.w;
    } else {
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (col + u < M.n) {
          float b = B[row * M.n + col + u];
          if (nesterov) b = fmaf(mu, b, G[row * M.n + col + u]);
          h[k][u] = b;
        }
    }
  }
  if (!M.trans) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t row = r0 + ry + 16 * k, col = c0 + cx;
      if (row >= M.m) continue;
      if (col + 3 < M.n) {
        *reinterpret_cast<uint2*>(X + row * Gi.lp + col) =
            pack4(h[k][0] * scale, h[k][1] * scale, h[k][2] * scale, h[k][3] * scale, kFp16);
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (col + u < M.n) X[row * Gi.lp + col + u] = half_bits<kFp16>(h[k][u] * scale);
      }
    }
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
      for (int u = 0; u < 4; ++u) tile[ry + 16 * k][cx + u] = h[k][u] * scale;
    __syncthreads();
    // X row = W column c0 + xr; X columns = W rows r0 + cx .. + 3.
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int xr = ry + 16 * k;
      const int64_t xrow = c0 + xr, xcol = r0 + cx;
      if (xrow >= M.n) continue;
      if (xcol + 3 < M.m) {
        *reinterpret_cast<uint2*>(X + xrow * Gi.lp + xcol) =
            pack4(tile[cx][xr], tile[cx + 1][xr], tile[cx + 2][xr], tile[cx + 3][xr], kFp16);
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (xcol + u < M.m) X[xrow * Gi.lp + xcol + u] = half_bits<kFp16>(tile[cx + u][xr]);
      }
    }
  }
}

// ----------------------------------------------------------------- statistics
// sum_{k < count} p[k * stride] with eight independent partial sums (term k
// goes to partial k % 8) so that the loads overlap; fixed order.
__device__ __forceinline__ float strided_sum8(const float* __restrict__ p, int64_t count, int64_t stride) {
  float a8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  int64_t k = 0;
  for (; k + 8 <= count; k += 8) {
#pragma unroll
    for (int u = 0; u < 8; ++u) a8[u] += p[(k + u) * stride];
  }
  for (; k < count; ++k) a8[k & 7] += p[k * stride];
  return ((a8[0] + a8[1]) + (a8[2] + a8[3])) + ((a8[4] + a8[5]) + (a8[6] + a8[7]));
}

// K block sums at once: each value goes through the same warp tree and the
// same in-order sum over warps as block_sum_f32 gives it alone, with one set
// of barriers for all of them. sh holds at least 33 * K floats.
template <int K>
__device__ __forceinline__ void block_sum_multi(float (&v)[K], float* sh) {
  const unsigned FULL = 0xffffffffu;
#pragma unroll
  for (int k = 0; k < K; ++k)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_xor_sync(FULL, v[k], o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) {
#pragma unroll
    for (int k = 0; k < K; ++k) sh[32 * k + w] = v[k];
  }
  __syncthreads();
  if (threadIdx.x < K) {
    float r = 0.f;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) r += sh[32 * threadIdx.x + i];
    sh[32 * K + threadIdx.x] = r;
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < K; ++k) v[k] = sh[32 * K + k];
}

// Two-pass fp32 CVs of Eq. (8) of a (length la) and b (length lb) over their
// entries above delta, both at once: the mean pass, then the squared
// deviations.
__device__ void block_cv2(const float* a, int64_t la, const float* b, int64_t lb, float delta, float* sh, float* ga,
                          float* gb) {
  float p[4] = {0.f, 0.f, 0.f, 0.f};  // count and sum over a, then over b
  for (int64_t i = threadIdx.x; i < la; i += blockDim.x) {
    const float x = a[i];
    if (x > delta) p[0] += 1.f, p[1] += x;
  }
  for (int64_t i = threadIdx.x; i < lb; i += blockDim.x) {
    const float x = b[i];
    if (x > delta) p[2] += 1.f, p[3] += x;
  }
  block_sum_multi<4>(p, sh);
  const float mean_a = p[0] > 0.f ? p[1] / p[0] : 0.f;
  const float mean_b = p[2] > 0.f ? p[3] / p[2] : 0.f;
  float q[2] = {0.f, 0.f};
  for (int64_t i = threadIdx.x; i < la; i += blockDim.x) {
    const float x = a[i];
    if (x > delta) q[0] += (x - mean_a) * (x - mean_a);
  }
  for (int64_t i = threadIdx.x; i < lb; i += blockDim.x) {
    const float x = b[i];
    if (x > delta) q[1] += (x - mean_b) * (x - mean_b);
  }
  block_sum_multi<2>(q, sh);
  *ga = p[0] > 0.f ? sqrtf(q[0] / p[0]) / mean_a : 0.f;
  *gb = p[2] > 0.f ? sqrtf(q[1] / p[2]) / mean_b : 0.f;
}

// Statistics and normalisation scales, one block per parameter.
//   hidden     : r, c of U (Eq. (7)) from the partial sums the last NS
//                epilogue wrote, gamma_r, gamma_c (Eq. (8)), the side of
//                Eq. (11) and its scale vector (Eq. (9)) in svec;
//   remaining 2D: r = row RMS of B, c = column RMS of N_r(B) (Eq. (12)),
//                1/r in svec, 1/c in tvec, their CVs for inspection;
//   vector     : r[0] = RMS of B, 1/r[0] in svec (Eq. (13)).
// RMS values at or below eps are treated as zero (scale 0).
__global__ void __launch_bounds__(kFinThreads) finalize_kernel(const MatInfo* __restrict__ mats,
                                                               const StepScalars* __restrict__ sc,
                                                               const float* __restrict__ parts,
                                                               float* __restrict__ rvec, float* __restrict__ cvec,
                                                               float* __restrict__ svec, float* __restrict__ tvec,
                                                               MatStats* __restrict__ stats,
                                                               unsigned long long* __restrict__ dircount,
                                                               int* __restrict__ nonfinite) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  __shared__ float shf[33 * 4];
  const MatInfo& M = mats[blockIdx.x];
  const float delta = sc->eps;
  float* r = rvec + M.vec_off;
  float* c = cvec + M.vec_off;
  float* s = svec + M.vec_off;
  const float inv_n = 1.0f / static_cast<float>(M.n);
  const float inv_m = 1.0f / static_cast<float>(M.m);
  if (M.kind == KIND_VECTOR) {
    if (threadIdx.x == 0) {
      if (!isfinite(r[0])) atomicCAS(nonfinite, 0, static_cast<int>(blockIdx.x) + 1);
      const float rms = sqrtf(r[0] * inv_n);  // r[0] holds the sum of squares
      r[0] = rms;
      s[0] = rms > delta ? 1.0f / rms : 0.f;
      stats[blockIdx.x].gamma_r = 0.0;
      stats[blockIdx.x].gamma_c = 0.0;
      stats[blockIdx.x].direction = 3;
    }
    return;
  }
  if (M.kind == KIND_TWO_SIDED) {
    float* t = tvec + M.vec_off;
    for (int64_t i = threadIdx.x; i < M.m; i += blockDim.x) {
      if (!isfinite(r[i])) atomicCAS(nonfinite, 0, static_cast<int>(blockIdx.x) + 1);
      const float rms = sqrtf(r[i] * inv_n);  // r holds the row sums of squares
      r[i] = rms;
      s[i] = rms > delta ? 1.0f / rms : 0.f;
    }
    // column sums over the slabs
    const int64_t nslabs = (M.m + kColSlab - 1) / kColSlab;
    for (int64_t j = threadIdx.x; j < M.n; j += blockDim.x) {
      const float tot = strided_sum8(parts + M.cpart_off + j, nslabs, M.n);
      const float rms = sqrtf(tot * inv_m);
      c[j] = rms;
      t[j] = rms > delta ? 1.0f / rms : 0.f;
    }
    __syncthreads();
    float gr, gc;
    block_cv2(r, M.m, c, M.n, delta, shf, &gr, &gc);
    if (threadIdx.x == 0) {
      stats[blockIdx.x].gamma_r = static_cast<double>(gr);
      stats[blockIdx.x].gamma_c = static_cast<double>(gc);
      stats[blockIdx.x].direction = 2;
    }
    return;
  }
  // NS rows (s of them) are the weight's rows, or its columns when transposed.
  const int64_t tiles_n = 2 * ((M.l + 255) / 256);  // two epilogue halves per 256-column tile
  const int64_t nrb = (M.s + 31) / 32;
  for (int64_t i = threadIdx.x; i < M.s; i += blockDim.x) {
    const float acc = strided_sum8(parts + M.rpart_off + i, tiles_n, M.s);
    if (!M.trans) r[i] = sqrtf(acc * inv_n);
    else c[i] = sqrtf(acc * inv_m);
  }
  for (int64_t j = threadIdx.x; j < M.l; j += blockDim.x) {
    const float acc = strided_sum8(parts + M.cpart_off + j, nrb, M.l);
    if (!M.trans) c[j] = sqrtf(acc * inv_m);
    else r[j] = sqrtf(acc * inv_n);
  }
  __syncthreads();
  // Eq. (8) over entries > delta: two passes (mean, then squared deviations),
  // fp32 with fixed-order block reductions.
  float gam0, gam1;
  block_cv2(r, M.m, c, M.n, delta, shf, &gam0, &gam1);
  int dir;
  if (sc->rule == 1) {
    // Eq. (6): every row scaled by sqrt(max(m, n)), no equilibration
    dir = 4;
    const float f = sqrtf(static_cast<float>(max(M.m, M.n)));
    for (int64_t i = threadIdx.x; i < M.m; i += blockDim.x) s[i] = f;
  } else {
    dir = gam0 >= gam1 - sc->tie_atol ? 0 : 1;
    const float* v = dir == 0 ? r : c;
    const int64_t len = dir == 0 ? M.m : M.n;
    for (int64_t i = threadIdx.x; i < len; i += blockDim.x) {
      const float x = v[i];
      s[i] = x > delta ? 1.0f / x : 0.0f;   // RMS at or below delta: treated as zero
    }
  }
  if (threadIdx.x == 0) {
    stats[blockIdx.x].gamma_r = static_cast<double>(gam0);
    stats[blockIdx.x].gamma_c = static_cast<double>(gam1);
    stats[blockIdx.x].direction = dir;
    if (dir < 2) dircount[2 * blockIdx.x + dir] += 1ull;  // one block per entry: no other writer
  }
}

// ----------------------------------------------------------------------- apply
// W <- (1 - lr wd) W - rho lr U~ (Eq. (14)), U~ = scaled U (hidden) or scaled
// B (remaining 2D: s_i t_j B_ij; vector: s_0 B_j). Under the Muon rule the
// hidden scale is sqrt(max(m, n)) for every row (Eq. (6)).
__global__ void __launch_bounds__(kThreads, 8) apply_kernel(const MatInfo* __restrict__ mats, int nmat,
                                                         float* const* __restrict__ params,
                                                         const uint16_t* __restrict__ uslab,
                                                         const float* __restrict__ mom,
                                                         const float* __restrict__ svec,
                                                         const float* __restrict__ tvec,
                                                         const MatStats* __restrict__ stats,
                                                         const StepScalars* __restrict__ sc) {
  pdl_allow_dependents();
  pdl_wait_predecessor();
  const int64_t chunk = blockIdx.x;
  const int mi = find_mat(mats, nmat, chunk, 0);
  const MatInfo& M = mats[mi];
  const int64_t numel = M.m * M.n;
  const int64_t e0 = (chunk - M.chunk_begin) * kChunk;
  const int64_t e1 = min(e0 + kChunk, numel);
  const float decay = 1.0f - sc->lr * sc->wd;
  const bool hidden = M.kind == KIND_HIDDEN;
  // hidden: U is fp16(kUScale U) with row stride un; others: the momentum, fp32, contiguous
  const float step = sc->rho * sc->lr * (hidden ? 1.0f / kUScale : 1.0f);
  // mode 0: per-row scale (also the uniform scale of Eq. (6), held per row);
  // 1: per-column scale; 2: row scale x column scale
  const int dir = hidden ? stats[mi].direction : (M.kind == KIND_TWO_SIDED ? 2 : 0);
  const int mode = dir == 4 ? 0 : dir;
  const float* sv = svec + M.vec_off;
  const float* tv = tvec + M.vec_off;
  const uint16_t* U16 = uslab + M.u_off;
  const float* U32 = mom + M.mom_off;
  float* W = params[mi];
  if ((M.n & 3) == 0) {
    // four columns of one row per thread (m n is a multiple of 4, so e + 3 < e1)
    const bool small32 = numel <= static_cast<int64_t>(UINT32_MAX);
    for (int64_t e = e0 + 4 * threadIdx.x; e < e1; e += 4 * kThreads) {
      int64_t i, j;
      row_col(e, M.n, small32, i, j);
      float4 w = *reinterpret_cast<const float4*>(W + e);
      float u[4];
      if (hidden) {
        const uint2 h = __ldcs(reinterpret_cast<const uint2*>(U16 + i * M.un + j));
        const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&h.x));
        const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&h.y));
        u[0] = a.x, u[1] = a.y, u[2] = b.x, u[3] = b.y;
      } else {
        const float4 b = __ldcs(reinterpret_cast<const float4*>(U32 + e));
        u[0] = b.x, u[1] = b.y, u[2] = b.z, u[3] = b.w;
      }
      float s0, s1, s2, s3;
      if (mode == 0) {
        s0 = s1 = s2 = s3 = sv[i];
      } else {
        const float4 s4 = *reinterpret_cast<const float4*>((mode == 1 ? sv : tv) + j);
        s0 = s4.x, s1 = s4.y, s2 = s4.z, s3 = s4.w;
        if (mode == 2) {
          const float si = sv[i];
          s0 *= si, s1 *= si, s2 *= si, s3 *= si;
        }
      }
      w.x = fmaf(decay, w.x, -step * (s0 * u[0]));
      w.y = fmaf(decay, w.y, -step * (s1 * u[1]));
      w.z = fmaf(decay, w.z, -step * (s2 * u[2]));
      w.w = fmaf(decay, w.w, -step * (s3 * u[3]));
      *reinterpret_cast<float4*>(W + e) = w;
    }
  } else {
    // rows of any length: a warp reads and writes 32 consecutive elements
    // of W (and of a row of U); each thread has four elements in flight
    int64_t e = e0 + threadIdx.x;
    int64_t i = e / M.n, j = e - i * M.n;
    for (; e < e1; e += 4 * kThreads) {
      float w[4], u[4], f[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int64_t ek = e + k * kThreads;
        w[k] = u[k] = f[k] = 0.f;
        if (ek < e1) {
          w[k] = W[ek];
          u[k] = hidden ? __half2float(__ushort_as_half(__ldcs(U16 + i * M.un + j))) : __ldcs(U32 + ek);
          f[k] = mode == 0 ? sv[i] : (mode == 1 ? sv[j] : sv[i] * tv[j]);
        }
        for (j += kThreads; j >= M.n; j -= M.n) ++i;
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int64_t ek = e + k * kThreads;
        if (ek < e1) W[ek] = fmaf(decay, w[k], -step * (f[k] * u[k]));
      }
    }
  }
}

// The normalised update of one entry that apply_kernel applies, W <- (1 -
// lr wd) W - rho lr U~: U~ = diag(r^-1) U or U diag(c^-1) (Eqs. (9), (11)),
// sqrt(max(m, n)) U under the Eq. (6) rule, N_c(N_r(B)) (Eq. (12)) or
// B / RMS(B) (Eq. (13)), with the same scale factors and operands.
__global__ void __launch_bounds__(kThreads) update_kernel(MatInfo M, int mi, const uint16_t* __restrict__ uslab,
                                                          const float* __restrict__ mom,
                                                          const float* __restrict__ svec,
                                                          const float* __restrict__ tvec,
                                                          const MatStats* __restrict__ stats, float* __restrict__ dst) {
  const bool hidden = M.kind == KIND_HIDDEN;
  const int dir = hidden ? stats[mi].direction : (M.kind == KIND_TWO_SIDED ? 2 : 0);
  const int mode = dir == 4 ? 0 : dir;
  const float* sv = svec + M.vec_off;
  const float* tv = tvec + M.vec_off;
  const uint16_t* U16 = uslab + M.u_off;
  const float* U32 = mom + M.mom_off;
  const float back = hidden ? 1.0f / kUScale : 1.0f;  // a power of two: exact
  const int64_t numel = M.m * M.n;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; e < numel;
       e += static_cast<int64_t>(gridDim.x) * kThreads) {
    const int64_t i = e / M.n, j = e - i * M.n;
    const float u = hidden ? __half2float(__ushort_as_half(U16[i * M.un + j])) : U32[e];
    const float f = mode == 0 ? sv[i] : (mode == 1 ? sv[j] : sv[i] * tv[j]);
    dst[e] = (f * u) * back;
  }
}

// Bounded-wait self test: waits on a flag nobody sets and reports a timeout.
__global__ void wait_selftest_kernel(const volatile int* flag, int* err, unsigned long long timeout_ns) {
  unsigned long long t0;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  for (unsigned int it = 0;; ++it) {
    if (*flag != 0) return;
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    if (t - t0 > timeout_ns || it >= (1u << 28)) {
      atomicCAS(err, 0, DEV_TIMEOUT_TEST);
      return;
    }
  }
}

}  // namespace

cudaError_t launch_momentum_norm(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(momentum_norm_kernel, dim3((unsigned)L.total_hchunks), dim3(kThreads), 0, st, 1, L.mats, L.nmat,
                    L.groups, L.mom, L.grads, L.sc, L.partials, L.counters, L.x0scale, L.nonfinite);
}

cudaError_t launch_momentum_x0(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(momentum_x0_kernel, dim3((unsigned)L.total_xblks), dim3(kThreads), 0, st, 1, L.mats, L.nmat,
                    L.groups, L.mom, L.grads, L.sc, L.partials);
}

cudaError_t launch_x0norm(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(x0norm_kernel, dim3((unsigned)L.nmat), dim3(kThreads), 0, st, 1, L.mats, L.groups,
                    static_cast<const float*>(L.partials), L.ginv, L.nonfinite);
}

cudaError_t launch_rows(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(rows_kernel, dim3((unsigned)L.total_rblks), dim3(kThreads), 0, st, 1, L.mats, L.nmat, L.mom,
                    L.grads, L.sc, L.rvec);
}

cudaError_t launch_colpart(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(colpart_kernel, dim3((unsigned)L.total_slabs), dim3(kThreads), 0, st, 1, L.mats, L.nmat,
                    static_cast<const float*>(L.mom), static_cast<const float*>(L.rvec), L.sc, L.parts);
}

cudaError_t launch_cast_x0(const LaunchCtx& L, bool fp16, cudaStream_t st) {
  if (fp16)
    return launch_pdl(cast_x0_kernel<true>, dim3((unsigned)L.total_tiles), dim3(kThreads), 0, st, 1, L.mats, L.nmat,
                      L.groups, static_cast<const float*>(L.mom), L.grads, L.sc, static_cast<const float*>(L.x0scale));
  return launch_pdl(cast_x0_kernel<false>, dim3((unsigned)L.total_tiles), dim3(kThreads), 0, st, 1, L.mats, L.nmat,
                    L.groups, static_cast<const float*>(L.mom), L.grads, L.sc, static_cast<const float*>(L.x0scale));
}

cudaError_t launch_stats(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(finalize_kernel, dim3(L.nmat), dim3(kFinThreads), 0, st, 1, L.mats, L.sc,
                    static_cast<const float*>(L.parts), L.rvec, L.cvec, L.svec, L.tvec, L.stats, L.dircount,
                    L.nonfinite);
}

cudaError_t launch_apply(const LaunchCtx& L, cudaStream_t st) {
  return launch_pdl(apply_kernel, dim3((unsigned)L.total_chunks), dim3(kThreads), 0, st, 1, L.mats, L.nmat, L.params,
                    static_cast<const uint16_t*>(L.uslab), static_cast<const float*>(L.mom),
                    static_cast<const float*>(L.svec), static_cast<const float*>(L.tvec),
                    static_cast<const MatStats*>(L.stats), L.sc);
}

cudaError_t launch_update(const LaunchCtx& L, const MatInfo& M, int mi, float* dst, cudaStream_t st) {
  const int64_t blocks = std::min<int64_t>((M.m * M.n + kThreads - 1) / kThreads, 4096);
  update_kernel<<<static_cast<unsigned>(blocks), kThreads, 0, st>>>(
      M, mi, static_cast<const uint16_t*>(L.uslab), static_cast<const float*>(L.mom),
      static_cast<const float*>(L.svec), static_cast<const float*>(L.tvec), static_cast<const MatStats*>(L.stats), dst);
  return cudaPeekAtLastError();
}

cudaError_t launch_wait_selftest(const int* flag, int* err, unsigned long long timeout_ns, cudaStream_t st) {
  wait_selftest_kernel<<<1, 1, 0, st>>>(flag, err, timeout_ns);
  return cudaGetLastError();
}

}  // namespace meq
