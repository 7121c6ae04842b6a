// Newton-Schulz GEMMs on the sm_103a tensor cores (tcgen05 + TMA + TMEM).
//
// One persistent, warp-specialised kernel computes every product of the
// quintic iteration, Eq. (5) of the paper, for a batch of same-shape groups:
//
//   MODE_GRAM : A   = X X^T / alpha^2           (s x s, contraction over l)
//   MODE_POLY : P   = a I + b A + c (A A)       (s x s, contraction over s)
//               a I + b A is added in fp32 from the same 16-bit A the
//               product uses, so P is exactly a polynomial of that matrix
//   MODE_XUPD : X'  = P X * (alpha'/alpha)      (s x l, contraction over s)
//   MODE_XLAST: U   = P X / alpha, written as fp16(2^14 U) in the weight's own
//               layout, with the sums of squares of the stored U's rows and
//               columns (Eq. (7)) reduced into per-tile partials
//
// P X equals a X + (b A + c A^2) X of Eq. (5) exactly in real arithmetic.
// A and P are symmetric: their launches run only the tiles that hold a 32 x 32
// block on or above the diagonal and store each strictly-upper block twice
// (as is, and transposed in shared memory with ldmatrix.trans / stmatrix), so
// every element is written from one accumulator.
// X is stored scaled by a power of two alpha so its entries stay in the
// normal range of fp16; the epilogues undo the scale in fp32.
//
// Roles (352 threads, one CTA per SM):
//   warp 0 : TMA producer (one thread), shared-memory ring of 4 stages
//            (single CTA) or 6 (CTA pair)
//   warp 1 : TMEM allocator and tcgen05.mma issuer (one thread; with CTA
//            pairs, the leader's thread issues cta_group::2 MMAs for both)
//   warps 2-9 : epilogue; warp w reads TMEM lanes 32*(w%4) .. +31 and takes
//               every other 32-column chunk (two warps per lane quarter, so
//               each SM sub-partition can hide one warp's latencies behind
//               the other's work)
//   warp 10 : tile scheduler (one thread, leader CTA)
// Tiles are handed out dynamically: each unit (CTA or CTA pair) starts on
// its own index and then draws from an atomic counter, so a launch ends
// within about one tile on every unit whatever the mix of tile sizes and SM
// speeds. The leader's scheduler thread claims each index one tile ahead of
// the producer, decodes it (group, matrix, tile row and column, k-block
// count) and passes the decoded entry to every role of both CTAs through a
// ring in shared memory. The producer and the MMA issuer run ahead of the
// tensor pipe by only a few k-blocks, so neither can afford the decode, a
// dependent integer chain of one thread: measured at 0.35-0.6 us per tile,
// it left the tensor pipe idle for about 0.5 us between tiles when they did
// it themselves.
// Two 128x256 fp32 accumulators (512 TMEM columns) let the epilogue of one
// tile overlap the MMAs of the next. The epilogue stages 32 x 32 blocks in
// swizzled shared memory; the symmetric A and P (each block stored twice)
// leave by TMA stores, X and U by coalesced 16-byte stores from the threads
// (the update launches keep the SM's TMA unit for their operand loads).
//
// Every mbarrier wait is bounded (time and iteration count). On expiry the
// waiting role records an error code, the others see it and stop, in-flight
// TMA copies and MMAs are drained with bounded waits, TMEM is freed and the
// CTA returns.
#include "meq_internal.cuh"

namespace meq {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, UK = 16;  // per-CTA rows, tile columns, k-block, MMA K
constexpr int A_BYTES = BM * BK * 2;                 // 16 KB
constexpr int NUM_EPI_WARPS = kNsEpilogueWarps;      // two per TMEM lane quarter
constexpr int SCHED_WARP = 2 + NUM_EPI_WARPS;
constexpr int NUM_THREADS = 64 + 32 * NUM_EPI_WARPS + 32;
constexpr uint32_t TMEM_COLS = 512;
constexpr int SLOT_BYTES = 2048;                     // one 32 x 32 16-bit block (two per epilogue warp)
constexpr int SCHED_D = 16;                          // entries of the tile ring (16 bytes each)
constexpr float kUInvScale2 = 1.0f / (kUScale * kUScale);  // exact: kUScale is a power of two

// kPair = 1: one CTA computes a 128 x 256 tile (tcgen05 cta_group::1).
// kPair = 2: a cluster of two CTAs computes a 256 x 256 tile with
// cta_group::2 MMAs: each CTA holds its own 128 rows of A and half of B
// (128 rows / columns), so a stage is 32 KB instead of 48 KB per SM and six
// stages fit.
template <int kPair>
struct Cfg {
  static constexpr int TILE_M = BM * kPair;
  static constexpr int BN_LOCAL = BN / kPair;
  static constexpr int B_BYTES = BN_LOCAL * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = kPair == 1 ? 4 : 6;
  // full, empty, tmem full x2, tmem empty x2, drain, tile ring full / empty,
  // entry taken by the producer
  static constexpr int NUM_BARS = 2 * STAGES + 4 + 1 + 2 * SCHED_D + 1;
  static constexpr int SMEM_EPI_OFF = STAGES * STAGE_BYTES;
  static constexpr int SMEM_BAR_OFF = SMEM_EPI_OFF + NUM_EPI_WARPS * 2 * SLOT_BYTES;
  // barriers, the TMEM address word (16 bytes reserved), the tile ring
  // (16-byte aligned), alignment slack of the dynamic shared memory
  static constexpr int SMEM_BYTES = SMEM_BAR_OFF + NUM_BARS * 8 + 16 + 15 + 16 * SCHED_D + 1024;
  static_assert(SMEM_BYTES <= 232448, "shared memory budget of one sm_103a CTA");
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ uint32_t mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.b32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Single-thread bounded wait. Returns false when it gave up (its own timeout,
// recorded in *err, or an error another role recorded).
__device__ bool wait_bounded(uint32_t bar, uint32_t parity, int* err, int code, uint64_t timeout_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 127u) == 0) {
      if (*reinterpret_cast<volatile int*>(err) != 0) return false;
      if (global_ns() - t0 > timeout_ns || it >= (1u << 28)) {
        atomicCAS(err, 0, code);
        return false;
      }
    }
  }
}

// Bounded wait that does not stop early on another role's error: for the
// MMA issuer's drain, which must see its MMAs complete before TMEM is freed
// (they always do, so the bound is a safety net only).
__device__ bool wait_bounded_drain(uint32_t bar, uint32_t parity, int* err, int code, uint64_t timeout_ns) {
  const uint64_t t0 = global_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 127u) == 127u && (global_ns() - t0 > timeout_ns || it >= (1u << 28))) {
      atomicCAS(err, 0, code);
      return false;
    }
  }
}

// Warp-uniform bounded wait (all 32 lanes call it; all get the same answer).
__device__ bool wait_bounded_warp(uint32_t bar, uint32_t parity, int* err, int code, uint64_t timeout_ns) {
  const unsigned FULL = 0xffffffffu;
  if (__all_sync(FULL, mbar_try_wait(bar, parity))) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (__all_sync(FULL, mbar_try_wait(bar, parity))) return true;
    if ((it & 127u) == 0) {
      int stop = 0;
      if ((threadIdx.x & 31) == 0) {
        if (*reinterpret_cast<volatile int*>(err) != 0) {
          stop = 1;
        } else if (global_ns() - t0 > timeout_ns || it >= (1u << 28)) {
          atomicCAS(err, 0, code);
          stop = 1;
        }
      }
      if (__shfl_sync(FULL, stop, 0)) return false;
    }
  }
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* tm, uint32_t bar, int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(bar), "r"(x), "r"(y), "r"(z)
      : "memory");
}
// Pair variant: the copy lands in this CTA's shared memory and completes on
// an mbarrier that may live in the peer CTA (the pair leader's).
__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap* tm, uint32_t bar_cluster, int x, int y,
                                                 int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, "
      "%5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(bar_cluster), "r"(x), "r"(y), "r"(z)
      : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t smem_addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Accumulator release by the epilogue. Only the warp's tcgen05.ld reads must
// precede it, and tcgen05.wait::ld has already completed them; a release
// would also hold the warp until its earlier global stores are visible to
// the cluster, which the MMA issuer does not need.
__device__ __forceinline__ void mbar_arrive_relaxed_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}
// Writes a 16-byte tile-ring entry into the peer CTA's shared memory and
// completes it as a 16-byte transaction on the peer's barrier, which this
// call also arms (one arrival). A waiter on that barrier then sees the value,
// as after a TMA load; no fence of the writer's other memory operations is
// involved.
__device__ __forceinline__ void st_async_peer_v4(uint32_t addr_cluster, uint32_t bar_cluster, uint4 v) {
  asm volatile("mbarrier.arrive.expect_tx.relaxed.cluster.shared::cluster.b64 _, [%0], 16;" ::"r"(bar_cluster)
               : "memory");
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                   addr_cluster),
               "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(bar_cluster)
               : "memory");
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr)
               : "memory");
  return v;
}
__device__ __forceinline__ void mbar_arrive_local(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* tm) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tc_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_mma_pair(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the barrier at this shared-memory offset in both CTAs of the pair
// once all prior cta_group::2 MMAs of this thread have completed.
__device__ __forceinline__ void tc_commit_pair_both(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}
__device__ __forceinline__ void tc_commit_pair_local(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// Shared-memory matrix descriptor for a 128-byte-swizzled tile (sm_100 format:
// start >> 4 in bits 0-13, leading byte offset >> 4 in 16-29, stride byte
// offset >> 4 in 32-45, descriptor version 1 at bit 46, swizzle mode 2
// (128B) in bits 61-63).
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// 32 lanes x 32 consecutive fp32 columns from TMEM.
__device__ __forceinline__ void tmem_ld_32cols(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

struct TileCoord {
  int g, mat, tm, tn;
};

// Tiles of a group are numbered matrix by matrix (walked backwards when
// p.reverse is set, so a launch starts on the matrices its predecessor wrote
// last, which are still in L2). Dense outputs (X' = P X) run in bands of
// G.band tile rows, each band column by column (the host sizes a band so
// its row panels of P fit in a quarter of L2): the tiles in flight at once
// (one per CTA pair) then share one or a few column panels of X and the
// band's panels of P, where a row-by-row walk re-read every column panel of
// a wide X once per tile row (measured at 4096 x 11008: 4.5 times the
// launch's algorithmic bytes from DRAM). Symmetric outputs (Gram, polynomial) run tn-major over
// the tiles with tm * TILE_M < (tn + 1) * 256, i.e. those holding a 32 x 32
// block on or above the diagonal.
__device__ __forceinline__ int find_segment(const GemmParams& p, int t) {
  int lo = 0, hi = p.ngroups - 1;  // the last segment whose tile_begin <= t
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.g[mid].tile_begin <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}
template <int kPair>
__device__ __forceinline__ TileCoord decode_tile(const GemmParams& p, int t) {
  if (p.reverse) t = p.total_tiles - 1 - t;
  const int g = find_segment(p, t);
  const GemmGroup& G = p.g[g];
  const int local = t - G.tile_begin;
  const int mat = local / G.tiles_per_mat;
  int r = local - mat * G.tiles_per_mat;
  TileCoord c;
  c.g = g;
  c.mat = mat;
  if (!G.sym) {
    const int band = r / (G.band * G.tiles_n);
    const int in = r - band * G.band * G.tiles_n;
    const int rows = min(G.band, G.tiles_m - band * G.band);
    c.tm = band * G.band + in % rows;
    c.tn = in / rows;
  } else {
    int tn = 0;
    for (;;) {
      const int cnt = min(G.tiles_m, ((tn + 1) * BN) / Cfg<kPair>::TILE_M);
      if (r < cnt) break;
      r -= cnt;
      ++tn;
    }
    c.tm = r;
    c.tn = tn;
  }
  return c;
}

// A decoded tile as the scheduler publishes it: x = tile index, y = matrix,
// z = group | tm << 4 | tn << 18, w = k-blocks | (diagonal tile whose B half
// is its A half) << 16.
__device__ __forceinline__ TileCoord entry_coord(uint4 e) {
  TileCoord c;
  c.g = static_cast<int>(e.z & 15u);
  c.mat = static_cast<int>(e.y);
  c.tm = static_cast<int>((e.z >> 4) & 0x3FFFu);
  c.tn = static_cast<int>(e.z >> 18);
  return c;
}

__device__ __forceinline__ uint32_t pack_half2(float a, float b, int fp16) {
  if (fp16) {
    __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
  }
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ float2 unpack_half2(uint32_t w, int fp16) {
  if (fp16) {
    __half2 h = *reinterpret_cast<__half2*>(&w);
    return __half22float2(h);
  }
  __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&w);
  return __bfloat1622float2(h);
}

// ---- epilogue block staging ----------------------------------------------------
// A warp stages one 32-row block in its shared-memory slot with a swizzled
// layout (conflict-free for the per-row writes below), then writes it back out
// with coalesced 16-byte global stores: lane L takes 16-byte chunk (L % 4) of
// rows L / 4, L / 4 + 8, ... so one warp instruction covers 8 rows x 64 bytes.

// Row-major 32 x 32 16-bit block, 64-byte rows, 64B swizzle (16-byte chunk k
// of row r sits at chunk k ^ ((r >> 1) & 3)).
__device__ __forceinline__ void fill_half_rows(uint8_t* slot, int r, const float* v, int fp16) {
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    uint4 w;
    w.x = pack_half2(v[8 * k + 0], v[8 * k + 1], fp16);
    w.y = pack_half2(v[8 * k + 2], v[8 * k + 3], fp16);
    w.z = pack_half2(v[8 * k + 4], v[8 * k + 5], fp16);
    w.w = pack_half2(v[8 * k + 6], v[8 * k + 7], fp16);
    *reinterpret_cast<uint4*>(slot + r * 64 + ((k ^ ((r >> 1) & 3)) << 4)) = w;
  }
}
// The transposed block: element (row j, col r) = v[j] of lane r.
// Writes the transpose of the 32 x 32 16-bit block in `src` into `dst` (both
// 64-byte rows of four 16-byte chunks, chunk k of row r at k ^ ((r >> 1) & 3)):
// ldmatrix .trans reads each 8 x 8 sub-block (g, q) as its transpose and
// stmatrix writes it as sub-block (q, g).
__device__ __forceinline__ void transpose_slot(const uint8_t* src, uint8_t* dst, int lane) {
  const uint32_t base = smem_u32(src), dbase = smem_u32(dst);
  const int r8 = lane & 7, q = lane >> 3;
  uint32_t f[4][4];
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const int row = 8 * g + r8;  // lane group q addresses sub-block (g, q)
    const uint32_t addr = base + row * 64 + ((q ^ ((row >> 1) & 3)) << 4);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(f[g][0]), "=r"(f[g][1]), "=r"(f[g][2]), "=r"(f[g][3])
                 : "r"(addr)
                 : "memory");
  }
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const int row = 8 * q + r8;  // the transpose of sub-block (g, q) is sub-block (q, g)
    const uint32_t addr = dbase + row * 64 + ((g ^ ((row >> 1) & 3)) << 4);
    asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(f[g][0]),
                 "r"(f[g][1]), "r"(f[g][2]), "r"(f[g][3])
                 : "memory");
  }
}
// 32 rows x 64 bytes (a staged 16-bit 32 x 32 block) -> global with 16-byte
// stores: rows r < rows_valid, 16-byte chunks k < chunks_valid of each row.
__device__ __forceinline__ void store_block64(const uint8_t* slot, int lane, uint8_t* dst, int64_t ld_bytes,
                                              int rows_valid, int chunks_valid) {
  const int k = lane & 3;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = (lane >> 2) + 8 * i;
    const uint4 w = *reinterpret_cast<const uint4*>(slot + r * 64 + ((k ^ ((r >> 1) & 3)) << 4));
    if (r < rows_valid && k < chunks_valid) *reinterpret_cast<uint4*>(dst + r * ld_bytes + k * 16) = w;
  }
}
// A staged 32 x 32 16-bit block -> global by TMA (tensor map box {32, 32, 1},
// 64-byte swizzle = the staging layout). Rows and columns outside the
// tensor's extent are not written. The writing threads make their
// shared-memory stores visible to the TMA unit first (fence.proxy.async).
__device__ __forceinline__ void tma_store_block(const CUtensorMap* tm, const uint8_t* src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(tm)),
               "r"(smem_u32(src)), "r"(x), "r"(y), "r"(z)
               : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// The shared-memory reads of every committed store have completed.
__device__ __forceinline__ void bulk_wait_reads() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// Every committed store has completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
template <int kPair>
__global__ void __launch_bounds__(NUM_THREADS, 1) ns_gemm_kernel(const __grid_constant__ GemmParams p) {
  using C_ = Cfg<kPair>;
  constexpr int STAGES = C_::STAGES;
  constexpr int STAGE_BYTES = C_::STAGE_BYTES;
  constexpr int TILE_M = C_::TILE_M;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t bar0 = base + C_::SMEM_BAR_OFF;
  const uint32_t drain_bar = bar0 + 8 * (2 * STAGES + 4);
  const uint32_t tmem_slot = bar0 + 8 * C_::NUM_BARS;
  volatile uint32_t* tmem_slot_ptr = reinterpret_cast<volatile uint32_t*>(gbase + C_::SMEM_BAR_OFF + 8 * C_::NUM_BARS);
#define FULL_BAR(s) (bar0 + 8u * (s))
#define EMPTY_BAR(s) (bar0 + 8u * (STAGES + (s)))
#define TFULL_BAR(a) (bar0 + 8u * (2 * STAGES + (a)))
#define TEMPTY_BAR(a) (bar0 + 8u * (2 * STAGES + 2 + (a)))
#define SFULL_BAR(i) (bar0 + 8u * (2 * STAGES + 5 + (i)))
#define SEMPTY_BAR(i) (bar0 + 8u * (2 * STAGES + 5 + SCHED_D + (i)))
#define PTAKEN_BAR (bar0 + 8u * (2 * STAGES + 5 + 2 * SCHED_D))
  const uint32_t ring = (tmem_slot + 16u + 15u) & ~15u;  // SCHED_D entries of 16 bytes

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int* err = p.err;
  const uint64_t tmo = p.timeout_ns;
  // Pair mode: rank 0 of each 2-CTA cluster issues the MMAs for both.
  const uint32_t rank = kPair == 2 ? cluster_rank() : 0u;
  const bool leader = rank == 0;
  const int unit = kPair == 2 ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int nunits = kPair == 2 ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(FULL_BAR(s), 1);
      mbar_init(EMPTY_BAR(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(TFULL_BAR(a), 1);
      mbar_init(TEMPTY_BAR(a), kPair * NUM_EPI_WARPS);
    }
    mbar_init(drain_bar, 1);
    for (int i = 0; i < SCHED_D; ++i) {
      mbar_init(SFULL_BAR(i), 1);
      // consumers of each entry: the producer and epilogue warps of each
      // CTA, and the leader's MMA issuer
      mbar_init(SEMPTY_BAR(i), 1 + kPair * (1 + NUM_EPI_WARPS));
    }
    mbar_init(PTAKEN_BAR, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    for (int g = 0; g < p.ngroups; ++g) {
      prefetch_tmap(&p.g[g].tmA);
      prefetch_tmap(&p.g[g].tmB);
      if (p.g[g].sym) prefetch_tmap(&p.g[g].tmO);
    }
  }
  if (warp == 1) {
    if (kPair == 2) {
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(tmem_slot), "r"(TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(tmem_slot), "r"(TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  if (kPair == 2) cluster_sync_all();  // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot_ptr;
  pdl_allow_dependents();
  // The wait for the previous kernel of the step (griddepcontrol.wait, per
  // thread) is taken by the roles that touch global memory, each before its
  // first access: the producer, the epilogue warps and the scheduler (after
  // it has published the unit's first tile). The MMA issuer works on shared
  // memory and TMEM only.

  // ------------------------------------------------------------------ tile queue
  // Each unit (CTA pair) starts on tile `unit`; further tiles are handed out
  // by the launch's atomic counter, so units that finish early take more and
  // the launch ends within about one tile on every unit. The leader's
  // scheduler claims entry n + 1 once the producer has taken entry n (the
  // claim stays one tile ahead, as the load balance needs), decodes it and
  // publishes it in the tile ring of both CTAs (the peer's copy by st.async,
  // which completes on the peer's barrier like a TMA load, so no memory
  // fence is waited on); every other role reads the ring in the same order.
  // A reader hands its slot back with a relaxed arrive (a release would
  // first wait for the epilogue's outstanding global stores). Its read has
  // completed long before the slot can be written again: entry n + 16 is
  // written after the producer took entry n + 15, by which time every role
  // has used entry n -- the operand ring holds at most 6 k-blocks and the
  // accumulators 2 tiles.
  auto sched_put = [&](int n, uint4 e) -> bool {
    const int i = n & (SCHED_D - 1);
    if (!wait_bounded(SEMPTY_BAR(i), ((n / SCHED_D) & 1) ^ 1u, err, DEV_TIMEOUT_SCHED_PUT, tmo)) return false;
    if (kPair == 2) st_async_peer_v4(map_to_rank(ring + 16u * i, 1), map_to_rank(SFULL_BAR(i), 1), e);
    st_shared_v4(ring + 16u * i, e);
    mbar_arrive_local(SFULL_BAR(i));  // release (CTA scope) of the store above
    return true;
  };
  auto sched_take = [&](int n, uint4& e) -> bool {
    const int i = n & (SCHED_D - 1);
    if (!wait_bounded(SFULL_BAR(i), (n / SCHED_D) & 1, err, DEV_TIMEOUT_SCHED_TAKE, tmo)) return false;
    e = ld_shared_v4(ring + 16u * i);
    mbar_arrive_relaxed_cluster((kPair == 2 && !leader) ? map_to_rank(SEMPTY_BAR(i), 0) : SEMPTY_BAR(i));
    return true;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- TMA producer
      pdl_wait_predecessor();  // operands come from the previous kernel of the step
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_mask = 0, issued_parity = 0;  // bit s: stage s was filled / parity of its last fill
      bool ok = true;
      for (int n = 0; ok; ++n) {
        uint4 e;
        if (!sched_take(n, e)) break;
        if (leader) mbar_arrive_local(PTAKEN_BAR);  // the scheduler may claim the next tile
        if (static_cast<int>(e.x) >= p.total_tiles) break;
        const TileCoord c = entry_coord(e);
        const GemmGroup& G = p.g[c.g];
        const int nk = static_cast<int>(e.w & 0xFFFFu);
        // Mode, descriptor and B layout are per launch: reading them at a
        // fixed index keeps them launch-uniform for the compiler (measured:
        // 2% of the step).
        const int b_mn_major = p.g[0].b_mn_major;
        const int arow = c.tm * TILE_M + static_cast<int>(rank) * BM;
        const int bcol = c.tn * BN + static_cast<int>(rank) * C_::BN_LOCAL;
        // A diagonal tile of a symmetric product (X X^T, A A) has each CTA's
        // B half equal to its A half (same rows of the same buffer, same box):
        // only A is loaded, and the MMA reads it as B too.
        const bool b_is_a = (e.w >> 16) & 1u;
        for (int kb = 0; kb < nk; ++kb) {
          if (!wait_bounded(EMPTY_BAR(stage), phase ^ 1u, err, DEV_TIMEOUT_PRODUCER, tmo)) {
            ok = false;
            break;
          }
          const uint32_t sa = base + stage * STAGE_BYTES;
          const uint32_t sb = sa + A_BYTES;
          if (kPair == 1) {
            mbar_expect_tx(FULL_BAR(stage), STAGE_BYTES);
            tma_load_3d(sa, &G.tmA, FULL_BAR(stage), kb * BK, arow, c.mat);
            if (!b_mn_major) {
              tma_load_3d(sb, &G.tmB, FULL_BAR(stage), kb * BK, bcol, c.mat);
            } else {
#pragma unroll
              for (int j = 0; j < C_::BN_LOCAL / 64; ++j)
                tma_load_3d(sb + j * (64 * BK * 2), &G.tmB, FULL_BAR(stage), bcol + j * 64, kb * BK, c.mat);
            }
          } else {
            // Both CTAs' copies complete on the leader's full barrier, which
            // the leader arms with the bytes of both.
            if (leader) mbar_expect_tx(FULL_BAR(stage), b_is_a ? 2 * A_BYTES : 2 * STAGE_BYTES);
            const uint32_t fb = leader ? FULL_BAR(stage) : map_to_rank(FULL_BAR(stage), 0);
            // tests (debug_skip_load): the stage is armed but this CTA's half never
            // comes, so the MMA issuer's bounded wait on it expires
            const bool skip = p.debug_skip_load && leader && unit == 0 && n == 0 && kb == 0;
            if (!skip) {
              tma_load_3d_pair(sa, &G.tmA, fb, kb * BK, arow, c.mat);
              if (b_is_a) {
                // B is this stage's A
              } else if (!b_mn_major) {
                tma_load_3d_pair(sb, &G.tmB, fb, kb * BK, bcol, c.mat);
              } else {
#pragma unroll
                for (int j = 0; j < C_::BN_LOCAL / 64; ++j)
                  tma_load_3d_pair(sb + j * (64 * BK * 2), &G.tmB, fb, bcol + j * 64, kb * BK, c.mat);
              }
            }
          }
          issued_mask |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      // Drain: every copy issued into this CTA has landed before it exits (for
      // the pair, the leader's full barriers count the peer's bytes as well).
      if (leader)
        for (int s = 0; s < STAGES; ++s)
          if ((issued_mask >> s) & 1u)
            wait_bounded(FULL_BAR(s), (issued_parity >> s) & 1u, err, DEV_TIMEOUT_DRAIN, tmo);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------------------------------------------------------- MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int n = 0; ok; ++n) {
        uint4 e;
        if (!sched_take(n, e) || static_cast<int>(e.x) >= p.total_tiles) break;
        const int nk = static_cast<int>(e.w & 0xFFFFu);
        const int b_mn_major = p.g[0].b_mn_major;
        const uint32_t idesc = p.g[0].idesc;
        const uint32_t b_lbo = b_mn_major ? (64u * BK * 2u) : 16u;
        // diagonal tile of a symmetric product: B is read from the A half (the producer loads A only)
        const bool b_is_a = (e.w >> 16) & 1u;
        if (!wait_bounded(TEMPTY_BAR(acc), acc_phase ^ 1u, err, DEV_TIMEOUT_MMA_TMEM, tmo)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(acc * BN);
        for (int kb = 0; kb < nk; ++kb) {
          if (!wait_bounded(FULL_BAR(stage), phase, err, DEV_TIMEOUT_MMA_FULL, tmo)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = base + stage * STAGE_BYTES;
          const uint32_t sb = b_is_a ? sa : sa + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / UK; ++k) {
            const uint64_t adesc = smem_desc(sa + k * (UK * 2), 16u, 1024u);
            const uint64_t bdesc = b_mn_major ? smem_desc(sb + k * (UK * 128), b_lbo, 1024u)
                                                : smem_desc(sb + k * (UK * 2), 16u, 1024u);
            if (kPair == 2) tc_mma_pair(d, adesc, bdesc, idesc, (kb > 0 || k > 0) ? 1u : 0u);
            else tc_mma(d, adesc, bdesc, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          }
          if (kPair == 2) tc_commit_pair_both(EMPTY_BAR(stage));
          else tc_commit(EMPTY_BAR(stage));
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if (kPair == 2) tc_commit_pair_both(TFULL_BAR(acc));
        else tc_commit(TFULL_BAR(acc));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      // Drain: all MMAs issued by this thread are complete before TMEM is freed.
      if (kPair == 2) tc_commit_pair_local(drain_bar);
      else tc_commit(drain_bar);
      wait_bounded_drain(drain_bar, 0, err, DEV_TIMEOUT_DRAIN, tmo);
    }
    __syncwarp();
  } else if (warp < 2 + NUM_EPI_WARPS) {
    // ------------------------------------------------------------------ epilogue
    pdl_wait_predecessor();  // reads A (polynomial) and overwrites buffers of earlier kernels
    // Warp ew (0..7) owns TMEM lanes 32*q .. +31 (q = warp % 4), i.e. rows
    // 32q .. 32q+31 of the tile, chunks ch with ch % 2 == half, and two 2 KB
    // shared-memory slots: `slot` takes the polynomial's A block (prefetched
    // into registers one chunk ahead) and then the block as computed, `slot_t`
    // its transpose (mirrored blocks, transposed U). The symmetric outputs
    // (A, P: twice the stores, with the mirrors) leave by TMA stores, and a
    // slot is rewritten only after the stores of the previous chunk have read
    // it; X and U leave by 16-byte stores from the threads, which keeps the
    // TMA unit free for the operand loads of the longer update launches.
    const int q = warp & 3;
    const int ew = warp - 2;
    const int half = ew >> 2;
    uint8_t* slot = gbase + C_::SMEM_EPI_OFF + ew * (2 * SLOT_BYTES);
    uint8_t* slot_t = slot + SLOT_BYTES;
    int acc = 0;
    uint32_t acc_phase = 0;

    // The leader's tmem-empty barrier counts the epilogue warps of both CTAs.
    const uint32_t tempty_target0 = (kPair == 2 && !leader) ? map_to_rank(TEMPTY_BAR(0), 0) : TEMPTY_BAR(0);
    const uint32_t tempty_target1 = (kPair == 2 && !leader) ? map_to_rank(TEMPTY_BAR(1), 0) : TEMPTY_BAR(1);
    for (int n = 0;; ++n) {
      uint4 e = make_uint4(0u, 0u, 0u, 0u);
      int got = 1;
      if (lane == 0) got = sched_take(n, e) ? 1 : 0;
      got = __shfl_sync(0xffffffffu, got, 0);
      e.x = __shfl_sync(0xffffffffu, e.x, 0);
      e.y = __shfl_sync(0xffffffffu, e.y, 0);
      e.z = __shfl_sync(0xffffffffu, e.z, 0);
      if (!got || static_cast<int>(e.x) >= p.total_tiles) break;
      const TileCoord c = entry_coord(e);
      const GemmGroup& G = p.g[c.g];
      const int mode = p.g[0].mode;  // one mode per launch (a launch-uniform read)
      const int row0 = c.tm * TILE_M + static_cast<int>(rank) * BM + q * 32;
      const int R = row0 / 32;  // 32-row block index
      const int rows_valid = min(32, G.M - row0);
      float rsum = 0.f;            // XLAST: this lane's row, sum of squares over the tile
      const int nch = min(BN / 32, (G.N - c.tn * BN + 31) / 32);
      int ch0 = G.sym ? max(0, R - c.tn * 8) : 0;  // blocks strictly below the diagonal come from mirrors
      if ((ch0 & 1) != half) ++ch0;                // this warp's chunks: ch % 2 == half
      if (row0 >= G.M) ch0 = nch;
      uint8_t* outm = static_cast<uint8_t*>(G.out) + static_cast<int64_t>(c.mat) * G.out_mstride;
      // POLY: A block of the chunk, lane L holds 16-byte chunk (L % 4) of rows L/4 + 8i.
      uint4 aux[4];
      const uint8_t* auxm = reinterpret_cast<const uint8_t*>(G.aux) + static_cast<int64_t>(c.mat) * G.aux_mstride;
      auto load_aux = [&](int col0) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int r = (lane >> 2) + 8 * i;
          aux[i] = make_uint4(0u, 0u, 0u, 0u);
          if (r < rows_valid) {
            const uint4* src = reinterpret_cast<const uint4*>(auxm + static_cast<int64_t>(row0 + r) * G.aux_ld +
                                                              static_cast<int64_t>(col0) * 2 + (lane & 3) * 16);
            aux[i] = __ldg(src);
          }
        }
      };
      // What needs no accumulator is requested before waiting for it: the
      // polynomial's first A block, and the output scale (iteration 0 reads
      // its matrix's 1/||H||_F from global memory).
      if (mode == MODE_POLY && ch0 < nch) load_aux(c.tn * BN + ch0 * 32);
      float sc = G.scale;
      if (mode != MODE_POLY && G.minv_pow) {
        const float iv = G.minv[c.mat];
        sc *= G.minv_pow == 2 ? iv * iv : iv;
      }
      if (!wait_bounded_warp(TFULL_BAR(acc), acc_phase, err, DEV_TIMEOUT_EPI, tmo)) break;
      tc_fence_after();
      for (int ch = ch0; ch < nch; ch += 2) {
        const int col0 = c.tn * BN + ch * 32;
        const int C = c.tn * 8 + ch;
        float v[32];
        tmem_ld_32cols(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN + ch * 32), v);
        if (G.tma_out) {
          if (lane == 0) bulk_wait_reads();  // both slots free
        }
        __syncwarp();
        if (mode == MODE_POLY) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int r = (lane >> 2) + 8 * i, k = lane & 3;
            *reinterpret_cast<uint4*>(slot + r * 64 + ((k ^ ((r >> 1) & 3)) << 4)) = aux[i];
          }
          __syncwarp();
          if (ch + 2 < nch) load_aux(col0 + 64);  // in flight while this chunk is processed
          const int row = row0 + lane;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint4 w = *reinterpret_cast<const uint4*>(slot + lane * 64 + ((k ^ ((lane >> 1) & 3)) << 4));
            const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const float2 a2 = unpack_half2(ws[h], G.aux_fp16);
              const int j = 8 * k + 2 * h;
              v[j] = fmaf(p.cc, v[j], fmaf(p.cb, a2.x, (col0 + j == row) ? p.ca : 0.f));
              v[j + 1] = fmaf(p.cc, v[j + 1], fmaf(p.cb, a2.y, (col0 + j + 1 == row) ? p.ca : 0.f));
            }
          }
          __syncwarp();  // slot free for the output block
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] *= sc;
        }
        if (mode == MODE_XLAST) {
          // U is stored as fp16(kUScale U). The sums of squares are taken from
          // those stored values and scaled back by kUScale^-2 (a power of
          // two) when written, so the statistics describe the U the update
          // applies. Each pair is rounded once: the packed halves go to the
          // staging slot, their exact fp32 values back into v.
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            uint32_t wv[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int j = 8 * k + 2 * h;
              const __half2 hh = __floats2half2_rn(v[j] * kUScale, v[j + 1] * kUScale);
              wv[h] = *reinterpret_cast<const uint32_t*>(&hh);
              const float2 f = __half22float2(hh);
              v[j] = f.x;
              v[j + 1] = f.y;
            }
            *reinterpret_cast<uint4*>(slot + lane * 64 + ((k ^ ((lane >> 1) & 3)) << 4)) =
                make_uint4(wv[0], wv[1], wv[2], wv[3]);
          }
          // Column sums of squares over the warp's 32 rows: transpose-reduce
          // so that lane j ends with the sum for column col0 + j.
          float sq[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            sq[j] = v[j] * v[j];
            rsum += sq[j];
          }
#pragma unroll
          for (int o = 16; o >= 1; o >>= 1) {
#pragma unroll
            for (int i = 0; i < o; ++i) {
              const bool up = (lane & o) != 0;
              const float send = up ? sq[i] : sq[i + o];
              const float keep = up ? sq[i + o] : sq[i];
              sq[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
            }
          }
          if (col0 + lane < G.N)
            G.cpart[(static_cast<int64_t>(c.mat) * ((G.M + 31) / 32) + R) * G.N + col0 + lane] = sq[0] * kUInvScale2;
          // 8-element chunks that start below the row length stay inside the
          // padded row (stride = row length rounded up to 8); the slot holds
          // the block (filled above)
          __syncwarp();
          if (!G.trans) {
            // U rows = NS rows row0 + r, U columns = NS columns col0 + j
            store_block64(slot, lane, outm + static_cast<int64_t>(row0) * G.out_ld + col0 * 2, G.out_ld, rows_valid,
                          min(4, (G.N - col0 + 7) / 8));
          } else {
            // U rows = NS columns col0 + j, U columns = NS rows row0 + r
            transpose_slot(slot, slot_t, lane);
            __syncwarp();
            store_block64(slot_t, lane, outm + static_cast<int64_t>(col0) * G.out_ld + row0 * 2, G.out_ld,
                          min(32, G.N - col0), min(4, (G.M - row0 + 7) / 8));
          }
        } else if (!G.tma_out) {
          // X rows are padded to a multiple of 64 elements: whole 32-column blocks stay inside them
          fill_half_rows(slot, lane, v, G.out_fp16);
          __syncwarp();
          store_block64(slot, lane, outm + static_cast<int64_t>(row0) * G.out_ld + col0 * 2, G.out_ld, rows_valid, 4);
        } else {
          fill_half_rows(slot, lane, v, G.out_fp16);
          const bool mirror = G.sym && C > R;  // strictly above the diagonal: also store the transpose
          if (mirror) {
            __syncwarp();
            transpose_slot(slot, slot_t, lane);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_block(&G.tmO, slot, col0, row0, c.mat);
            if (mirror) tma_store_block(&G.tmO, slot_t, row0, col0, c.mat);
            bulk_commit();
          }
        }
        __syncwarp();  // reconverge before the next warp-wide tcgen05.ld
      }
      if (mode == MODE_XLAST && row0 < G.M && row0 + lane < G.M)  // one partial per (tile column, half)
        G.rpart[(static_cast<int64_t>(c.mat) * G.tiles_n * 2 + c.tn * 2 + half) * G.M + row0 + lane] = rsum * kUInvScale2;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive_relaxed_cluster(kPair == 2 ? (acc == 0 ? tempty_target0 : tempty_target1) : TEMPTY_BAR(acc));
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    // The outputs are in global memory before the CTA leaves.
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  } else if (warp == SCHED_WARP) {
    if (lane == 0 && leader) {
      // ---------------------------------------------------------------- tile scheduler
      int t = unit;
      int fetched = 0;  // the counter value for the next tile
      for (int n = 0;; ++n) {
        if (n > 0) {
          // the producer has taken entry n - 1 (its phase n - 1 is complete)
          if (!wait_bounded(PTAKEN_BAR, static_cast<uint32_t>(n - 1) & 1u, err, DEV_TIMEOUT_SCHED_PUT, tmo)) break;
          t = nunits + fetched;
        }
        uint4 e = make_uint4(static_cast<uint32_t>(t), 0u, 0u, 0u);
        if (t < p.total_tiles) {
          const TileCoord c = decode_tile<kPair>(p, t);
          const GemmGroup& G = p.g[c.g];
          const int nk = (G.K + BK - 1) / BK;
          const bool b_is_a = kPair == 2 && G.sym && !p.g[0].b_mn_major && c.tm * TILE_M == c.tn * BN;
          e.y = static_cast<uint32_t>(c.mat);
          e.z = static_cast<uint32_t>(c.g) | (static_cast<uint32_t>(c.tm) << 4) | (static_cast<uint32_t>(c.tn) << 18);
          e.w = static_cast<uint32_t>(nk) | (b_is_a ? 0x10000u : 0u);
        }
        if (!sched_put(n, e)) break;
        if (t >= p.total_tiles) break;
        // Entry 0, the unit's own tile, depends only on the launch parameters
        // and is published while the previous kernel may still run; the
        // queue counter, which that kernel's last unit resets, only after it.
        if (n == 0) pdl_wait_predecessor();
        fetched = atomicAdd(p.sched, 1);  // read when the producer has taken this entry
      }
    }
    __syncwarp();
  }
#undef FULL_BAR
#undef EMPTY_BAR
#undef TFULL_BAR
#undef TEMPTY_BAR
#undef SFULL_BAR
#undef SEMPTY_BAR
#undef PTAKEN_BAR

  if (kPair == 2 && *reinterpret_cast<volatile int*>(err) != 0) {
    // After an early exit, give copies still in flight towards either CTA
    // time to land before the pair leaves (bounded: about 2 ms).
    const uint64_t t0 = global_ns();
    while (global_ns() - t0 < 2000000ull) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (kPair == 2) cluster_sync_all();  // no CTA leaves while its peer may still signal it
  tc_fence_after();
  if (threadIdx.x == 0 && leader) {
    // The last unit to finish resets the tile queue. Every unit's fetches
    // precede its count here, and the next launch reads the queue only after
    // this grid has completed.
    __threadfence();
    if (atomicAdd(p.sched + 1, 1) == nunits - 1) {
      p.sched[0] = 0;
      p.sched[1] = 0;
    }
  }
  if (warp == 1) {
    if (kPair == 2)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS) : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS) : "memory");
  }
}

}  // namespace

int ns_gemm_smem_bytes(int pair) { return pair == 2 ? Cfg<2>::SMEM_BYTES : Cfg<1>::SMEM_BYTES; }

cudaError_t prepare_ns_gemm() {
  cudaError_t e = cudaFuncSetAttribute(ns_gemm_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<1>::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(ns_gemm_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<2>::SMEM_BYTES);
}

cudaError_t launch_ns_gemm(const GemmParams& p, int grid, int pair, cudaStream_t st) {
  if (pair == 2) return launch_pdl(ns_gemm_kernel<2>, dim3(grid), dim3(NUM_THREADS), Cfg<2>::SMEM_BYTES, st, 2, p);
  return launch_pdl(ns_gemm_kernel<1>, dim3(grid), dim3(NUM_THREADS), Cfg<1>::SMEM_BYTES, st, 1, p);
}

}  // namespace meq
