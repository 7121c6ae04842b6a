// Host side of the MeqMuon C ABI: planning, workspace, launch sequence.
//
// Planning (at meq_init_state):
//   * every matrix W (m x n) is oriented for Newton-Schulz as s x l with
//     s = min(m, n): X = W for m <= n, X = W^T for m > n. In exact arithmetic
//     X (X^T X)^k = (X X^T)^k X, so the iterate of W^T is the transpose of the
//     iterate of W and the result is the same matrix (Eq. (5));
//   * matrices with the same (s, l) form a group whose X buffers are stacked
//     [count][s][l_pad] so one 3D TMA tensor map covers the whole group, and
//     one GEMM launch covers up to kMaxGroups groups;
//   * one device arena holds momentum, NS buffers and statistics.
// Per step (meq_step), on the caller's stream:
//   upload step scalars + pointer tables, then
//   momentum_norm, cast_x0, K x (GRAM, POLY, XUPD|XLAST), stats, finalize, apply
// optionally replayed from a CUDA graph captured at the first step.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <limits>
#include <map>
#include <tuple>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/meq.h"

#include <nvtx3/nvToolsExt.h>
#include "meq_elementwise.cuh"

using namespace meq;

namespace {

constexpr int64_t kAlignBytes = 1024;

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

std::string g_init_error;  // last meq_init_state failure text

struct Group {
  int64_t s = 0, l = 0, lp = 0, sp = 0, count = 0;
  int trans = 0;           // members are tall (W = X^T)
  int64_t m = 0, n = 0, un = 0;  // weight shape of every member, U row stride
  int64_t u_base = 0;      // element offset of the group's fp16 U block [count][m][un]
  int64_t mbase = 0;       // first slot of the group in the per-matrix inverse-norm array
  int64_t rpart_base = 0;  // float offsets of the fused-statistics partials
  int64_t cpart_base = 0;
  std::vector<int> mats;
  uint16_t* x[2] = {nullptr, nullptr};
  uint16_t* a16 = nullptr;
  uint16_t* p16 = nullptr;
  float alpha0 = 1.f, alpha = 1.f;
};

// Sub-allocation plan of the arena (offsets in bytes).
// With guards on (option debug_canaries), a band of kGuardBytes precedes the
// first buffer and follows every buffer; it is filled with kGuardByte at init
// and meq_check_canaries looks for bytes a kernel wrote into it.
constexpr int64_t kGuardBytes = 4096;
constexpr int kGuardByte = 0xA5;

struct Layout {
  int64_t total = 0;
  bool guards = false;
  std::vector<std::pair<int64_t, int64_t>> guard_ranges;  // (offset, bytes)
  explicit Layout(bool with_guards = false) : guards(with_guards) {
    if (guards) guard(0);
  }
  void guard(int64_t off) {
    guard_ranges.emplace_back(off, kGuardBytes);
    total = off + kGuardBytes;
  }
  int64_t add(int64_t bytes) {
    const int64_t off = total;
    total += round_up(std::max<int64_t>(bytes, 1), kAlignBytes);
    if (guards) guard(total);
    return off;
  }
};

}  // namespace

void meq::set_global_error(const std::string& msg) { g_init_error = msg; }

struct meq_state {
  int n = 0;
  std::vector<meq_shape> shapes;
  std::vector<int> kinds;                     // meq_kind per entry
  int n_hidden = 0, n_rows = 0, n_two = 0;    // hidden / row-pass (remaining 2D + vectors) / two-sided
  meq_options opt{};
  int device = 0;
  int num_sms = 0;
  std::vector<MatInfo> mats;
  std::vector<Group> groups;
  int64_t total_chunks = 0, total_hchunks = 0, total_tiles = 0, total_rblks = 0, total_slabs = 0, total_xblks = 0;
  int64_t mom_floats = 0, u_halves = 0, vec_floats = 0, parts_floats = 0;
  char* arena = nullptr;
  int64_t arena_bytes = 0;
  // device views
  MatInfo* d_mats = nullptr;
  GroupInfo* d_groups = nullptr;
  float* d_mom = nullptr;
  uint16_t* d_u = nullptr;
  float* d_rvec = nullptr;
  float* d_cvec = nullptr;
  float* d_svec = nullptr;
  float* d_tvec = nullptr;
  float* d_parts = nullptr;
  float* d_partials = nullptr;
  unsigned int* d_counters = nullptr;
  float* d_x0scale = nullptr;
  float* d_ginv = nullptr;
  MatStats* d_stats = nullptr;
  unsigned long long* d_dircount = nullptr;  // [n][2]: row / column choices of Eq. (11)
  char* d_step = nullptr;  // StepScalars, params[n], grads[n]
  int* d_err = nullptr;
  int* d_flag = nullptr;
  int* d_nonfinite = nullptr;  // 1 + first entry with a non-finite momentum norm, 0 if none
  int* d_sched = nullptr;      // NS GEMM tile queue (two ints, zero between launches)
  int64_t step_bytes = 0;
  std::vector<char> step_host;
  // launch plan
  std::vector<GemmParams> gemm;  // in launch order
  std::vector<int> gemm_grid;
  LaunchCtx ctx{};
  bool graph_ready = false;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t gexec = nullptr;
  // meq_step_prepare / meq_step_apply: one graph each, captured on first use
  cudaGraph_t graph_prep = nullptr, graph_apply = nullptr;
  cudaGraphExec_t gexec_prep = nullptr, gexec_apply = nullptr;
  bool prepared = false;  // a prepare is waiting for its apply
  cudaStream_t last_stream = nullptr;
  int kernels_per_step = 0;
  bool profiling = false;
  std::vector<std::vector<cudaEvent_t>> prof_events;  // eager launches: 6 events per profiled step
  // graph replay: one graph with event-record nodes between the phases, its
  // 6 events, and the summed phase times of the replays read so far
  cudaGraph_t graph_prof = nullptr;
  cudaGraphExec_t gexec_prof = nullptr;
  std::vector<cudaEvent_t> prof_graph_events;
  double prof_sum[5] = {0, 0, 0, 0, 0};
  int64_t prof_graph_steps = 0;
  std::string last_error;
  int64_t persistent_bytes = 0;
  std::vector<std::pair<int64_t, int64_t>> guard_ranges;  // arena guard bands (debug_canaries)
};

namespace {

// IEEE 754 binary16 -> binary32 (exact): sign, 5-bit exponent with bias 15,
// 10-bit fraction; exponent 0 holds zero and the subnormals, 31 inf / NaN.
float half_bits_to_float(uint16_t h) {
  const float sign = (h & 0x8000u) ? -1.0f : 1.0f;
  const int ex = (h >> 10) & 0x1f;
  const int fr = h & 0x3ff;
  if (ex == 0) return sign * std::ldexp(static_cast<float>(fr), -24);
  if (ex == 31) return fr ? std::numeric_limits<float>::quiet_NaN() : sign * std::numeric_limits<float>::infinity();
  return sign * std::ldexp(static_cast<float>(fr | 0x400), ex - 25);
}

meq_status fail(meq_state* st, meq_status s, const std::string& msg) {
  if (st) st->last_error = msg; else g_init_error = msg;
  return s;
}

meq_status cuda_fail(meq_state* st, cudaError_t e, const char* what) {
  return fail(st, MEQ_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

bool valid_options(const meq_options& o, std::string* why) {
  if (o.ns_steps < 1 || o.ns_steps > 32) { *why = "ns_steps must be in 1..32"; return false; }
  if (!(o.rho > 0.f) || !std::isfinite(o.rho)) { *why = "rho must be positive and finite"; return false; }
  if (!std::isfinite(o.ns_a) || !std::isfinite(o.ns_b) || !std::isfinite(o.ns_c)) { *why = "NS coefficients must be finite"; return false; }
  if (!(o.tie_atol >= 0.f)) { *why = "tie_atol must be >= 0"; return false; }
  if (!(o.wait_timeout_ms > 0.f)) { *why = "wait_timeout_ms must be > 0"; return false; }
  if (o.workspace_limit_bytes < 0) { *why = "workspace_limit_bytes must be >= 0"; return false; }
  if (o.ns_cta_pair != 0 && o.ns_cta_pair != 1) { *why = "ns_cta_pair must be 0 or 1"; return false; }
  if (o.ns_x0_fused != 0 && o.ns_x0_fused != 1) { *why = "ns_x0_fused must be 0 or 1"; return false; }
  if (o.debug_canaries != 0 && o.debug_canaries != 1) { *why = "debug_canaries must be 0 or 1"; return false; }
  if (o.debug_skip_load != 0 && o.debug_skip_load != 1) { *why = "debug_skip_load must be 0 or 1"; return false; }
  if (o.debug_skip_load && !o.ns_cta_pair) {
    *why = "debug_skip_load requires ns_cta_pair = 1";
    return false;
  }
  if (o.update_rule != MEQ_RULE_MEQMUON && o.update_rule != MEQ_RULE_MUON) {
    *why = "update_rule must be MEQ_RULE_MEQMUON or MEQ_RULE_MUON";
    return false;
  }
  return true;
}

bool valid_kinds(const meq_shape* shapes, const int* kinds, int n, int rule, std::string* why) {
  if (!kinds) return true;
  for (int i = 0; i < n; ++i) {
    if (rule == MEQ_RULE_MUON && kinds[i] != KIND_HIDDEN) {
      *why = "MEQ_RULE_MUON (Eq. (6)) applies to hidden 2D weights only; entry " + std::to_string(i) + " is not one";
      return false;
    }
    if (kinds[i] < 0 || kinds[i] > 2) { *why = "kind of entry " + std::to_string(i) + " is not a meq_kind"; return false; }
    if (kinds[i] == KIND_VECTOR && shapes[i].rows != 1) {
      *why = "vector entry " + std::to_string(i) + " must have shape (1, d)";
      return false;
    }
  }
  return true;
}

bool valid_shapes(const meq_shape* shapes, int n, std::string* why) {
  if (n <= 0) { *why = "n must be positive"; return false; }
  if (!shapes) { *why = "shapes is NULL"; return false; }
  for (int i = 0; i < n; ++i) {
    const int64_t m = shapes[i].rows, c = shapes[i].cols;
    if (m <= 0 || c <= 0) { *why = "matrix " + std::to_string(i) + " has a non-positive dimension"; return false; }
    // TMA coordinates are 32-bit and the GEMM tile counters are int.
    if (m > (int64_t(1) << 20) || c > (int64_t(1) << 20) || m * c > (int64_t(1) << 34)) {
      *why = "matrix " + std::to_string(i) + " exceeds the supported size (dims <= 2^20, elements <= 2^34)";
      return false;
    }
  }
  return true;
}

float pow2_round(double x) { return static_cast<float>(std::ldexp(1.0, static_cast<int>(std::lround(std::log2(std::max(x, 1.0)))))); }

// Builds the whole plan (shapes -> groups, offsets, sizes). Allocation-free.
void plan(meq_state* st, Layout* L, int64_t* off_mom, int64_t* off_u, int64_t* off_vec4, int64_t* off_cpart,
          int64_t* off_partials, int64_t* off_counters, int64_t* off_x0s, int64_t* off_stats, int64_t* off_step,
          int64_t* off_err, int64_t* off_mats, int64_t* off_groups,
          std::vector<int64_t>* group_offs) {
  const int n = st->n;
  st->mats.assign(n, MatInfo{});
  std::map<std::tuple<int64_t, int64_t, int>, int> gmap;
  st->groups.clear();
  st->n_hidden = st->n_rows = st->n_two = 0;
  for (int i = 0; i < n; ++i) {
    const int64_t m = st->shapes[i].rows, c = st->shapes[i].cols;
    MatInfo& M = st->mats[i];
    M.m = m, M.n = c;
    M.s = std::min(m, c), M.l = std::max(m, c);
    M.trans = m > c ? 1 : 0;
    M.kind = st->kinds[i];
    M.group = -1;
    if (M.kind != KIND_HIDDEN) {
      ++st->n_rows;
      if (M.kind == KIND_TWO_SIDED) ++st->n_two;
      continue;
    }
    ++st->n_hidden;
    auto key = std::make_tuple(M.s, M.l, M.trans);
    auto it = gmap.find(key);
    int g;
    if (it == gmap.end()) {
      g = static_cast<int>(st->groups.size());
      gmap[key] = g;
      Group G;
      G.s = M.s, G.l = M.l;
      G.trans = M.trans;
      G.m = m, G.n = c, G.un = round_up(c, 8);  // whole 16-byte chunks per fp16 row
      G.lp = round_up(M.l, 64), G.sp = round_up(M.s, 64);
      G.alpha0 = std::min(pow2_round(std::sqrt(static_cast<double>(M.s) * static_cast<double>(M.l))), 16384.f);
      G.alpha = std::min(pow2_round(std::sqrt(static_cast<double>(M.l))), 16384.f);
      st->groups.push_back(G);
    } else {
      g = it->second;
    }
    M.group = g;
    M.gidx = st->groups[g].count++;
    st->groups[g].mats.push_back(i);
  }
  int64_t mom = 0, u = 0, vec = 0, parts = 0, chunks = 0, hchunks = 0, tiles = 0, rblks = 0, slabs = 0, xblks = 0;
  int64_t mslots = 0;
  for (auto& G : st->groups) {
    G.mbase = mslots;
    mslots += G.count;
  }
  for (auto& G : st->groups) {  // U is stored group by group: [count][m][un]
    G.u_base = u;
    u += round_up(G.count * G.m * G.un, 64);
    G.rpart_base = parts;
    parts += round_up(G.count * 2 * ((G.l + 255) / 256) * G.s, 64);
    G.cpart_base = parts;
    parts += round_up(G.count * ((G.s + 31) / 32) * G.l, 64);
  }
  for (int i = 0; i < n; ++i) {
    MatInfo& M = st->mats[i];
    M.mom_off = mom;
    mom += round_up(M.m * M.n, 64);
    M.vec_off = vec;
    vec += round_up(std::max(M.m, M.n), 64);
    M.chunk_begin = chunks;  // apply: every kind
    chunks += (M.m * M.n + kChunk - 1) / kChunk;
    M.hchunk_begin = hchunks;
    M.tile_begin = tiles;
    M.xblk_begin = xblks;
    M.rblk_begin = rblks;
    M.slab_begin = slabs;
    if (M.kind == KIND_HIDDEN) {
      const Group& G = st->groups[M.group];
      M.un = G.un;
      M.u_off = G.u_base + M.gidx * M.m * M.un;
      M.rpart_off = G.rpart_base + M.gidx * 2 * ((G.l + 255) / 256) * G.s;
      M.cpart_off = G.cpart_base + M.gidx * ((G.s + 31) / 32) * G.l;
      hchunks += (M.m * M.n + kChunk - 1) / kChunk;
      tiles += ((M.m + kCastTile - 1) / kCastTile) * ((M.n + kCastTile - 1) / kCastTile);
      // momentum + X_0: flat chunks of W, or 64 x 64 tiles when X_0 is W transposed
      xblks += M.trans ? ((M.m + kCastTile - 1) / kCastTile) * ((M.n + kCastTile - 1) / kCastTile)
                       : (M.m * M.n + kChunk - 1) / kChunk;
    } else {
      M.un = M.n;
      rblks += (M.m + 7) / 8;  // 8 rows (warps) per block
      if (M.kind == KIND_TWO_SIDED) {
        const int64_t ns = (M.m + kColSlab - 1) / kColSlab;
        M.cpart_off = parts;
        parts += round_up(ns * M.n, 64);
        slabs += ns * ((M.n + 255) / 256);  // blocks: slab x 256-column chunk
      }
    }
  }
  st->mom_floats = mom, st->u_halves = u, st->vec_floats = vec, st->parts_floats = parts;
  st->total_chunks = chunks, st->total_hchunks = hchunks, st->total_tiles = tiles, st->total_xblks = xblks;
  st->total_rblks = rblks, st->total_slabs = slabs;
  st->persistent_bytes = 0;
  for (int i = 0; i < n; ++i) st->persistent_bytes += 4 * st->mats[i].m * st->mats[i].n;

  *off_mom = L->add(mom * 4);
  *off_u = L->add(u * 2);
  *off_vec4 = L->add(vec * 4 * 4);  // r, c, s, t
  *off_cpart = L->add(parts * 4);
  *off_partials = L->add(std::max({hchunks, tiles, xblks}) * 4);  // per momentum chunk or block
  *off_counters = L->add(int64_t(n) * 4);  // per-matrix counters
  *off_x0s = L->add(int64_t(n) * 4 * 2);  // x0scale (cast pass) and the inverse norms (fused)
  *off_stats = L->add(int64_t(n) * sizeof(MatStats) + int64_t(n) * 2 * 8);  // stats, then direction counts
  st->step_bytes = sizeof(StepScalars) + 2 * int64_t(n) * sizeof(void*);
  *off_step = L->add(st->step_bytes);
  *off_err = L->add(64);  // ints 0: error word, 4: self-test flag, 8: non-finite flag, 12-13: tile queue
  *off_mats = L->add(int64_t(n) * sizeof(MatInfo));
  *off_groups = L->add(int64_t(st->groups.size()) * sizeof(GroupInfo));
  group_offs->clear();
  for (auto& G : st->groups) {
    const int64_t xb = G.count * G.s * G.lp * 2;
    const int64_t sb = G.count * G.s * G.sp;
    group_offs->push_back(L->add(xb));
    group_offs->push_back(L->add(xb));
    group_offs->push_back(L->add(sb * 2));
    group_offs->push_back(L->add(sb * 2));
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 3D tensor map over [count][rows][row_stride] elements of 2 or 4 bytes.
bool encode_map(CUtensorMap* m, void* base, int elem_bytes, int64_t inner, int64_t rows, int64_t count,
                int64_t row_stride_elems, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle swz) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(count)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(row_stride_elems * elem_bytes),
                           static_cast<cuuint64_t>(rows * row_stride_elems * elem_bytes)};
  cuuint32_t box[3] = {box_inner, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUtensorMapDataType dt = elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_UINT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  CUresult r = enc(m, dt, 3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}
constexpr CUtensorMapSwizzle SW128 = CU_TENSOR_MAP_SWIZZLE_128B;
constexpr CUtensorMapSwizzle SW64 = CU_TENSOR_MAP_SWIZZLE_64B;

// Tiles (tile_m rows x 256 columns) holding a 32 x 32 block on or above the diagonal.
int sym_tiles(int tiles_m, int tiles_n, int tile_m) {
  int t = 0;
  for (int tn = 0; tn < tiles_n; ++tn) t += std::min(tiles_m, ((tn + 1) * 256) / tile_m);
  return t;
}

// tcgen05 kind::f16 instruction descriptor: D fp32, A/B fp16 (0) or bf16 (1),
// A K-major, B K-major or MN-major, N = 256, M = 128 (one CTA) or 256 (pair).
uint32_t make_idesc(bool fp16, bool b_mn_major, int m) {
  const uint32_t fmt = fp16 ? 0u : 1u;
  return (1u << 4) | (fmt << 7) | (fmt << 10) | ((b_mn_major ? 1u : 0u) << 16) | ((256u >> 3) << 17) |
         ((static_cast<uint32_t>(m) >> 4) << 24);
}

bool iter_fp16(const meq_options& o, int k) { return k < 32 && ((o.ns_fp16_mask >> k) & 1u); }

// Prebuilds the GemmParams of every NS launch of one step.
bool build_gemm_plan(meq_state* st, std::string* why) {
  st->gemm.clear();
  st->gemm_grid.clear();
  const int K = st->opt.ns_steps;
  const int ng = static_cast<int>(st->groups.size());
  const int pair = st->opt.ns_cta_pair ? 2 : 1;
  const int tile_m = 128 * pair;
  const uint32_t b_rows = static_cast<uint32_t>(256 / pair);  // K-major B rows each CTA loads
  const bool fused = st->opt.ns_x0_fused != 0;
  // 16-bit formats: dA(k) of A_k (and of the polynomial's operands) is the
  // iteration's format; dX(k) of X_k (and of P_k, which multiplies it) too,
  // except that a fused X_0 is bf16 (written unnormalised by the momentum pass).
  auto dA = [&](int k) { return iter_fp16(st->opt, k); };
  auto dX = [&](int k) { return (fused && k == 0) ? false : iter_fp16(st->opt, k); };
  for (int k = 0; k < K; ++k) {
    const int cur = k & 1, nxt = cur ^ 1;
    for (int mode = MODE_GRAM; mode <= MODE_XUPD; ++mode) {
      const int real_mode = (mode == MODE_XUPD && k == K - 1) ? MODE_XLAST : mode;
      const bool in16 = mode == MODE_POLY ? dA(k) : dX(k);  // operand format of this launch
      for (int g0 = 0; g0 < ng; g0 += kMaxGroups) {
        GemmParams P;
        std::memset(&P, 0, sizeof(P));
        const int b_mn_major = (mode == MODE_XUPD) ? 1 : 0;
        const uint32_t idesc = make_idesc(in16, b_mn_major, tile_m);
        P.ca = st->opt.ns_a, P.cb = st->opt.ns_b, P.cc = st->opt.ns_c;
        P.err = st->d_err;
        P.sched = st->d_sched;
        P.timeout_ns = static_cast<unsigned long long>(static_cast<double>(st->opt.wait_timeout_ms) * 1e6);
        int tiles = 0;
        P.ngroups = std::min(kMaxGroups, ng - g0);
        for (int gi = 0; gi < P.ngroups; ++gi) {
          Group& G = st->groups[g0 + gi];
          GemmGroup& Q = P.g[gi];
          Q.mode = real_mode, Q.idesc = idesc, Q.b_mn_major = b_mn_major;
          // storage scale of X_k; a fused X_0 is unscaled and its 1/||H||_F is applied per matrix
          const float ak = (k == 0) ? (fused ? 1.0f : G.alpha0) : G.alpha;
          const bool per_matrix = fused && k == 0;
          Q.count = static_cast<int32_t>(G.count);
          Q.trans = G.trans;
          bool ok = true;
          const int64_t x_ld = G.lp * 2, x_ms = G.s * G.lp * 2;   // 16-bit X buffers, bytes
          const int64_t s_ld = G.sp * 2, s_ms = G.s * G.sp * 2;   // 16-bit A buffer, bytes
          if (mode == MODE_GRAM) {
            Q.M = (int32_t)G.s, Q.N = (int32_t)G.s, Q.K = (int32_t)G.l;
            Q.sym = 1;
            ok &= encode_map(&Q.tmA, G.x[cur], 2, G.l, G.s, G.count, G.lp, 64, 128, SW128);
            ok &= encode_map(&Q.tmB, G.x[cur], 2, G.l, G.s, G.count, G.lp, 64, b_rows, SW128);
            ok &= encode_map(&Q.tmO, G.a16, 2, G.s, G.s, G.count, G.sp, 32, 32, SW64);
            Q.tma_out = 1;
            Q.scale = 1.0f / (ak * ak);
            if (per_matrix) Q.minv = st->d_ginv + G.mbase, Q.minv_pow = 2;
            Q.out_fp16 = dA(k);
          } else if (mode == MODE_POLY) {
            Q.M = (int32_t)G.s, Q.N = (int32_t)G.s, Q.K = (int32_t)G.s;
            Q.sym = 1;
            ok &= encode_map(&Q.tmA, G.a16, 2, G.s, G.s, G.count, G.sp, 64, 128, SW128);
            ok &= encode_map(&Q.tmB, G.a16, 2, G.s, G.s, G.count, G.sp, 64, b_rows, SW128);
            ok &= encode_map(&Q.tmO, G.p16, 2, G.s, G.s, G.count, G.sp, 32, 32, SW64);
            Q.tma_out = 1;
            Q.aux = G.a16, Q.aux_ld = s_ld, Q.aux_mstride = s_ms;
            Q.scale = 1.0f;
            Q.out_fp16 = dX(k);
            Q.aux_fp16 = dA(k);
          } else {
            Q.M = (int32_t)G.s, Q.N = (int32_t)G.l, Q.K = (int32_t)G.s;
            Q.sym = 0;
            ok &= encode_map(&Q.tmA, G.p16, 2, G.s, G.s, G.count, G.sp, 64, 128, SW128);
            ok &= encode_map(&Q.tmB, G.x[cur], 2, G.l, G.s, G.count, G.lp, 64, 64, SW128);
            if (real_mode == MODE_XUPD) {
              Q.out = G.x[nxt], Q.out_ld = x_ld, Q.out_mstride = x_ms;
              Q.scale = G.alpha / ak;
              if (per_matrix) Q.minv = st->d_ginv + G.mbase, Q.minv_pow = 1;
              Q.out_fp16 = dX(k + 1);
            } else {
              Q.out = st->d_u + G.u_base, Q.out_ld = G.un * 2, Q.out_mstride = G.m * G.un * 2;
              Q.scale = 1.0f / ak;
              if (per_matrix) Q.minv = st->d_ginv + G.mbase, Q.minv_pow = 1;
              Q.out_fp16 = 1;  // fp16(kUScale * U)
              Q.rpart = st->d_parts + G.rpart_base;
              Q.cpart = st->d_parts + G.cpart_base;
            }
          }
          if (!ok) { *why = "cuTensorMapEncodeTiled failed"; return false; }
          Q.tiles_m = (int32_t)((Q.M + tile_m - 1) / tile_m);
          Q.tiles_n = (int32_t)((Q.N + 255) / 256);
          Q.tiles_per_mat = Q.sym ? sym_tiles(Q.tiles_m, Q.tiles_n, tile_m) : Q.tiles_m * Q.tiles_n;
          // Dense products walk bands of tile rows column by column; a band's
          // row panels of P (band * tile_m * K 16-bit values) stay within 32 MB,
          // about a quarter of L2, so every P panel is read from DRAM once.
          Q.band = static_cast<int32_t>(
              std::max<int64_t>(1, std::min<int64_t>(Q.tiles_m, (int64_t(32) << 20) / (int64_t(tile_m) * Q.K * 2))));
          Q.tile_begin = tiles;
          const int64_t t = int64_t(Q.tiles_per_mat) * Q.count;
          if (tiles + t > (int64_t(1) << 30)) { *why = "too many GEMM tiles in one launch"; return false; }
          tiles += static_cast<int>(t);
        }
        P.total_tiles = tiles;
        // Each launch walks the matrices in the opposite order of the one
        // before it (the X_0 cast writes in forward order), so it begins with
        // the outputs still resident in L2.
        P.reverse = (st->gemm.size() % 2 == 0) ? 1 : 0;
        P.debug_skip_load = (st->opt.debug_skip_load && st->gemm.empty()) ? 1 : 0;
        st->gemm.push_back(P);
        // persistent grid: one CTA (pair) per SM (pair of SMs), never more than the tiles
        st->gemm_grid.push_back(pair * std::max(1, std::min(tiles, st->num_sms / pair)));
      }
    }
  }
  return true;
}

}  // namespace

extern "C" {

void meq_default_options(meq_options* o) {
  if (!o) return;
  std::memset(o, 0, sizeof(*o));
  o->rho = 0.2f;
  o->ns_steps = 5;
  o->ns_a = 3.4445f;
  o->ns_b = -4.7750f;
  o->ns_c = 2.0315f;
  o->nesterov = 0;
  o->ns_fp16_mask = 0xFFFFFFFFu;
  o->tie_atol = 1e-6f;
  o->use_graph = 1;
  o->workspace_limit_bytes = 0;
  o->wait_timeout_ms = 4000.f;
  o->ns_cta_pair = 1;
  o->ns_x0_fused = 1;
  o->debug_canaries = 0;
  o->debug_skip_load = 0;
}

const char* meq_status_string(meq_status s) {
  switch (s) {
    case MEQ_OK: return "MEQ_OK";
    case MEQ_ERR_INVALID_ARG: return "MEQ_ERR_INVALID_ARG";
    case MEQ_ERR_OOM: return "MEQ_ERR_OOM";
    case MEQ_ERR_CUDA: return "MEQ_ERR_CUDA";
    case MEQ_ERR_NONFINITE: return "MEQ_ERR_NONFINITE";
    case MEQ_ERR_TIMEOUT: return "MEQ_ERR_TIMEOUT";
    case MEQ_ERR_UNSUPPORTED: return "MEQ_ERR_UNSUPPORTED";
    case MEQ_ERR_CORRUPTED: return "MEQ_ERR_CORRUPTED";
  }
  return "MEQ_ERR_UNKNOWN";
}

const char* meq_last_error(const meq_state* st) { return st ? st->last_error.c_str() : g_init_error.c_str(); }

meq_status meq_state_bytes(const meq_shape* shapes, int n, const meq_options* opt, size_t* persistent, size_t* workspace) {
  return meq_state_bytes_kinds(shapes, nullptr, n, opt, persistent, workspace);
}

meq_status meq_state_bytes_kinds(const meq_shape* shapes, const int* kinds, int n, const meq_options* opt,
                                 size_t* persistent, size_t* workspace) {
  meq_options o;
  if (opt) o = *opt; else meq_default_options(&o);
  std::string why;
  if (!valid_shapes(shapes, n, &why) || !valid_options(o, &why) || !valid_kinds(shapes, kinds, n, o.update_rule, &why))
    return fail(nullptr, MEQ_ERR_INVALID_ARG, why);
  meq_state tmp;
  tmp.n = n;
  tmp.shapes.assign(shapes, shapes + n);
  tmp.kinds.assign(n, KIND_HIDDEN);
  if (kinds) tmp.kinds.assign(kinds, kinds + n);
  tmp.opt = o;
  Layout L(o.debug_canaries != 0);
  int64_t a[13];
  std::vector<int64_t> goffs;
  plan(&tmp, &L, &a[0], &a[1], &a[2], &a[3], &a[4], &a[5], &a[6], &a[7], &a[8], &a[9], &a[10], &a[11], &goffs);
  if (persistent) *persistent = static_cast<size_t>(tmp.persistent_bytes);
  if (workspace) *workspace = static_cast<size_t>(L.total - tmp.persistent_bytes);
  return MEQ_OK;
}

meq_status meq_init_state(const meq_shape* shapes, int n, const meq_options* opt, void* cuda_stream, meq_state** out) {
  return meq_init_state_kinds(shapes, nullptr, n, opt, cuda_stream, out);
}

meq_status meq_init_state_kinds(const meq_shape* shapes, const int* kinds, int n, const meq_options* opt,
                                void* cuda_stream, meq_state** out) {
  if (!out) return fail(nullptr, MEQ_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  meq_options o;
  if (opt) o = *opt; else meq_default_options(&o);
  std::string why;
  if (!valid_shapes(shapes, n, &why) || !valid_options(o, &why) || !valid_kinds(shapes, kinds, n, o.update_rule, &why))
    return fail(nullptr, MEQ_ERR_INVALID_ARG, why);

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(nullptr, MEQ_ERR_UNSUPPORTED, std::string("no CUDA device: ") + cudaGetErrorString(e));
  cudaDeviceProp prop;
  e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) return fail(nullptr, MEQ_ERR_CUDA, std::string("cudaGetDeviceProperties: ") + cudaGetErrorString(e));
  if (prop.major != 10 || prop.minor != 3)
    return fail(nullptr, MEQ_ERR_UNSUPPORTED,
                "this library is built for sm_103a (GB300); device is sm_" + std::to_string(prop.major) + std::to_string(prop.minor));
  if (prop.sharedMemPerBlockOptin < static_cast<size_t>(ns_gemm_smem_bytes(o.ns_cta_pair ? 2 : 1)))
    return fail(nullptr, MEQ_ERR_UNSUPPORTED, "not enough opt-in shared memory per block");
  if (!get_encode()) return fail(nullptr, MEQ_ERR_UNSUPPORTED, "cuTensorMapEncodeTiled is not available from the driver");

  e = prepare_ns_gemm();
  if (e != cudaSuccess) return fail(nullptr, MEQ_ERR_CUDA, std::string("cudaFuncSetAttribute: ") + cudaGetErrorString(e));

  meq_state* st = new meq_state();
  st->n = n;
  st->shapes.assign(shapes, shapes + n);
  st->kinds.assign(n, KIND_HIDDEN);
  if (kinds) st->kinds.assign(kinds, kinds + n);
  st->opt = o;
  st->device = dev;
  st->num_sms = prop.multiProcessorCount;

  Layout L(o.debug_canaries != 0);
  int64_t off_mom, off_u, off_vec4, off_cpart, off_partials, off_counters, off_x0s, off_stats, off_step, off_err, off_mats,
      off_groups;
  std::vector<int64_t> goffs;
  plan(st, &L, &off_mom, &off_u, &off_vec4, &off_cpart, &off_partials, &off_counters, &off_x0s, &off_stats, &off_step,
       &off_err, &off_mats, &off_groups, &goffs);
  if (o.workspace_limit_bytes > 0 && L.total > o.workspace_limit_bytes) {
    delete st;
    return fail(nullptr, MEQ_ERR_OOM, "state needs " + std::to_string(L.total) + " bytes, above workspace_limit_bytes");
  }
  e = cudaMalloc(reinterpret_cast<void**>(&st->arena), static_cast<size_t>(L.total));
  if (e != cudaSuccess) {
    cudaGetLastError();
    delete st;
    return fail(nullptr, MEQ_ERR_OOM, "cudaMalloc of " + std::to_string(L.total) + " bytes failed");
  }
  st->arena_bytes = L.total;
  char* A = st->arena;
  st->d_mom = reinterpret_cast<float*>(A + off_mom);
  st->d_u = reinterpret_cast<uint16_t*>(A + off_u);
  st->d_rvec = reinterpret_cast<float*>(A + off_vec4);
  st->d_cvec = st->d_rvec + st->vec_floats;
  st->d_svec = st->d_cvec + st->vec_floats;
  st->d_tvec = st->d_svec + st->vec_floats;
  st->d_parts = reinterpret_cast<float*>(A + off_cpart);
  st->d_partials = reinterpret_cast<float*>(A + off_partials);
  st->d_counters = reinterpret_cast<unsigned int*>(A + off_counters);
  st->d_x0scale = reinterpret_cast<float*>(A + off_x0s);
  st->d_ginv = st->d_x0scale + n;
  st->d_stats = reinterpret_cast<MatStats*>(A + off_stats);
  st->d_dircount = reinterpret_cast<unsigned long long*>(st->d_stats + n);
  st->d_step = A + off_step;
  st->d_err = reinterpret_cast<int*>(A + off_err);
  st->d_flag = st->d_err + 4;
  st->d_nonfinite = st->d_err + 8;
  st->d_sched = st->d_err + 12;
  st->d_mats = reinterpret_cast<MatInfo*>(A + off_mats);
  st->d_groups = reinterpret_cast<GroupInfo*>(A + off_groups);
  for (size_t g = 0; g < st->groups.size(); ++g) {
    Group& G = st->groups[g];
    G.x[0] = reinterpret_cast<uint16_t*>(A + goffs[4 * g + 0]);
    G.x[1] = reinterpret_cast<uint16_t*>(A + goffs[4 * g + 1]);
    G.a16 = reinterpret_cast<uint16_t*>(A + goffs[4 * g + 2]);
    G.p16 = reinterpret_cast<uint16_t*>(A + goffs[4 * g + 3]);
  }

  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  std::vector<GroupInfo> gi(st->groups.size());
  for (size_t g = 0; g < st->groups.size(); ++g) {
    const Group& G = st->groups[g];
    gi[g].s = G.s, gi[g].l = G.l, gi[g].lp = G.lp, gi[g].sp = G.sp, gi[g].count = G.count;
    gi[g].x0 = G.x[0];
    gi[g].alpha0 = G.alpha0;
    gi[g].mbase = G.mbase;
  }
  bool ok = cudaMemsetAsync(st->arena, 0, static_cast<size_t>(L.total), s) == cudaSuccess;
  st->guard_ranges = L.guard_ranges;
  for (const auto& g : st->guard_ranges)
    ok = ok && cudaMemsetAsync(st->arena + g.first, kGuardByte, static_cast<size_t>(g.second), s) == cudaSuccess;
  ok = ok && cudaMemcpyAsync(st->d_mats, st->mats.data(), sizeof(MatInfo) * n, cudaMemcpyHostToDevice, s) == cudaSuccess;
  ok = ok && cudaMemcpyAsync(st->d_groups, gi.data(), sizeof(GroupInfo) * gi.size(), cudaMemcpyHostToDevice, s) == cudaSuccess;
  ok = ok && cudaStreamSynchronize(s) == cudaSuccess;
  if (!ok) {
    cudaError_t ee = cudaGetLastError();
    cudaFree(st->arena);
    delete st;
    return fail(nullptr, MEQ_ERR_CUDA, std::string("initialising the state failed: ") + cudaGetErrorString(ee));
  }

  if (!build_gemm_plan(st, &why)) {
    cudaFree(st->arena);
    delete st;
    return fail(nullptr, MEQ_ERR_UNSUPPORTED, why);
  }
  LaunchCtx& C = st->ctx;
  C.mats = st->d_mats;
  C.nmat = n;
  C.groups = st->d_groups;
  C.mom = st->d_mom;
  C.sc = reinterpret_cast<const StepScalars*>(st->d_step);
  C.params = reinterpret_cast<float* const*>(st->d_step + sizeof(StepScalars));
  C.grads = reinterpret_cast<const float* const*>(st->d_step + sizeof(StepScalars) + n * sizeof(void*));
  C.partials = st->d_partials;
  C.counters = st->d_counters;
  C.x0scale = st->d_x0scale;
  C.ginv = st->d_ginv;
  C.uslab = st->d_u;
  C.parts = st->d_parts;
  C.rvec = st->d_rvec;
  C.cvec = st->d_cvec;
  C.svec = st->d_svec;
  C.tvec = st->d_tvec;
  C.stats = st->d_stats;
  C.dircount = st->d_dircount;
  C.nonfinite = st->d_nonfinite;
  C.total_chunks = st->total_chunks;
  C.total_hchunks = st->total_hchunks;
  C.total_tiles = st->total_tiles;
  C.total_xblks = st->total_xblks;
  C.n_hidden = st->n_hidden;
  C.total_rblks = st->total_rblks;
  C.total_slabs = st->total_slabs;
  st->kernels_per_step = (st->n_hidden ? 2 : 0) + (st->n_rows ? 1 : 0) + (st->n_two ? 1 : 0) + 2 +
                         static_cast<int>(st->gemm.size());
  st->step_host.assign(static_cast<size_t>(st->step_bytes), 0);
  st->last_stream = s;
  *out = st;
  return MEQ_OK;
}


static void drop_profile(meq_state* st) {
  for (auto& v : st->prof_events)
    for (auto x : v) cudaEventDestroy(x);
  st->prof_events.clear();
  if (st->gexec_prof) cudaGraphExecDestroy(st->gexec_prof);
  if (st->graph_prof) cudaGraphDestroy(st->graph_prof);
  st->gexec_prof = nullptr;
  st->graph_prof = nullptr;
  for (auto x : st->prof_graph_events) cudaEventDestroy(x);
  st->prof_graph_events.clear();
  for (double& x : st->prof_sum) x = 0;
  st->prof_graph_steps = 0;
}

// One open NVTX range at a time (closed on the next stage and on scope exit).
struct NvtxStages {
  bool open = false;
  void next(const char* name) {
    if (open) nvtxRangePop();
    open = name != nullptr;
    if (open) nvtxRangePushA(name);
  }
  ~NvtxStages() { next(nullptr); }
};
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};

enum StepParts : int { PART_PREPARE = 1, PART_APPLY = 2, PART_ALL = 3 };

static meq_status enqueue_kernels(meq_state* st, cudaStream_t s, cudaEvent_t* ev = nullptr, int parts = PART_ALL,
                                  bool capturing = false) {
  const LaunchCtx& C = st->ctx;
  // NVTX ranges name the stages on the host timeline (each eager enqueue, or
  // the capture of the graph); CUDA events time them on the stream.
  // (nested in the "meq_step" range: ncu selects e.g. --nvtx-include "meq_step/ns_gemm/")
  static const char* const kStage[5] = {"momentum", "cast_x0", "ns_gemm", "statistics", "apply"};
  NvtxStages stage;
  auto mark = [&](int i) {
    // under stream capture, only an external record becomes a node that
    // records the event on each replay (a plain one just orders the capture)
    if (ev) cudaEventRecordWithFlags(ev[i], s, capturing ? cudaEventRecordExternal : cudaEventRecordDefault);
    stage.next(i < 5 ? kStage[i] : nullptr);
  };
  cudaError_t e = cudaSuccess;
  if (!(parts & PART_PREPARE)) {
    mark(4);
    e = launch_apply(C, s);
    return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "apply launch");
  }
  mark(0);
  const bool fused = st->opt.ns_x0_fused != 0;
  if (st->n_hidden) {
    e = fused ? launch_momentum_x0(C, s) : launch_momentum_norm(C, s);
    if (e != cudaSuccess) return cuda_fail(st, e, "momentum launch");
    if (fused) {
      e = launch_x0norm(C, s);
      if (e != cudaSuccess) return cuda_fail(st, e, "x0norm launch");
    }
  }
  if (st->n_rows) {
    e = launch_rows(C, s);
    if (e != cudaSuccess) return cuda_fail(st, e, "rows launch");
  }
  mark(1);
  if (st->n_hidden && !fused) {
    e = launch_cast_x0(C, iter_fp16(st->opt, 0), s);
    if (e != cudaSuccess) return cuda_fail(st, e, "cast_x0 launch");
  }
  mark(2);
  for (size_t i = 0; i < st->gemm.size(); ++i) {
    e = launch_ns_gemm(st->gemm[i], st->gemm_grid[i], st->opt.ns_cta_pair ? 2 : 1, s);
    if (e != cudaSuccess) return cuda_fail(st, e, "ns_gemm launch");
  }
  mark(3);
  if (st->n_two) {
    e = launch_colpart(C, s);
    if (e != cudaSuccess) return cuda_fail(st, e, "colpart launch");
  }
  e = launch_stats(C, s);
  if (e != cudaSuccess) return cuda_fail(st, e, "finalize launch");
  mark(4);
  if (!(parts & PART_APPLY)) return MEQ_OK;
  e = launch_apply(C, s);
  if (e != cudaSuccess) return cuda_fail(st, e, "apply launch");
  mark(5);
  return MEQ_OK;
}

static meq_status capture_graph(meq_state* st, int parts, cudaGraph_t* graph, cudaGraphExec_t* gexec,
                                cudaEvent_t* ev = nullptr) {
  cudaStream_t cs = nullptr;
  cudaError_t e = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamCreate");
  e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) {
    cudaStreamDestroy(cs);
    return cuda_fail(st, e, "cudaStreamBeginCapture");
  }
  meq_status ms = enqueue_kernels(st, cs, ev, parts, true);
  cudaGraph_t g = nullptr;
  e = cudaStreamEndCapture(cs, &g);
  cudaStreamDestroy(cs);
  if (ms != MEQ_OK) {
    if (g) cudaGraphDestroy(g);
    return ms;
  }
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamEndCapture");
  cudaGraphExec_t x = nullptr;
  e = cudaGraphInstantiate(&x, g, 0);
  if (e != cudaSuccess) {
    cudaGraphDestroy(g);
    return cuda_fail(st, e, "cudaGraphInstantiate");
  }
  *graph = g;
  *gexec = x;
  return MEQ_OK;
}

// Checks shapes and scalars and uploads the per-step block (scalars, then
// the params and grads pointer tables; params may be NULL: that table is
// left as it is).
static meq_status upload_step(meq_state* st, float* const* params, const float* const* grads, const meq_shape* shapes,
                              int n, float lr, float momentum, float weight_decay, float eps, cudaStream_t s) {
  if (!grads || !shapes) return fail(st, MEQ_ERR_INVALID_ARG, "grads and shapes must be non-NULL");
  if (n != st->n) return fail(st, MEQ_ERR_INVALID_ARG, "n differs from the init-time shape list");
  for (int i = 0; i < n; ++i) {
    if (shapes[i].rows != st->shapes[i].rows || shapes[i].cols != st->shapes[i].cols)
      return fail(st, MEQ_ERR_INVALID_ARG, "shape of matrix " + std::to_string(i) + " differs from init");
    if ((params && !params[i]) || !grads[i])
      return fail(st, MEQ_ERR_INVALID_ARG, "NULL params/grads pointer at " + std::to_string(i));
    if ((params && (reinterpret_cast<uintptr_t>(params[i]) & 15u)) || (reinterpret_cast<uintptr_t>(grads[i]) & 15u))
      return fail(st, MEQ_ERR_INVALID_ARG, "params/grads pointer " + std::to_string(i) + " is not 16-byte aligned");
  }
  if (!std::isfinite(lr) || !std::isfinite(momentum) || !std::isfinite(weight_decay) || !(eps >= 0.f) || !std::isfinite(eps))
    return fail(st, MEQ_ERR_INVALID_ARG, "lr, momentum, weight_decay must be finite and eps >= 0");
  StepScalars sc;
  std::memset(&sc, 0, sizeof(sc));
  sc.lr = lr, sc.mu = momentum, sc.wd = weight_decay, sc.eps = eps;
  sc.rho = st->opt.rho, sc.tie_atol = st->opt.tie_atol, sc.nesterov = st->opt.nesterov;
  sc.rule = st->opt.update_rule;
  char* h = st->step_host.data();
  std::memcpy(h, &sc, sizeof(sc));
  if (params) std::memcpy(h + sizeof(sc), params, n * sizeof(void*));
  std::memcpy(h + sizeof(sc) + n * sizeof(void*), grads, n * sizeof(void*));
  // Pageable source: the call returns once the bytes are staged, so the
  // host buffer can be reused by the next step right away.
  cudaError_t e;
  if (params) {
    e = cudaMemcpyAsync(st->d_step, h, static_cast<size_t>(st->step_bytes), cudaMemcpyHostToDevice, s);
  } else {
    e = cudaMemcpyAsync(st->d_step, h, sizeof(sc), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(st->d_step + sizeof(sc) + n * sizeof(void*), h + sizeof(sc) + n * sizeof(void*),
                          n * sizeof(void*), cudaMemcpyHostToDevice, s);
  }
  if (e != cudaSuccess) return cuda_fail(st, e, "step upload");
  st->last_stream = s;
  return MEQ_OK;
}

// Runs the given parts of the step on s: eagerly, or from its graph.
static meq_status run_parts(meq_state* st, int parts, cudaStream_t s) {
  if (st->opt.use_graph) {
    cudaGraph_t* g = parts == PART_ALL ? &st->graph : parts == PART_PREPARE ? &st->graph_prep : &st->graph_apply;
    cudaGraphExec_t* x = parts == PART_ALL ? &st->gexec : parts == PART_PREPARE ? &st->gexec_prep : &st->gexec_apply;
    if (!*x) {
      meq_status ms = capture_graph(st, parts, g, x);
      if (ms != MEQ_OK) return ms;
      if (parts == PART_ALL) st->graph_ready = true;
    }
    cudaError_t e = cudaGraphLaunch(*x, s);
    return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "cudaGraphLaunch");
  }
  return enqueue_kernels(st, s, nullptr, parts);
}

meq_status meq_step(float* const* params, const float* const* grads, meq_state* st, const meq_shape* shapes, int n,
                    float lr, float momentum, float weight_decay, float eps, void* cuda_stream) {
  NvtxRange range("meq_step");
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (!params) return fail(st, MEQ_ERR_INVALID_ARG, "params must be non-NULL");
  if (st->prepared) return fail(st, MEQ_ERR_INVALID_ARG, "a meq_step_prepare is waiting for its meq_step_apply");
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  meq_status ms = upload_step(st, params, grads, shapes, n, lr, momentum, weight_decay, eps, s);
  if (ms != MEQ_OK) return ms;
  if (st->profiling && st->opt.use_graph) {
    // the step's own graph, with an event-record node between its phases;
    // each replay is waited for and its phase times added up
    if (!st->gexec_prof) {
      st->prof_graph_events.assign(6, nullptr);
      for (auto& x : st->prof_graph_events) {
        cudaError_t e = cudaEventCreate(&x);
        if (e != cudaSuccess) return cuda_fail(st, e, "cudaEventCreate");
      }
      meq_status cs = capture_graph(st, PART_ALL, &st->graph_prof, &st->gexec_prof, st->prof_graph_events.data());
      if (cs != MEQ_OK) return cs;
    }
    cudaError_t e = cudaGraphLaunch(st->gexec_prof, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    for (int p = 0; e == cudaSuccess && p < 5; ++p) {
      float ms = 0.f;
      e = cudaEventElapsedTime(&ms, st->prof_graph_events[p], st->prof_graph_events[p + 1]);
      st->prof_sum[p] += ms;
    }
    if (e != cudaSuccess) return cuda_fail(st, e, "profiled graph replay");
    ++st->prof_graph_steps;
    return MEQ_OK;
  }
  if (st->profiling) {
    std::vector<cudaEvent_t> ev(6, nullptr);
    for (auto& x : ev) {
      cudaError_t e = cudaEventCreate(&x);
      if (e != cudaSuccess) return cuda_fail(st, e, "cudaEventCreate");
    }
    st->prof_events.push_back(ev);
    return enqueue_kernels(st, s, st->prof_events.back().data());
  }
  return run_parts(st, PART_ALL, s);
}

meq_status meq_step_prepare(const float* const* grads, meq_state* st, const meq_shape* shapes, int n, float lr,
                            float momentum, float weight_decay, float eps, void* cuda_stream) {
  NvtxRange range("meq_step");
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (st->prepared) return fail(st, MEQ_ERR_INVALID_ARG, "meq_step_prepare twice without meq_step_apply");
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  meq_status ms = upload_step(st, nullptr, grads, shapes, n, lr, momentum, weight_decay, eps, s);
  if (ms != MEQ_OK) return ms;
  ms = run_parts(st, PART_PREPARE, s);
  if (ms == MEQ_OK) st->prepared = true;
  return ms;
}

meq_status meq_step_apply(float* const* params, meq_state* st, void* cuda_stream) {
  NvtxRange range("meq_step");
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (!st->prepared) return fail(st, MEQ_ERR_INVALID_ARG, "meq_step_apply without a meq_step_prepare");
  if (!params) return fail(st, MEQ_ERR_INVALID_ARG, "params must be non-NULL");
  for (int i = 0; i < st->n; ++i) {
    if (!params[i]) return fail(st, MEQ_ERR_INVALID_ARG, "NULL params pointer at " + std::to_string(i));
    if (reinterpret_cast<uintptr_t>(params[i]) & 15u)
      return fail(st, MEQ_ERR_INVALID_ARG, "params pointer " + std::to_string(i) + " is not 16-byte aligned");
  }
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  char* h = st->step_host.data() + sizeof(StepScalars);
  std::memcpy(h, params, st->n * sizeof(void*));
  cudaError_t e = cudaMemcpyAsync(st->d_step + sizeof(StepScalars), h, st->n * sizeof(void*), cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(st, e, "step upload");
  st->last_stream = s;
  meq_status ms = run_parts(st, PART_APPLY, s);
  if (ms == MEQ_OK) st->prepared = false;
  return ms;
}

meq_status meq_sync(meq_state* st) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  cudaError_t e = cudaStreamSynchronize(st->last_stream);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamSynchronize");
  int err = 0;
  e = cudaMemcpy(&err, st->d_err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(st, e, "reading the device error word");
  if (err != 0) {
    int zero[2] = {0, 0};
    cudaMemcpy(st->d_err, zero, sizeof(int), cudaMemcpyHostToDevice);
    // a launch that returned early may have left its tile queue partly used
    cudaMemcpy(st->d_sched, zero, 2 * sizeof(int), cudaMemcpyHostToDevice);
    char buf[96];
    std::snprintf(buf, sizeof(buf), "device-side bounded wait expired (code 0x%x)", err);
    return fail(st, MEQ_ERR_TIMEOUT, buf);
  }
  int bad = 0;
  e = cudaMemcpy(&bad, st->d_nonfinite, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(st, e, "reading the non-finite flag");
  if (bad != 0) {
    int zero = 0;
    cudaMemcpy(st->d_nonfinite, &zero, sizeof(int), cudaMemcpyHostToDevice);
    return fail(st, MEQ_ERR_NONFINITE, "non-finite momentum (gradient, or a previous non-finite step) in entry " +
                                           std::to_string(bad - 1));
  }
  return MEQ_OK;
}

meq_status meq_free(meq_state* st) {
  if (!st) return MEQ_OK;
  cudaStreamSynchronize(st->last_stream);
  drop_profile(st);
  if (st->gexec) cudaGraphExecDestroy(st->gexec);
  if (st->graph) cudaGraphDestroy(st->graph);
  if (st->gexec_prep) cudaGraphExecDestroy(st->gexec_prep);
  if (st->graph_prep) cudaGraphDestroy(st->graph_prep);
  if (st->gexec_apply) cudaGraphExecDestroy(st->gexec_apply);
  if (st->graph_apply) cudaGraphDestroy(st->graph_apply);
  if (st->arena) cudaFree(st->arena);
  delete st;
  return MEQ_OK;
}

static meq_status check_index(meq_state* st, int i) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (i < 0 || i >= st->n) return fail(st, MEQ_ERR_INVALID_ARG, "matrix index out of range");
  cudaError_t e = cudaStreamSynchronize(st->last_stream);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamSynchronize");
  return MEQ_OK;
}

meq_status meq_read_momentum(meq_state* st, int i, float* dst) {
  meq_status ms = check_index(st, i);
  if (ms != MEQ_OK) return ms;
  if (!dst) return fail(st, MEQ_ERR_INVALID_ARG, "dst is NULL");
  const MatInfo& M = st->mats[i];
  cudaError_t e = cudaMemcpy(dst, st->d_mom + M.mom_off, M.m * M.n * sizeof(float), cudaMemcpyDefault);
  return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "cudaMemcpy");
}

meq_status meq_write_momentum(meq_state* st, int i, const float* src) {
  meq_status ms = check_index(st, i);
  if (ms != MEQ_OK) return ms;
  if (!src) return fail(st, MEQ_ERR_INVALID_ARG, "src is NULL");
  const MatInfo& M = st->mats[i];
  cudaError_t e = cudaMemcpy(st->d_mom + M.mom_off, src, M.m * M.n * sizeof(float), cudaMemcpyDefault);
  return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "cudaMemcpy");
}

meq_status meq_read_ns_output(meq_state* st, int i, float* dst) {
  meq_status ms = check_index(st, i);
  if (ms != MEQ_OK) return ms;
  if (!dst) return fail(st, MEQ_ERR_INVALID_ARG, "dst is NULL");
  if (st->kinds[i] != KIND_HIDDEN) return fail(st, MEQ_ERR_INVALID_ARG, "entry has no Newton-Schulz output (not hidden)");
  const MatInfo& M = st->mats[i];
  std::vector<uint16_t> h(static_cast<size_t>(M.m * M.n));
  cudaError_t e = cudaMemcpy2D(h.data(), M.n * sizeof(uint16_t), st->d_u + M.u_off, M.un * sizeof(uint16_t),
                               M.n * sizeof(uint16_t), M.m, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaMemcpy2D");
  std::vector<float> f(h.size());
  for (size_t k = 0; k < h.size(); ++k) f[k] = half_bits_to_float(h[k]) * (1.0f / kUScale);
  e = cudaMemcpy(dst, f.data(), f.size() * sizeof(float), cudaMemcpyDefault);
  return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "cudaMemcpy");
}

meq_status meq_read_update(meq_state* st, int i, float* dst) {
  meq_status ms = check_index(st, i);
  if (ms != MEQ_OK) return ms;
  if (!dst) return fail(st, MEQ_ERR_INVALID_ARG, "dst is NULL");
  const MatInfo& M = st->mats[i];
  const size_t bytes = static_cast<size_t>(M.m * M.n) * sizeof(float);
  // the kernel runs (and any temporary lives) on the state's device, whichever is current
  int prev_dev = st->device;
  cudaError_t e = cudaGetDevice(&prev_dev);
  if (e == cudaSuccess && prev_dev != st->device) e = cudaSetDevice(st->device);
  if (e != cudaSuccess) return cuda_fail(st, e, "selecting the state's device");
  struct Restore {
    int dev, cur;
    ~Restore() {
      if (dev != cur) cudaSetDevice(dev);
    }
  } restore{prev_dev, st->device};
  cudaPointerAttributes pa{};
  e = cudaPointerGetAttributes(&pa, dst);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaPointerGetAttributes");
  const bool on_device = (pa.type == cudaMemoryTypeDevice || pa.type == cudaMemoryTypeManaged) && pa.device == st->device;
  float* out = dst;
  if (!on_device) {
    e = cudaMalloc(reinterpret_cast<void**>(&out), bytes);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(st, MEQ_ERR_OOM, "scratch allocation for meq_read_update failed");
    }
  }
  e = launch_update(st->ctx, M, i, out, st->last_stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st->last_stream);
  if (e == cudaSuccess && !on_device) e = cudaMemcpy(dst, out, bytes, cudaMemcpyDefault);
  if (!on_device) cudaFree(out);
  return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "meq_read_update");
}

meq_status meq_read_stats(meq_state* st, int i, float* r, float* c, double* gamma_r, double* gamma_c, int* direction) {
  meq_status ms = check_index(st, i);
  if (ms != MEQ_OK) return ms;
  const MatInfo& M = st->mats[i];
  cudaError_t e = cudaSuccess;
  if (r) e = cudaMemcpy(r, st->d_rvec + M.vec_off, M.m * sizeof(float), cudaMemcpyDefault);
  if (e == cudaSuccess && c) e = cudaMemcpy(c, st->d_cvec + M.vec_off, M.n * sizeof(float), cudaMemcpyDefault);
  MatStats hs;
  if (e == cudaSuccess) e = cudaMemcpy(&hs, st->d_stats + i, sizeof(hs), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaMemcpy");
  if (gamma_r) *gamma_r = hs.gamma_r;
  if (gamma_c) *gamma_c = hs.gamma_c;
  if (direction) *direction = hs.direction;
  return MEQ_OK;
}

meq_status meq_ns_cv_trajectory(const float* h, int64_t rows, int64_t cols, int steps, float eps,
                                const meq_options* opt, double* gamma_r, double* gamma_c, void* cuda_stream) {
  if (!h || !gamma_r || !gamma_c) return fail(nullptr, MEQ_ERR_INVALID_ARG, "h, gamma_r and gamma_c must not be NULL");
  if (reinterpret_cast<uintptr_t>(h) & 15u) return fail(nullptr, MEQ_ERR_INVALID_ARG, "h is not 16-byte aligned");
  if (steps < 0 || steps > 32) return fail(nullptr, MEQ_ERR_INVALID_ARG, "steps must be in 0..32");
  if (!(eps >= 0.f) || !std::isfinite(eps)) return fail(nullptr, MEQ_ERR_INVALID_ARG, "eps must be finite and >= 0");
  meq_shape shape{rows, cols};
  std::string why;
  if (!valid_shapes(&shape, 1, &why)) return fail(nullptr, MEQ_ERR_INVALID_ARG, why);
  meq_options o;
  if (opt) o = *opt; else meq_default_options(&o);
  o.update_rule = MEQ_RULE_MEQMUON;
  o.use_graph = 0;
  o.ns_steps = 1;
  if (!valid_options(o, &why)) return fail(nullptr, MEQ_ERR_INVALID_ARG, why);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  // scratch: W (rows x cols, left unchanged by lr = 0), r, c, the two CVs and
  // the direction, then the statistics kernels' partial sums
  const int64_t wb = round_up(rows * cols * 4, 256), rb = round_up(rows * 4, 256), cb = round_up(cols * 4, 256);
  const int64_t pb = round_up(row_col_stats_scratch_floats(rows, cols) * 4, 256);
  char* tmp = nullptr;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&tmp), static_cast<size_t>(wb + rb + cb + 256 + pb));
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(nullptr, MEQ_ERR_OOM, "scratch allocation failed");
  }
  float* w = reinterpret_cast<float*>(tmp);
  float* r = reinterpret_cast<float*>(tmp + wb);
  float* c = reinterpret_cast<float*>(tmp + wb + rb);
  double* g = reinterpret_cast<double*>(tmp + wb + rb + cb);
  int* d = reinterpret_cast<int*>(g + 2);
  float* parts = reinterpret_cast<float*>(tmp + wb + rb + cb + 256);
  meq_status ms = MEQ_OK;
  e = cudaMemsetAsync(w, 0, static_cast<size_t>(rows * cols * 4), s);
  if (e != cudaSuccess) ms = cuda_fail(nullptr, e, "cudaMemsetAsync");
  // k = 0: the statistics of X_0 = H / ||H||_F (the threshold eps applies to
  // the RMS of X_0, as for every later iterate), in this call's own scratch
  if (ms == MEQ_OK) {
    const char* what = "";
    e = launch_row_col_stats(h, rows, cols, eps, o.tie_atol, 1, parts, r, c, g, d, s, &what);
    if (e != cudaSuccess) ms = cuda_fail(nullptr, e, what);
  }
  double hg[2] = {0.0, 0.0};
  if (ms == MEQ_OK) {
    e = cudaMemcpyAsync(hg, g, sizeof(hg), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) ms = cuda_fail(nullptr, e, "cudaMemcpyAsync");
  }
  if (ms == MEQ_OK) gamma_r[0] = hg[0], gamma_c[0] = hg[1];
  // k >= 1: the statistics of the k-step NS output of a one-matrix state fed
  // H with no momentum history and mu = 0 (so its NS input is H), lr = 0
  for (int k = 1; ms == MEQ_OK && k <= steps; ++k) {
    o.ns_steps = k;
    meq_state* st = nullptr;
    ms = meq_init_state(&shape, 1, &o, cuda_stream, &st);
    if (ms != MEQ_OK) break;
    float* wp = w;
    const float* hp = h;
    ms = meq_step(&wp, &hp, st, &shape, 1, 0.f, 0.f, 0.f, eps, cuda_stream);
    if (ms == MEQ_OK) ms = meq_sync(st);
    if (ms == MEQ_OK) ms = meq_read_stats(st, 0, nullptr, nullptr, gamma_r + k, gamma_c + k, nullptr);
    if (ms != MEQ_OK) g_init_error = st->last_error;
    meq_free(st);
  }
  cudaFree(tmp);
  return ms;
}

meq_status meq_check_canaries(meq_state* st, int64_t* bad_offset) {
  if (bad_offset) *bad_offset = -1;
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (st->guard_ranges.empty()) return fail(st, MEQ_ERR_INVALID_ARG, "the state was created without debug_canaries");
  cudaError_t e = cudaStreamSynchronize(st->last_stream);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamSynchronize");
  std::vector<unsigned char> h(static_cast<size_t>(kGuardBytes));
  for (const auto& g : st->guard_ranges) {
    e = cudaMemcpy(h.data(), st->arena + g.first, static_cast<size_t>(g.second), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(st, e, "cudaMemcpy");
    for (int64_t k = 0; k < g.second; ++k)
      if (h[static_cast<size_t>(k)] != kGuardByte) {
        if (bad_offset) *bad_offset = g.first + k;
        return fail(st, MEQ_ERR_CORRUPTED, "workspace guard band overwritten at arena offset " + std::to_string(g.first + k));
      }
  }
  return MEQ_OK;
}

meq_status meq_debug_corrupt_canary(meq_state* st, int index) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (index < 0 || index >= static_cast<int>(st->guard_ranges.size()))
    return fail(st, MEQ_ERR_INVALID_ARG, "no guard band with that index");
  const auto& g = st->guard_ranges[static_cast<size_t>(index)];
  cudaError_t e = cudaMemset(st->arena + g.first + g.second / 2, 0, 1);  // host-side write of one byte
  return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "cudaMemset");
}

int meq_canary_count(const meq_state* st) { return st ? static_cast<int>(st->guard_ranges.size()) : 0; }

meq_status meq_read_direction_counts(meq_state* st, int i, int64_t* rows, int64_t* cols) {
  meq_status ms = check_index(st, i);
  if (ms != MEQ_OK) return ms;
  unsigned long long h[2];
  cudaError_t e = cudaMemcpy(h, st->d_dircount + 2 * i, sizeof(h), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaMemcpy");
  if (rows) *rows = static_cast<int64_t>(h[0]);
  if (cols) *cols = static_cast<int64_t>(h[1]);
  return MEQ_OK;
}

meq_status meq_reset_direction_counts(meq_state* st) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  cudaError_t e = cudaMemsetAsync(st->d_dircount, 0, sizeof(unsigned long long) * 2 * st->n, st->last_stream);
  return e == cudaSuccess ? MEQ_OK : cuda_fail(st, e, "cudaMemsetAsync");
}

meq_status meq_set_profiling(meq_state* st, int enable) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  cudaError_t e = cudaStreamSynchronize(st->last_stream);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamSynchronize");
  drop_profile(st);
  st->profiling = enable != 0;
  return MEQ_OK;
}

meq_status meq_read_profile(meq_state* st, double* phase_ms, int64_t* steps) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  cudaError_t e = cudaStreamSynchronize(st->last_stream);
  if (e != cudaSuccess) return cuda_fail(st, e, "cudaStreamSynchronize");
  double acc[5] = {0, 0, 0, 0, 0};
  for (int p = 0; p < 5; ++p) acc[p] = st->prof_sum[p];
  for (auto& v : st->prof_events)
    for (int p = 0; p < 5; ++p) {
      float ms = 0.f;
      e = cudaEventElapsedTime(&ms, v[p], v[p + 1]);
      if (e != cudaSuccess) return cuda_fail(st, e, "cudaEventElapsedTime");
      acc[p] += ms;
    }
  if (phase_ms)
    for (int p = 0; p < 5; ++p) phase_ms[p] = acc[p];
  if (steps) *steps = static_cast<int64_t>(st->prof_events.size()) + st->prof_graph_steps;
  return MEQ_OK;
}

int meq_kernels_per_step(const meq_state* st) { return st ? st->kernels_per_step : 0; }

int meq_ns_gemm_launches_per_step(const meq_state* st) {
  return st ? static_cast<int>(st->gemm.size()) : 0;
}

meq_status meq_debug_wait_selftest(meq_state* st, float timeout_ms) {
  if (!st) return fail(nullptr, MEQ_ERR_INVALID_ARG, "state is NULL");
  if (!(timeout_ms > 0.f) || timeout_ms > 10000.f) return fail(st, MEQ_ERR_INVALID_ARG, "timeout_ms must be in (0, 10000]");
  cudaError_t e = cudaMemsetAsync(st->d_flag, 0, sizeof(int), st->last_stream);
  if (e == cudaSuccess)
    e = launch_wait_selftest(st->d_flag, st->d_err, static_cast<unsigned long long>(static_cast<double>(timeout_ms) * 1e6),
                             st->last_stream);
  if (e != cudaSuccess) return cuda_fail(st, e, "wait self-test launch");
  return meq_sync(st);
}

}  // extern "C"
