// C ABI of libasap_moe: argument validation, workspace layout, weight packing
// at handle creation and the launch sequence of every call.  Every call other
// than create / destroy / status only enqueues kernels on the caller's stream.
#include "../../include/asap_moe.h"
#include "common.cuh"
#include "internal.h"
#include "gemm_config.h"

#include <atomic>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#define ASAP_API extern "C" __attribute__((visibility("default")))

// Device copies of one layer's weights.
struct LayerWeights {
  void* router_w = nullptr;      // [E, H] bf16
  float* router_bias = nullptr;  // [E] fp32 or nullptr
  void* gate_up = nullptr;       // [E][2I, H], gate/up interleaved per 128 rows
  void* down = nullptr;          // [E][H, I]
  void* sh_gate_up = nullptr;    // [2Is, H]
  void* sh_down = nullptr;       // [H, Is]
  // FP8 only: block scales, gate/up rows interleaved like the weights
  float* gu_scales = nullptr;     // [E][2I/128][H/128]
  float* d_scales = nullptr;      // [E][H/128][I/128]
  float* sh_gu_scales = nullptr;  // [2Is/128][H/128]
  float* sh_d_scales = nullptr;   // [H/128][Is/128]
};

struct asap_moe_s {
  asap_moe_config cfg;
  int device = 0;
  int num_sms = 0;
  std::vector<LayerWeights> layers;
  asap::LayerEntry* table = nullptr;  // device [n_layers]: descriptors and pointers per layer
  int32_t* layer_ids = nullptr;       // device [n_layers] = 0, 1, ...: fixed layer ids
  uint32_t* status = nullptr;         // device status word
  bool tc_router = false;             // router GEMM on the tensor core (E == 256)
  bool fp8 = false;                   // e4m3 experts with fp32 128 x 128 block scales
  int tiling = ASAP_TILING_AUTO;       // BF16 grouped GEMM tile shape (asap_moe_set_tiling)
  int combine = ASAP_COMBINE_SEPARATE;  // where asap_moe_layer combines (asap_moe_set_combine)
  std::atomic<int> mailboxes{0};      // live mailboxes created on this handle
};

namespace {

thread_local std::string g_last_error;

int fail(int code, const std::string& msg) {
  g_last_error = msg;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(ASAP_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

#define CU_TRY(expr, what)                  \
  do {                                      \
    cudaError_t _e = (expr);                \
    if (_e != cudaSuccess) return cuda_fail(_e, what); \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int kMaxBatch = 64;  // micro-batches one asap_moe_layer_batched call may serve

constexpr int kHintA = ASAP_HINT_BF16_A, kHintB = ASAP_HINT_BF16_B, kHintDnA = ASAP_HINT_BF16_DN_A;
constexpr int kHintF8A = ASAP_HINT_FP8_A, kHintF8B = ASAP_HINT_FP8_B;

struct Layout {
  size_t logits, idx, w, hist, chunk_base, counts, offsets, perm_src, perm_dst, tile_counters, ticket;
  // bf16: x_perm (also y_perm in asap_moe_layer), h, h_sh, y_sh
  size_t x_perm, h, h_sh, y_sh, comb_cnt;
  // fp8: quantised rows and their per-128-channel scales, bf16 expert outputs
  size_t xq, xs, xq_sh, xs_sh, hq, hs, hq_sh, hs_sh, y_perm;
  size_t total;
};

Layout layout(const asap_moe_config& c, long long n) {
  Layout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = (off + bytes + 255) & ~static_cast<size_t>(255);
    return o;
  };
  const size_t nk = static_cast<size_t>(n) * c.top_k;
  const size_t N = static_cast<size_t>(n);
  // one extra chunk per micro-batch a batched call may serve
  const size_t chunks = (N + asap::kChunkTokens - 1) / asap::kChunkTokens + kMaxBatch;
  const size_t H = c.hidden, I = c.inter, Is = c.n_shared ? c.shared_inter : 0, E = c.n_experts;
  L.logits = take(asap::kMaxRouterSplits * N * E * 4);  // K-slice planes
  L.idx = take(nk * 4);
  L.w = take(nk * 4);
  L.hist = take(chunks * E * 4);
  L.chunk_base = take(chunks * E * 4);
  L.counts = take(E * 4);
  L.offsets = take((E + 1) * 4);
  L.perm_src = take(nk * 4);
  L.perm_dst = take(nk * 4);
  L.tile_counters = take(asap::kTileCounters * 4);
  L.ticket = take(4);
  if (c.dtype == ASAP_FP8_E4M3_BLOCK128) {
    L.xq = take(nk * H);
    L.xs = take(nk * (H / 128) * 4);
    L.xq_sh = take(N * H * (Is ? 1 : 0));
    L.xs_sh = take(N * (H / 128) * 4 * (Is ? 1 : 0));
    L.hq = take(nk * I);
    L.hs = take(nk * (I / 128) * 4);
    L.hq_sh = take(N * Is);
    L.hs_sh = take(N * (Is / 128) * 4);
    L.y_perm = take(nk * H * 2);
    L.y_sh = take(N * H * 2 * (Is ? 1 : 0));
  } else {
    L.x_perm = take(nk * H * 2);  // also holds y_perm in asap_moe_layer
    L.h = take(nk * I * 2);
    L.h_sh = take(N * Is * 2);
    L.y_sh = take(N * H * 2 * (Is ? 1 : 0));
    L.comb_cnt = take(N * (H / asap::kGemmBN) * 4);  // slice arrivals of the fused combine
  }
  L.total = off;
  return L;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

cudaStream_t S(void* s) { return static_cast<cudaStream_t>(s); }

// The layer-table entry a launch reads: *layer, resolved on the device.
asap::LayerRef lref(asap_moe_t h, const int32_t* layer) {
  return asap::LayerRef{h->table, layer, static_cast<int>(h->layers.size())};
}

int check_call(asap_moe_t h, int32_t n, void* ws, size_t ws_bytes, bool needs_ws) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  if (n < 0 || n > h->cfg.max_tokens)
    return fail(ASAP_ERR_INVALID, "n = " + std::to_string(n) + " outside [0, max_tokens = " +
                                      std::to_string(h->cfg.max_tokens) + "]");
  if (needs_ws && n > 0) {
    if (!ws) return fail(ASAP_ERR_WORKSPACE, "NULL workspace");
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
      return fail(ASAP_ERR_INVALID, "workspace must be 256-byte aligned");
    const size_t need = layout(h->cfg, n).total;
    if (ws_bytes < need)
      return fail(ASAP_ERR_WORKSPACE, "workspace has " + std::to_string(ws_bytes) + " bytes, needs " +
                                          std::to_string(need));
  }
  return ASAP_OK;
}

// ------------------------------------------------------------ launch helpers

// Number of K slices of the tensor-core router GEMM for n tokens: enough
// CTAs to cover the SMs (one 128-row tile x one 256-expert tile per slice),
// at least 8 k-blocks per slice, and 1, 2 or 4 (the fused route kernel's
// cluster gives each CTA 4 / slices of a tile's 32-token quarters).
int router_splits(asap_moe_t h, int n) {
  if (!h->tc_router) return 1;
  const int mtiles = asap::ceil_div(n, asap::kGemmBM);
  const int kit = h->cfg.hidden / asap::kGemmBK;
  int s = h->num_sms / std::max(mtiles, 1);
  s = std::min(s, kit / 8);
  s = std::min(s, asap::kMaxRouterSplits);
  int p = 1;
  while (p * 2 <= s) p *= 2;
  return p;
}

// Routing in one launch (router GEMM + gating + scan): E = 256 with grouped
// sigmoid gating in 1, 2, 4 or 8 groups.  Other configurations run the
// router, gate and scan kernels one after the other.
bool fused_route(asap_moe_t h) {
  const asap_moe_config& c = h->cfg;
  return h->tc_router && c.gating == ASAP_GATE_SIGMOID_GROUPED &&
         (c.n_groups == 1 || c.n_groups == 2 || c.n_groups == 4 || c.n_groups == 8);
}

// The fused route launch for n tokens of x.  With ticket (zero at launch)
// its last CTA scans the histogram into chunk_base, counts and offsets and
// zeroes tile_counters (nullable); without, hist columns [chunk0, chunk0 +
// ceil(n/32)) of n_chunks_total are left for one scan over several
// micro-batches.
// narrow: no cluster; each CTA computes its tile's K slices one after the
// other (same logits bits), so concurrent routes share the GPU in one wave.
int run_route_fused(asap_moe_t h, const void* x, int n, int32_t* idx, float* w, int32_t* hist, int chunk0,
                    int n_chunks_total, int32_t* ticket, int32_t* counts, int32_t* offsets, int32_t* chunk_base,
                    int32_t* tile_counters, const int32_t* layer, cudaStream_t st, bool narrow = false);

// Router logits as ``splits`` planes of partial sums [splits][n][E] (planes
// are added in order by the consumer); splits == 1 writes the logits.
int run_router_logits(asap_moe_t h, const void* x, int n, float* logits, int splits, const int32_t* layer,
                      cudaStream_t st) {
  const asap_moe_config& c = h->cfg;
  if (h->tc_router) {
    CUtensorMap maps[4];
    std::string err;
    if (!asap::encode_tmap_bf16(&maps[0], x, n, c.hidden, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "x: " + err);
    maps[1] = maps[2] = maps[3] = maps[0];  // the fp32 logits are stored without TMA
    asap::GemmArgs a{};
    a.lref = lref(h, layer);
    a.bmap0 = a.bmap1 = asap::MAP_ROUTER;
    a.offsets = nullptr;
    a.groups = 1;
    a.m0 = n;
    a.b_stride0 = 0;
    a.n_tiles0 = 1;
    a.k_iters0 = c.hidden / asap::kGemmBK;
    a.out0 = logits;
    a.ldo0 = c.n_experts;
    a.m1 = 0;
    a.status = h->status;
    a.hint_a = 0;
    a.hint_b = 2;
    a.k_splits = splits;
    a.split_rows0 = n;
    const int tiles = asap::ceil_div(n, asap::kGemmBM) * splits;
    CU_TRY(asap::gemm_launch(asap::EPI_F32, false, maps, a, std::min(tiles, h->num_sms), st), "router GEMM launch");
  } else {
    CU_TRY(asap::launch_router_small(x, lref(h, layer), n, c.hidden, c.n_experts, logits, h->status, st),
           "router launch");
  }
  return ASAP_OK;
}

int run_route_fused(asap_moe_t h, const void* x, int n, int32_t* idx, float* w, int32_t* hist, int chunk0,
                    int n_chunks_total, int32_t* ticket, int32_t* counts, int32_t* offsets, int32_t* chunk_base,
                    int32_t* tile_counters, const int32_t* layer, cudaStream_t st, bool narrow) {
  const asap_moe_config& c = h->cfg;
  CUtensorMap tmx;
  std::string err;
  if (!asap::encode_tmap_bf16(&tmx, x, n, c.hidden, asap::kGemmBM, &err)) return fail(ASAP_ERR_INVALID, "x: " + err);
  asap::RouteFusedArgs a{};
  a.lref = lref(h, layer);
  a.status = h->status;
  a.n = n;
  a.k_iters = c.hidden / asap::kGemmBK;
  const int splits = router_splits(h, n);
  a.splits = narrow ? 1 : splits;
  a.seq_slices = narrow ? splits : 1;
  a.top_k = c.top_k;
  a.n_groups = c.n_groups;
  a.topk_groups = c.topk_groups;
  a.route_scale = c.route_scale;
  a.idx = idx;
  a.w = w;
  a.hist = hist;
  a.chunk0 = chunk0;
  a.n_chunks_total = n_chunks_total;
  a.ticket = ticket;
  a.counts = counts;
  a.offsets = offsets;
  a.chunk_base = chunk_base;
  a.tile_counters = tile_counters;
  CU_TRY(asap::launch_route_fused(tmx, a, st), "fused route launch");
  return ASAP_OK;
}

// Routing of one micro-batch into idx, w, counts, offsets and the
// workspace's chunk bases; also zeroes the workspace's tile counters for the
// grouped GEMMs that follow on the stream.
int run_route(asap_moe_t h, const void* x, int n, int32_t* idx, float* w, int32_t* counts, int32_t* offsets,
              void* ws, const int32_t* layer, cudaStream_t st);

// ticket: the scan's ticket in the call's scratch (zeroed by the gate launch).
asap::GateParams gate_params(asap_moe_t h, const int32_t* layer, int32_t* ticket) {
  const asap_moe_config& c = h->cfg;
  asap::GateParams p{};
  p.n_experts = c.n_experts;
  p.top_k = c.top_k;
  p.gating = c.gating;
  p.n_groups = c.gating == ASAP_GATE_SIGMOID_GROUPED ? c.n_groups : 1;
  p.topk_groups = c.gating == ASAP_GATE_SIGMOID_GROUPED ? c.topk_groups : 1;
  p.route_scale = c.route_scale;
  p.lref = lref(h, layer);
  p.status = h->status;
  p.ticket = ticket;
  return p;
}

int run_gate_scan(asap_moe_t h, const float* logits, int splits, int n, int32_t* idx, float* w, int32_t* counts,
                  int32_t* offsets, void* ws, const int32_t* layer, cudaStream_t st) {
  const Layout L = layout(h->cfg, n);
  int32_t* hist = at<int32_t>(ws, L.hist);
  int32_t* base = at<int32_t>(ws, L.chunk_base);
  int32_t* ticket = at<int32_t>(ws, L.ticket);
  CU_TRY(asap::launch_gate(logits, splits, n, gate_params(h, layer, ticket), idx, w, hist, st), "gate launch");
  CU_TRY(asap::launch_scan(hist, asap::ceil_div(n, asap::kChunkTokens), h->cfg.n_experts, counts, offsets, base,
                           ticket, st, at<int32_t>(ws, L.tile_counters)),
         "scan launch");
  return ASAP_OK;
}

int run_route(asap_moe_t h, const void* x, int n, int32_t* idx, float* w, int32_t* counts, int32_t* offsets,
              void* ws, const int32_t* layer, cudaStream_t st) {
  const Layout L = layout(h->cfg, n);
  if (fused_route(h)) {
    // the tile counters and the ticket, one memset (the ticket follows them)
    static_assert(asap::kTileCounters * 4 <= 256, "tile counters fit before the ticket");
    CU_TRY(cudaMemsetAsync(at<char>(ws, L.tile_counters), 0, L.ticket - L.tile_counters + 4, st), "ticket");
    return run_route_fused(h, x, n, idx, w, at<int32_t>(ws, L.hist), 0, asap::ceil_div(n, asap::kChunkTokens),
                           at<int32_t>(ws, L.ticket), counts, offsets, at<int32_t>(ws, L.chunk_base),
                           at<int32_t>(ws, L.tile_counters), layer, st);
  }
  float* logits = at<float>(ws, L.logits);
  const int splits = router_splits(h, n);
  int r = run_router_logits(h, x, n, logits, splits, layer, st);
  if (r != ASAP_OK) return r;
  return run_gate_scan(h, logits, splits, n, idx, w, counts, offsets, ws, layer, st);
}

// Paired m-tiles (two 128-row m-tiles per GEMM tile sharing the weight
// boxes, a half tile for a segment's last <= 128 rows) when
//  - the segments hold at least one m-tile (128 rows) per expert on average:
//    below that nearly every paired tile is a half tile, and the paired rings
//    (3 + 3 stages) keep fewer weight bytes in flight than the single-tile
//    rings (4 + 4).  Measured on a GB300 at the DeepSeek-V3 shape (gate/up |
//    down ms, paired vs single): 3072 tokens (96 rows per expert) 2.26 |
//    1.23 vs 2.19 | 1.16; 4096 tokens (128) 2.35 | 1.31 vs 2.39 | 1.33;
//  - and the launch has at least ASAP_PAIR_MIN_WAVES waves of paired tiles
//    (estimate: nk / 256 full tiles plus half a tile of rounding per
//    non-empty segment).  With few tiles the larger tile rounds the launch to
//    whole waves more coarsely than it saves.
bool use_pair(asap_moe_t h, long long nk, int n_tiles0, long long m1, int n_tiles1) {
  if (h->tiling != ASAP_TILING_AUTO) return h->tiling == ASAP_TILING_PAIRED;
  const asap_moe_config& c = h->cfg;
  if (nk < static_cast<long long>(asap::kGemmBM) * c.n_experts) return false;
  const long long seg = std::min<long long>(c.n_experts, nk);
  const long long est = (asap::ceil_div(nk, 2 * asap::kGemmBM) + seg / 2) * n_tiles0 +
                        asap::ceil_div(m1, 2 * asap::kGemmBM) * n_tiles1;
  return est >= static_cast<long long>(ASAP_PAIR_MIN_WAVES) * h->num_sms;
}

// Upper bound of the m-tiles of bm rows over the routed segments.
int ub_mtiles(const asap_moe_config& c, long long nk, int bm = asap::kGemmBM) {
  return asap::ceil_div(nk, bm) + static_cast<int>(std::min<long long>(c.n_experts, nk));
}

// Rows of the output boxes the bf16 GEMM epilogues store with TMA (one epilogue
// warp's 32 rows).
constexpr uint32_t kStoreRows = 32;

// GEMM1: h = silu(X Wg^T) * (X Wu^T) on the routed segments, plus the shared
// expert on x (problem 1 of the same launch).
// counter: a zeroed int the launch claims its tiles from (nullptr: static order).
// m1_dev (nullable): the shared expert's row count read when the launch runs
// (at most n); the tile count and the maps are sized for n.
int run_gate_up(asap_moe_t h, const void* x_perm, const int32_t* offsets, const void* x, int n, void* hbuf,
                void* hsh, const int32_t* layer, int32_t* counter, cudaStream_t st,
                const int32_t* m1_dev = nullptr) {
  const asap_moe_config& c = h->cfg;
  const long long nk = static_cast<long long>(n) * c.top_k;
  const bool sh = c.n_shared != 0;
  const bool pair = use_pair(h, nk, c.inter / 128, sh ? n : 0, c.shared_inter / 128);
  const int bm = pair ? 2 * asap::kGemmBM : asap::kGemmBM;
  std::string err;
  CUtensorMap maps[4];
  if (!asap::encode_tmap_bf16(&maps[0], x_perm, nk, c.hidden, asap::kGemmBM, &err))
    return fail(ASAP_ERR_INVALID, "x_perm: " + err);
  if (!asap::encode_tmap_bf16(&maps[2], hbuf, nk, c.inter, kStoreRows, &err))
    return fail(ASAP_ERR_INVALID, "h: " + err);
  if (sh) {
    if (!asap::encode_tmap_bf16(&maps[1], x, n, c.hidden, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "x: " + err);
    if (!asap::encode_tmap_bf16(&maps[3], hsh, n, c.shared_inter, kStoreRows, &err))
      return fail(ASAP_ERR_INVALID, "h_shared: " + err);
  } else {
    maps[1] = maps[0];
    maps[3] = maps[2];
  }
  asap::GemmArgs a{};
  a.lref = lref(h, layer);
  a.bmap0 = asap::MAP_GATE_UP;
  a.bmap1 = sh ? asap::MAP_SH_GATE_UP : asap::MAP_GATE_UP;
  a.offsets = offsets;
  a.groups = c.n_experts;
  a.m0 = static_cast<int>(nk);
  a.b_stride0 = 2 * c.inter;
  a.n_tiles0 = c.inter / 128;
  a.k_iters0 = c.hidden / asap::kGemmBK;
  a.out0 = hbuf;
  a.ldo0 = c.inter;
  a.m1 = sh ? n : 0;
  a.m1_dev = sh ? m1_dev : nullptr;
  a.n_tiles1 = sh ? c.shared_inter / 128 : 0;
  a.k_iters1 = c.hidden / asap::kGemmBK;
  a.out1 = hsh;
  a.ldo1 = c.shared_inter;
  a.status = h->status;
  a.hint_a = kHintA;
  a.hint_b = kHintB;
  a.k_splits = 1;
  a.tile_counter = counter;
  a.b_tiled = 1;  // weights in tile-contiguous order (pack_layer)
  const long long tiles = static_cast<long long>(ub_mtiles(c, nk, bm)) * a.n_tiles0 +
                          (sh ? static_cast<long long>(asap::ceil_div(n, bm)) * a.n_tiles1 : 0);
  CU_TRY(asap::gemm_launch(asap::EPI_SWIGLU, pair, maps, a, static_cast<int>(std::min<long long>(tiles, h->num_sms)),
                           st),
         "gate/up GEMM launch");
  return ASAP_OK;
}

// GEMM2: y = h Wd^T on the routed segments, plus the shared expert.
// The combine fused into the down GEMM (see combine_slices): slice arrival
// counters (zeroed before the launch), the permutation and the routing
// weights of the call, and its output.
struct CombineFuse {
  int* cnt = nullptr;
  const int32_t* src = nullptr;
  const int32_t* dst = nullptr;
  const float* w = nullptr;
  void* out = nullptr;
};

int run_down(asap_moe_t h, const void* hbuf, const int32_t* offsets, const void* hsh, int n, void* y_perm,
             void* y_sh, const int32_t* layer, int32_t* counter, cudaStream_t st, const int32_t* m1_dev = nullptr,
             const CombineFuse& cf = CombineFuse()) {
  const asap_moe_config& c = h->cfg;
  const long long nk = static_cast<long long>(n) * c.top_k;
  const bool sh = c.n_shared != 0;
  const bool pair = use_pair(h, nk, c.hidden / asap::kGemmBN, sh ? n : 0, c.hidden / asap::kGemmBN);
  const int bm = pair ? 2 * asap::kGemmBM : asap::kGemmBM;
  std::string err;
  CUtensorMap maps[4];
  if (!asap::encode_tmap_bf16(&maps[0], hbuf, nk, c.inter, asap::kGemmBM, &err))
    return fail(ASAP_ERR_INVALID, "h: " + err);
  if (!asap::encode_tmap_bf16(&maps[2], y_perm, nk, c.hidden, kStoreRows, &err))
    return fail(ASAP_ERR_INVALID, "y_perm: " + err);
  if (sh) {
    if (!asap::encode_tmap_bf16(&maps[1], hsh, n, c.shared_inter, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "h_shared: " + err);
    if (!asap::encode_tmap_bf16(&maps[3], y_sh, n, c.hidden, kStoreRows, &err))
      return fail(ASAP_ERR_INVALID, "y_shared: " + err);
  } else {
    maps[1] = maps[0];
    maps[3] = maps[2];
  }
  asap::GemmArgs a{};
  a.lref = lref(h, layer);
  a.bmap0 = asap::MAP_DOWN;
  a.bmap1 = sh ? asap::MAP_SH_DOWN : asap::MAP_DOWN;
  a.offsets = offsets;
  a.groups = c.n_experts;
  a.m0 = static_cast<int>(nk);
  a.b_stride0 = c.hidden;
  a.n_tiles0 = c.hidden / asap::kGemmBN;
  a.k_iters0 = c.inter / asap::kGemmBK;
  a.out0 = y_perm;
  a.ldo0 = c.hidden;
  a.m1 = sh ? n : 0;
  a.m1_dev = sh ? m1_dev : nullptr;
  a.n_tiles1 = sh ? c.hidden / asap::kGemmBN : 0;
  a.k_iters1 = sh ? c.shared_inter / asap::kGemmBK : 0;
  a.out1 = y_sh;
  a.ldo1 = c.hidden;
  a.status = h->status;
  a.hint_a = kHintDnA;
  a.hint_b = kHintB;
  a.k_splits = 1;
  a.tile_counter = counter;
  a.b_tiled = 1;  // weights in tile-contiguous order (pack_layer)
  a.comb_cnt = cf.cnt;
  a.comb_src = cf.src;
  a.comb_dst = cf.dst;
  a.comb_w = cf.w;
  a.comb_out = cf.out;
  a.comb_n = n;
  a.comb_k = c.top_k;
  const long long tiles = static_cast<long long>(ub_mtiles(c, nk, bm)) * a.n_tiles0 +
                          (sh ? static_cast<long long>(asap::ceil_div(n, bm)) * a.n_tiles1 : 0);
  CU_TRY(asap::gemm_launch(asap::EPI_BF16, pair, maps, a, static_cast<int>(std::min<long long>(tiles, h->num_sms)), st),
         "down GEMM launch");
  return ASAP_OK;
}

// counters: kTileCounters zeroed ints (or nullptr)
int run_expert_ffn(asap_moe_t h, const void* x_perm, const int32_t* offsets, const void* x, int n,
                   void* y_perm, void* y_sh, void* hbuf, void* hsh, const int32_t* layer, int32_t* counters,
                   cudaStream_t st) {
  int r = run_gate_up(h, x_perm, offsets, x, n, hbuf, hsh, layer, counters, st);
  if (r != ASAP_OK) return r;
  return run_down(h, hbuf, offsets, hsh, n, y_perm, y_sh, layer, counters ? counters + 1 : nullptr, st);
}

// FP8 GEMM1: hq = e4m3(silu(Xq Wg^T) * (Xq Wu^T)) with its row scales, routed
// segments plus the shared expert on the quantised x.
int run_gate_up_fp8(asap_moe_t h, const void* xq, const float* xs, const int32_t* offsets, const void* xq_sh,
                    const float* xs_sh, int n, void* hq, float* hs, void* hq_sh, float* hs_sh, const int32_t* layer,
                    int32_t* counter, cudaStream_t st, const int32_t* m1_dev = nullptr) {
  const asap_moe_config& c = h->cfg;
  const long long nk = static_cast<long long>(n) * c.top_k;
  const bool sh = c.n_shared != 0;
  std::string err;
  CUtensorMap maps[2];
  if (!asap::encode_tmap_u8(&maps[0], xq, nk, c.hidden, asap::kGemmBM, &err)) return fail(ASAP_ERR_INVALID, "x_perm: " + err);
  if (sh) {
    if (!asap::encode_tmap_u8(&maps[1], xq_sh, n, c.hidden, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "quantised x: " + err);
  } else {
    maps[1] = maps[0];
  }
  asap::Fp8Args f{};
  asap::GemmArgs& a = f.g;
  a.lref = lref(h, layer);
  a.bmap0 = asap::MAP_GATE_UP;
  a.bmap1 = sh ? asap::MAP_SH_GATE_UP : asap::MAP_GATE_UP;
  a.offsets = offsets;
  a.groups = c.n_experts;
  a.m0 = static_cast<int>(nk);
  a.b_stride0 = 2 * c.inter;
  a.n_tiles0 = c.inter / 128;
  a.k_iters0 = c.hidden / asap::kFp8BK;
  a.out0 = hq;
  a.ldo0 = c.inter;
  a.m1 = sh ? n : 0;
  a.m1_dev = sh ? m1_dev : nullptr;
  a.n_tiles1 = sh ? c.shared_inter / 128 : 0;
  a.k_iters1 = c.hidden / asap::kFp8BK;
  a.out1 = hq_sh;
  a.ldo1 = c.shared_inter;
  a.status = h->status;
  a.hint_a = kHintF8A;
  a.hint_b = kHintF8B;
  a.k_splits = 1;
  a.tile_counter = counter;
  a.b_tiled = 1;  // weights in tile-contiguous order (pack_layer)
  f.a_scale0 = xs;
  f.a_sld0 = c.hidden / 128;
  f.a_scale1 = xs_sh;
  f.a_sld1 = c.hidden / 128;
  f.b_nblk0 = 2 * c.inter / 128;
  f.b_nblk1 = sh ? 2 * c.shared_inter / 128 : 0;
  f.out_scale0 = hs;
  f.o_sld0 = c.inter / 128;
  f.out_scale1 = hs_sh;
  f.o_sld1 = sh ? c.shared_inter / 128 : 0;
  const long long tiles = static_cast<long long>(ub_mtiles(c, nk)) * a.n_tiles0 +
                          (sh ? static_cast<long long>(asap::ceil_div(n, asap::kGemmBM)) * a.n_tiles1 : 0);
  CU_TRY(asap::fp8_gemm_launch(asap::EPI_SWIGLU, maps, f, static_cast<int>(std::min<long long>(tiles, h->num_sms)), st),
         "fp8 gate/up GEMM launch");
  return ASAP_OK;
}

// FP8 GEMM2: y = (hq * hs) (Wd * sd)^T, bf16 out.
int run_down_fp8(asap_moe_t h, const void* hq, const float* hs, const int32_t* offsets, const void* hq_sh,
                 const float* hs_sh, int n, void* y_perm, void* y_sh, const int32_t* layer, int32_t* counter,
                 cudaStream_t st, const int32_t* m1_dev = nullptr) {
  const asap_moe_config& c = h->cfg;
  const long long nk = static_cast<long long>(n) * c.top_k;
  const bool sh = c.n_shared != 0;
  std::string err;
  CUtensorMap maps[2];
  if (!asap::encode_tmap_u8(&maps[0], hq, nk, c.inter, asap::kGemmBM, &err)) return fail(ASAP_ERR_INVALID, "h: " + err);
  if (sh) {
    if (!asap::encode_tmap_u8(&maps[1], hq_sh, n, c.shared_inter, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "h_shared: " + err);
  } else {
    maps[1] = maps[0];
  }
  asap::Fp8Args f{};
  asap::GemmArgs& a = f.g;
  a.lref = lref(h, layer);
  a.bmap0 = asap::MAP_DOWN;
  a.bmap1 = sh ? asap::MAP_SH_DOWN : asap::MAP_DOWN;
  a.offsets = offsets;
  a.groups = c.n_experts;
  a.m0 = static_cast<int>(nk);
  a.b_stride0 = c.hidden;
  a.n_tiles0 = c.hidden / asap::kGemmBN;
  a.k_iters0 = c.inter / asap::kFp8BK;
  a.out0 = y_perm;
  a.ldo0 = c.hidden;
  a.m1 = sh ? n : 0;
  a.m1_dev = sh ? m1_dev : nullptr;
  a.n_tiles1 = sh ? c.hidden / asap::kGemmBN : 0;
  a.k_iters1 = sh ? c.shared_inter / asap::kFp8BK : 0;
  a.out1 = y_sh;
  a.ldo1 = c.hidden;
  a.status = h->status;
  a.hint_a = kHintF8A;
  a.hint_b = kHintF8B;
  a.k_splits = 1;
  a.tile_counter = counter;
  a.b_tiled = 1;  // weights in tile-contiguous order (pack_layer)
  f.a_scale0 = hs;
  f.a_sld0 = c.inter / 128;
  f.a_scale1 = hs_sh;
  f.a_sld1 = sh ? c.shared_inter / 128 : 0;
  f.b_nblk0 = c.hidden / 128;
  f.b_nblk1 = c.hidden / 128;
  const long long tiles = static_cast<long long>(ub_mtiles(c, nk)) * a.n_tiles0 +
                          (sh ? static_cast<long long>(asap::ceil_div(n, asap::kGemmBM)) * a.n_tiles1 : 0);
  CU_TRY(asap::fp8_gemm_launch(asap::EPI_BF16, maps, f, static_cast<int>(std::min<long long>(tiles, h->num_sms)), st),
         "fp8 down GEMM launch");
  return ASAP_OK;
}

}  // namespace

// ============================================================ public API

ASAP_API const char* asap_moe_last_error(void) { return g_last_error.c_str(); }

ASAP_API int asap_moe_check_config(const asap_moe_config* c) {
  if (!c) return fail(ASAP_ERR_INVALID, "NULL config");
  if (c->hidden <= 0 || c->hidden % 256 != 0) return fail(ASAP_ERR_INVALID, "hidden must be a positive multiple of 256");
  if (c->n_experts < 1 || c->n_experts > ASAP_MOE_MAX_EXPERTS)
    return fail(ASAP_ERR_INVALID, "n_experts must be in [1, 256]");
  if (c->top_k < 1 || c->top_k > ASAP_MOE_MAX_TOPK || c->top_k > c->n_experts)
    return fail(ASAP_ERR_INVALID, "top_k must be in [1, min(8, n_experts)]");
  if (c->inter <= 0 || c->inter % 128 != 0) return fail(ASAP_ERR_INVALID, "inter must be a positive multiple of 128");
  if (c->n_shared != 0 && c->n_shared != 1) return fail(ASAP_ERR_INVALID, "n_shared must be 0 or 1");
  if (c->n_shared == 1 && (c->shared_inter <= 0 || c->shared_inter % 128 != 0))
    return fail(ASAP_ERR_INVALID, "shared_inter must be a positive multiple of 128");
  if (c->gating < 0 || c->gating > 2) return fail(ASAP_ERR_INVALID, "unknown gating");
  if (c->gating == ASAP_GATE_SIGMOID_GROUPED) {
    if (c->n_groups < 1 || c->n_groups > 32 || c->n_experts % c->n_groups != 0)
      return fail(ASAP_ERR_INVALID, "n_groups must divide n_experts and be <= 32");
    const int gsz = c->n_experts / c->n_groups;
    if (gsz < 2) return fail(ASAP_ERR_INVALID, "groups need at least 2 experts");
    if (c->topk_groups < 1 || c->topk_groups > c->n_groups)
      return fail(ASAP_ERR_INVALID, "topk_groups must be in [1, n_groups]");
    if (c->top_k > c->topk_groups * gsz) return fail(ASAP_ERR_INVALID, "top_k exceeds the experts of the kept groups");
    if (!(c->route_scale > 0.0f)) return fail(ASAP_ERR_INVALID, "route_scale must be positive");
  }
  if (c->dtype != ASAP_BF16 && c->dtype != ASAP_FP8_E4M3_BLOCK128) return fail(ASAP_ERR_INVALID, "unknown dtype");
  if (c->max_tokens < 1 || static_cast<long long>(c->max_tokens) * c->top_k >= (1ll << 31))
    return fail(ASAP_ERR_INVALID, "max_tokens * top_k must be in [1, 2^31)");
  return ASAP_OK;
}

ASAP_API int asap_moe_workspace_size(const asap_moe_config* cfg, int32_t n_tokens, size_t* bytes) {
  const int r = asap_moe_check_config(cfg);
  if (r != ASAP_OK) return r;
  if (!bytes) return fail(ASAP_ERR_INVALID, "NULL bytes");
  if (n_tokens < 0 || n_tokens > cfg->max_tokens) return fail(ASAP_ERR_INVALID, "n_tokens outside [0, max_tokens]");
  *bytes = n_tokens == 0 ? 0 : layout(*cfg, n_tokens).total;
  return ASAP_OK;
}

ASAP_API int asap_moe_destroy(asap_moe_t h) {
  if (!h) return ASAP_OK;
  if (const int live = h->mailboxes.load())
    return fail(ASAP_ERR_INVALID, std::to_string(live) +
                                      " mailbox(es) created on this handle are still alive; destroy them first");
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  for (LayerWeights& L : h->layers) {
    cudaFree(L.router_w);
    cudaFree(L.router_bias);
    cudaFree(L.gate_up);
    cudaFree(L.down);
    cudaFree(L.sh_gate_up);
    cudaFree(L.sh_down);
    cudaFree(L.gu_scales);
    cudaFree(L.d_scales);
    cudaFree(L.sh_gu_scales);
    cudaFree(L.sh_d_scales);
  }
  cudaFree(h->table);
  cudaFree(h->layer_ids);
  cudaFree(h->status);
  cudaSetDevice(prev);
  delete h;
  return ASAP_OK;
}

namespace {

constexpr int kMaxLayers = 4096;

int check_weights(const asap_moe_config& c, const asap_moe_weights* wts) {
  if (!wts || !wts->router_w || !wts->w_gate || !wts->w_up || !wts->w_down)
    return fail(ASAP_ERR_INVALID, "router and expert weights are required");
  if (c.n_shared && (!wts->sh_gate || !wts->sh_up || !wts->sh_down))
    return fail(ASAP_ERR_INVALID, "shared-expert weights are required when n_shared == 1");
  if (c.dtype == ASAP_FP8_E4M3_BLOCK128 &&
      (!wts->s_gate || !wts->s_up || !wts->s_down ||
       (c.n_shared && (!wts->sh_s_gate || !wts->sh_s_up || !wts->sh_s_down))))
    return fail(ASAP_ERR_INVALID, "the FP8 configuration needs the fp32 block scales of every expert matrix");
  return ASAP_OK;
}

// Allocate one layer's device copies and enqueue the copies / packing on st.
int pack_layer(asap_moe_t h, const asap_moe_weights* wts, LayerWeights& L, cudaStream_t st) {
  const asap_moe_config& c = h->cfg;
  const size_t H = c.hidden, E = c.n_experts, I = c.inter, Is = c.shared_inter;
  const size_t wb = h->fp8 ? 1 : 2;  // bytes per expert-weight element
  const size_t router_bytes = E * H * 2, gu_bytes = E * 2 * I * H * wb, down_bytes = E * H * I * wb;
  cudaError_t e;
  if ((e = cudaMalloc(&L.router_w, router_bytes)) != cudaSuccess) return cuda_fail(e, "cudaMalloc router");
  if ((e = cudaMemcpyAsync(L.router_w, wts->router_w, router_bytes, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
    return cuda_fail(e, "copy router");
  if (wts->router_bias) {
    if ((e = cudaMalloc(&L.router_bias, E * 4)) != cudaSuccess) return cuda_fail(e, "cudaMalloc bias");
    if ((e = cudaMemcpyAsync(L.router_bias, wts->router_bias, E * 4, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
      return cuda_fail(e, "copy bias");
  }
  // expert weights in the tile-contiguous order of the GEMMs' weight boxes
  // (gate/up interleaved per 128 rows), so each box is one 32 KB read
  if ((e = cudaMalloc(&L.gate_up, gu_bytes)) != cudaSuccess) return cuda_fail(e, "cudaMalloc gate/up");
  if ((e = asap::launch_retile(wts->w_gate, wts->w_up, static_cast<int>(E), static_cast<int>(2 * I),
                               static_cast<long long>(H * wb), true, L.gate_up, st)) != cudaSuccess)
    return cuda_fail(e, "pack gate/up");
  if ((e = cudaMalloc(&L.down, down_bytes)) != cudaSuccess) return cuda_fail(e, "cudaMalloc down");
  if ((e = asap::launch_retile(wts->w_down, nullptr, static_cast<int>(E), static_cast<int>(H),
                               static_cast<long long>(I * wb), false, L.down, st)) != cudaSuccess)
    return cuda_fail(e, "pack down");
  if (c.n_shared) {
    if ((e = cudaMalloc(&L.sh_gate_up, 2 * Is * H * wb)) != cudaSuccess) return cuda_fail(e, "cudaMalloc shared");
    if ((e = asap::launch_retile(wts->sh_gate, wts->sh_up, 1, static_cast<int>(2 * Is), static_cast<long long>(H * wb),
                                 true, L.sh_gate_up, st)) != cudaSuccess)
      return cuda_fail(e, "pack shared");
    if ((e = cudaMalloc(&L.sh_down, H * Is * wb)) != cudaSuccess) return cuda_fail(e, "cudaMalloc shared down");
    if ((e = asap::launch_retile(wts->sh_down, nullptr, 1, static_cast<int>(H), static_cast<long long>(Is * wb), false,
                                 L.sh_down, st)) != cudaSuccess)
      return cuda_fail(e, "pack shared down");
  }
  if (h->fp8) {
    // scale rows interleaved like the weight rows: gate block b -> 2b, up block b -> 2b+1
    const size_t kb = H / 128, rowb = kb * 4;
    auto interleave = [&](float** dst, const float* g, const float* u, size_t blocks) -> cudaError_t {
      cudaError_t r = cudaMalloc(dst, 2 * blocks * rowb);
      if (r == cudaSuccess) r = cudaMemcpy2DAsync(*dst, 2 * rowb, g, rowb, rowb, blocks, cudaMemcpyDeviceToDevice, st);
      if (r == cudaSuccess)
        r = cudaMemcpy2DAsync(reinterpret_cast<char*>(*dst) + rowb, 2 * rowb, u, rowb, rowb, blocks,
                              cudaMemcpyDeviceToDevice, st);
      return r;
    };
    if ((e = interleave(&L.gu_scales, wts->s_gate, wts->s_up, E * (I / 128))) != cudaSuccess)
      return cuda_fail(e, "gate/up scales");
    const size_t dsb = E * (H / 128) * (I / 128) * 4;
    if ((e = cudaMalloc(&L.d_scales, dsb)) != cudaSuccess ||
        (e = cudaMemcpyAsync(L.d_scales, wts->s_down, dsb, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
      return cuda_fail(e, "down scales");
    if (c.n_shared) {
      if ((e = interleave(&L.sh_gu_scales, wts->sh_s_gate, wts->sh_s_up, Is / 128)) != cudaSuccess)
        return cuda_fail(e, "shared gate/up scales");
      const size_t sdb = (H / 128) * (Is / 128) * 4;
      if ((e = cudaMalloc(&L.sh_d_scales, sdb)) != cudaSuccess ||
          (e = cudaMemcpyAsync(L.sh_d_scales, wts->sh_s_down, sdb, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
        return cuda_fail(e, "shared down scales");
    }
  }
  return ASAP_OK;
}

// The table entry of one layer: TMA descriptors of its packed weights (the
// pre-computed addresses of Section 3.4.2) and its plain pointers.
int encode_layer(asap_moe_t h, const LayerWeights& L, asap::LayerEntry* out) {
  const asap_moe_config& c = h->cfg;
  const uint64_t H = c.hidden, E = c.n_experts, I = c.inter, Is = c.shared_inter;
  std::memset(out, 0, sizeof(*out));
  std::string err;
  if (h->tc_router && !asap::encode_tmap_bf16(&out->map[asap::MAP_ROUTER], L.router_w, E, H, asap::kGemmBN, &err))
    return fail(ASAP_ERR_CUDA, "router map: " + err);
  // tile-contiguous expert weights (launch_retile): 128-byte rows, boxes of
  // 256 consecutive rows
  const uint64_t wb = h->fp8 ? 1 : 2;
  auto enc = [&](int which, const void* p, uint64_t rows, uint64_t cols) {
    const uint64_t rows128 = rows * cols * wb / 128;
    return h->fp8 ? asap::encode_tmap_u8(&out->map[which], p, rows128, 128, asap::kGemmBN, &err)
                  : asap::encode_tmap_bf16(&out->map[which], p, rows128, 64, asap::kGemmBN, &err);
  };
  if (!enc(asap::MAP_GATE_UP, L.gate_up, E * 2 * I, H)) return fail(ASAP_ERR_CUDA, "gate/up map: " + err);
  if (!enc(asap::MAP_DOWN, L.down, E * H, I)) return fail(ASAP_ERR_CUDA, "down map: " + err);
  if (c.n_shared) {
    if (!enc(asap::MAP_SH_GATE_UP, L.sh_gate_up, 2 * Is, H)) return fail(ASAP_ERR_CUDA, "shared gate/up map: " + err);
    if (!enc(asap::MAP_SH_DOWN, L.sh_down, H, Is)) return fail(ASAP_ERR_CUDA, "shared down map: " + err);
  }
  out->scale[asap::MAP_GATE_UP] = L.gu_scales;
  out->scale[asap::MAP_DOWN] = L.d_scales;
  out->scale[asap::MAP_SH_GATE_UP] = L.sh_gu_scales;
  out->scale[asap::MAP_SH_DOWN] = L.sh_d_scales;
  out->router_w = L.router_w;
  out->router_bias = L.router_bias;
  return ASAP_OK;
}

}  // namespace

ASAP_API int asap_moe_create_layers(const asap_moe_config* cfg, const asap_moe_weights* wts, int32_t n_layers,
                                    asap_moe_t* out) {
  if (!out) return fail(ASAP_ERR_INVALID, "NULL out");
  *out = nullptr;
  int r = asap_moe_check_config(cfg);
  if (r != ASAP_OK) return r;
  if (n_layers < 1 || n_layers > kMaxLayers)
    return fail(ASAP_ERR_INVALID, "n_layers must be in [1, " + std::to_string(kMaxLayers) + "]");
  if (!wts) return fail(ASAP_ERR_INVALID, "router and expert weights are required");
  for (int l = 0; l < n_layers; ++l)
    if ((r = check_weights(*cfg, wts + l)) != ASAP_OK) return fail(r, "layer " + std::to_string(l) + ": " + g_last_error);
  const asap_moe_config& c = *cfg;
  asap_moe_s* h = new asap_moe_s();
  h->cfg = c;
  h->layers.resize(n_layers);
  cudaStream_t st = nullptr;
  auto bail = [&](int code) {
    if (st) cudaStreamDestroy(st);
    asap_moe_destroy(h);
    return code;
  };
  cudaError_t e = cudaGetDevice(&h->device);
  if (e != cudaSuccess) return bail(cuda_fail(e, "cudaGetDevice"));
  // The weights may still be in flight on any of the caller's streams; the
  // copies below run on a private non-blocking stream, so wait for all of it.
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return bail(cuda_fail(e, "synchronise before reading the weights"));
  e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (e != cudaSuccess) return bail(cuda_fail(e, "SM count"));
  int cc_major = 0, cc_minor = 0;
  cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, h->device);
  cudaDeviceGetAttribute(&cc_minor, cudaDevAttrComputeCapabilityMinor, h->device);
  if (cc_major != 10 || cc_minor != 3)
    return bail(fail(ASAP_ERR_UNSUPPORTED, "libasap_moe is built for sm_103a (GB300) only; device is sm_" +
                                               std::to_string(cc_major) + std::to_string(cc_minor)));
  e = asap::gemm_set_attributes();
  if (e == cudaSuccess) e = asap::fp8_gemm_set_attributes();
  if (e == cudaSuccess) e = asap::route_fused_set_attributes();
  if (e != cudaSuccess) return bail(cuda_fail(e, "GEMM attributes"));
  h->fp8 = c.dtype == ASAP_FP8_E4M3_BLOCK128;
  h->tc_router = (c.n_experts == asap::kGemmBN);
  e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking);
  if (e != cudaSuccess) return bail(cuda_fail(e, "stream"));
  if ((e = cudaMalloc(&h->status, 256)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc status"));
  if ((e = cudaMemsetAsync(h->status, 0, 256, st)) != cudaSuccess) return bail(cuda_fail(e, "memset"));
  for (int l = 0; l < n_layers; ++l)
    if ((r = pack_layer(h, wts + l, h->layers[l], st)) != ASAP_OK)
      return bail(fail(r, "layer " + std::to_string(l) + ": " + g_last_error));
  // the layer table and the fixed ids 0 .. n_layers-1
  std::vector<asap::LayerEntry> table(n_layers);
  std::vector<int32_t> ids(n_layers);
  for (int l = 0; l < n_layers; ++l) {
    if ((r = encode_layer(h, h->layers[l], &table[l])) != ASAP_OK)
      return bail(fail(r, "layer " + std::to_string(l) + ": " + g_last_error));
    ids[l] = l;
  }
  const size_t tb = sizeof(asap::LayerEntry) * n_layers;
  if ((e = cudaMalloc(&h->table, tb)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc layer table"));
  if ((e = cudaMalloc(&h->layer_ids, 4 * n_layers)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc layer ids"));
  // (pageable host sources, complete by the stream synchronisation below)
  if ((e = cudaMemcpyAsync(h->table, table.data(), tb, cudaMemcpyHostToDevice, st)) != cudaSuccess ||
      (e = cudaMemcpyAsync(h->layer_ids, ids.data(), 4 * n_layers, cudaMemcpyHostToDevice, st)) != cudaSuccess)
    return bail(cuda_fail(e, "copy layer table"));
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return bail(cuda_fail(e, "create sync"));
  cudaStreamDestroy(st);
  st = nullptr;
  *out = h;
  return ASAP_OK;
}

ASAP_API int asap_moe_create(const asap_moe_config* cfg, const asap_moe_weights* wts, asap_moe_t* out) {
  if (!out) return fail(ASAP_ERR_INVALID, "NULL out");
  *out = nullptr;
  int r = asap_moe_check_config(cfg);
  if (r != ASAP_OK) return r;
  if ((r = check_weights(*cfg, wts)) != ASAP_OK) return r;
  return asap_moe_create_layers(cfg, wts, 1, out);
}

ASAP_API int asap_moe_router_logits(asap_moe_t h, const void* x, int32_t n, float* logits, void* ws,
                                    size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !logits || !aligned16(x) || !aligned16(logits))
    return fail(ASAP_ERR_INVALID, "x and logits must be non-NULL and 16-byte aligned");
  const int splits = router_splits(h, n);
  if (splits == 1) return run_router_logits(h, x, n, logits, 1, h->layer_ids, S(stream));
  // the same K slices and the same order of addition as asap_moe_route
  float* parts = at<float>(ws, layout(h->cfg, n).logits);
  if ((r = run_router_logits(h, x, n, parts, splits, h->layer_ids, S(stream))) != ASAP_OK) return r;
  CU_TRY(asap::launch_reduce_splits(parts, splits, static_cast<long long>(n) * h->cfg.n_experts, logits, S(stream)),
         "logit reduction launch");
  return ASAP_OK;
}

ASAP_API int asap_moe_route_logits(asap_moe_t h, const float* logits, int32_t n, int32_t* idx, float* w,
                                   int32_t* counts, int32_t* offsets, void* ws, size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!logits || !idx || !w || !counts || !offsets) return fail(ASAP_ERR_INVALID, "NULL tensor");
  return run_gate_scan(h, logits, 1, n, idx, w, counts, offsets, ws, h->layer_ids, S(stream));
}

ASAP_API int asap_moe_route(asap_moe_t h, const void* x, int32_t n, int32_t* idx, float* w, int32_t* counts,
                            int32_t* offsets, void* ws, size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !idx || !w || !counts || !offsets || !aligned16(x)) return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  return run_route(h, x, n, idx, w, counts, offsets, ws, h->layer_ids, S(stream));
}

ASAP_API int asap_moe_dispatch(asap_moe_t h, const void* x, int32_t n, const int32_t* idx, void* x_perm,
                               float* x_perm_scales, int32_t* perm_src, int32_t* perm_dst, void* ws,
                               size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !idx || !x_perm || !perm_src || !perm_dst || !aligned16(x) || !aligned16(x_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->fp8 && !x_perm_scales) return fail(ASAP_ERR_INVALID, "the FP8 configuration needs x_perm_scales");
  const asap_moe_config& c = h->cfg;
  const Layout L = layout(c, n);
  const int chunks = asap::ceil_div(n, asap::kChunkTokens);
  cudaStream_t st = S(stream);
  int32_t* hist = at<int32_t>(ws, L.hist);
  int32_t* base = at<int32_t>(ws, L.chunk_base);
  int32_t* ticket = at<int32_t>(ws, L.ticket);
  int32_t* offs = at<int32_t>(ws, L.offsets);
  CU_TRY(asap::launch_hist(idx, n, c.top_k, c.n_experts, hist, h->status, ticket, st), "hist launch");
  CU_TRY(asap::launch_scan(hist, chunks, c.n_experts, at<int32_t>(ws, L.counts), offs, base, ticket, st),
         "scan launch");
  if (h->fp8)
    CU_TRY(asap::launch_dispatch_fp8(x, n, c.hidden, c.top_k, c.n_experts, idx, base, offs, x_perm, x_perm_scales,
                                     nullptr, nullptr, perm_src, perm_dst, h->status, st),
           "dispatch launch");
  else
    CU_TRY(asap::launch_dispatch(x, n, c.hidden, c.top_k, c.n_experts, idx, base, offs, x_perm, perm_src, perm_dst,
                                 h->status, st),
           "dispatch launch");
  return ASAP_OK;
}

ASAP_API int asap_moe_expert_ffn(asap_moe_t h, const void* x_perm, const float* x_perm_scales,
                                 const int32_t* offsets, const void* x, int32_t n, void* y_perm, void* y_shared,
                                 void* ws, size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x_perm || !offsets || !y_perm || !aligned16(x_perm) || !aligned16(y_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->cfg.n_shared && (!x || !y_shared || !aligned16(x) || !aligned16(y_shared)))
    return fail(ASAP_ERR_INVALID, "x and y_shared are required for the shared expert");
  const Layout L = layout(h->cfg, n);
  cudaStream_t st = S(stream);
  int32_t* counters = at<int32_t>(ws, L.tile_counters);
  CU_TRY(cudaMemsetAsync(counters, 0, asap::kTileCounters * sizeof(int32_t), st), "tile counters");
  if (h->fp8) {
    if (!x_perm_scales) return fail(ASAP_ERR_INVALID, "the FP8 configuration needs x_perm_scales");
    const asap_moe_config& c = h->cfg;
    void* xq_sh = c.n_shared ? at<void>(ws, L.xq_sh) : nullptr;
    float* xs_sh = c.n_shared ? at<float>(ws, L.xs_sh) : nullptr;
    if (c.n_shared) CU_TRY(asap::launch_quantize_rows(x, n, c.hidden, xq_sh, xs_sh, st), "quantise launch");
    if ((r = run_gate_up_fp8(h, x_perm, x_perm_scales, offsets, xq_sh, xs_sh, n, at<void>(ws, L.hq),
                             at<float>(ws, L.hs), at<void>(ws, L.hq_sh), at<float>(ws, L.hs_sh), h->layer_ids,
                             counters, st)) != ASAP_OK)
      return r;
    return run_down_fp8(h, at<void>(ws, L.hq), at<float>(ws, L.hs), offsets, at<void>(ws, L.hq_sh),
                        at<float>(ws, L.hs_sh), n, y_perm, y_shared, h->layer_ids, counters + 1, st);
  }
  return run_expert_ffn(h, x_perm, offsets, x, n, y_perm, y_shared, at<void>(ws, L.h), at<void>(ws, L.h_sh),
                        h->layer_ids, counters, st);
}

namespace {

// Tile counter of a standalone GEMM call: workspace slot 0, cleared on the
// stream; nullptr (static tile order) without a workspace.
int standalone_counter(asap_moe_t h, int32_t n, void* ws, size_t ws_bytes, cudaStream_t st, int32_t** out) {
  *out = nullptr;
  if (!ws) return ASAP_OK;
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK) return r;
  *out = at<int32_t>(ws, layout(h->cfg, n).tile_counters);
  CU_TRY(cudaMemsetAsync(*out, 0, sizeof(int32_t), st), "tile counter");
  return ASAP_OK;
}

}  // namespace

ASAP_API int asap_moe_expert_gate_up(asap_moe_t h, const void* x_perm, const float* x_perm_scales,
                                     const int32_t* offsets, const void* x, int32_t n, void* h_perm,
                                     void* h_shared, void* ws, size_t ws_bytes, void* stream) {
  (void)x_perm_scales;
  int r = check_call(h, n, nullptr, 0, false);
  if (r != ASAP_OK || n == 0) return r;
  if (h->fp8) return fail(ASAP_ERR_UNSUPPORTED, "the FP8 configuration runs the FFN through asap_moe_expert_ffn");
  if (!x_perm || !offsets || !h_perm || !aligned16(x_perm) || !aligned16(h_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->cfg.n_shared && (!x || !h_shared || !aligned16(x) || !aligned16(h_shared)))
    return fail(ASAP_ERR_INVALID, "x and h_shared are required for the shared expert");
  int32_t* counter = nullptr;
  if ((r = standalone_counter(h, n, ws, ws_bytes, S(stream), &counter)) != ASAP_OK) return r;
  return run_gate_up(h, x_perm, offsets, x, n, h_perm, h_shared, h->layer_ids, counter, S(stream));
}

ASAP_API int asap_moe_expert_down(asap_moe_t h, const void* h_perm, const float* h_perm_scales,
                                  const int32_t* offsets, const void* h_shared, int32_t n, void* y_perm,
                                  void* y_shared, void* ws, size_t ws_bytes, void* stream) {
  (void)h_perm_scales;
  int r = check_call(h, n, nullptr, 0, false);
  if (r != ASAP_OK || n == 0) return r;
  if (h->fp8) return fail(ASAP_ERR_UNSUPPORTED, "the FP8 configuration runs the FFN through asap_moe_expert_ffn");
  if (!h_perm || !offsets || !y_perm || !aligned16(h_perm) || !aligned16(y_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->cfg.n_shared && (!h_shared || !y_shared || !aligned16(h_shared) || !aligned16(y_shared)))
    return fail(ASAP_ERR_INVALID, "h_shared and y_shared are required for the shared expert");
  int32_t* counter = nullptr;
  if ((r = standalone_counter(h, n, ws, ws_bytes, S(stream), &counter)) != ASAP_OK) return r;
  return run_down(h, h_perm, offsets, h_shared, n, y_perm, y_shared, h->layer_ids, counter, S(stream));
}

ASAP_API int asap_moe_combine(asap_moe_t h, const void* y_perm, const void* y_shared, const float* w,
                              const int32_t* perm_dst, int32_t n, void* out, void* stream) {
  int r = check_call(h, n, nullptr, 0, false);
  if (r != ASAP_OK || n == 0) return r;
  if (!y_perm || !w || !perm_dst || !out || !aligned16(y_perm) || !aligned16(out) ||
      (y_shared && !aligned16(y_shared)))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  CU_TRY(asap::launch_combine(y_perm, y_shared, w, perm_dst, n, h->cfg.hidden, h->cfg.top_k, out, h->status,
                              S(stream)),
         "combine launch");
  return ASAP_OK;
}

namespace {

// Events that asap_moe_time_layer asked this thread's next layer call to
// record: before its first kernel and after each of its five steps.
constexpr int kLayerEvents = 6;
thread_local cudaEvent_t g_layer_ev[kLayerEvents] = {};

// The pending events of this thread, taken (the request is cleared) when a
// layer call starts, so each request serves one call whatever its outcome.
struct LayerEvents {
  cudaEvent_t ev[kLayerEvents] = {};
  LayerEvents() {
    for (int i = 0; i < kLayerEvents; ++i) {
      ev[i] = g_layer_ev[i];
      g_layer_ev[i] = nullptr;
    }
  }
  cudaError_t mark(int i, cudaStream_t st) const { return ev[i] ? cudaEventRecord(ev[i], st) : cudaSuccess; }
};

// The whole layer for one micro-batch, weights of layer *layer (device).
int run_layer(asap_moe_t h, const void* x, int32_t n, void* out, void* ws, size_t ws_bytes, const int32_t* layer,
              void* stream, const LayerEvents& tev) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !out || !aligned16(x) || !aligned16(out)) return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  const asap_moe_config& c = h->cfg;
  const Layout L = layout(c, n);
  cudaStream_t st = S(stream);
  float* logits = at<float>(ws, L.logits);
  int32_t* idx = at<int32_t>(ws, L.idx);
  float* w = at<float>(ws, L.w);
  int32_t* counts = at<int32_t>(ws, L.counts);
  int32_t* offsets = at<int32_t>(ws, L.offsets);
  int32_t* perm_src = at<int32_t>(ws, L.perm_src);
  int32_t* perm_dst = at<int32_t>(ws, L.perm_dst);
  int32_t* counters = at<int32_t>(ws, L.tile_counters);  // zeroed by the scan kernel
  void* y_sh = c.n_shared ? at<void>(ws, L.y_sh) : nullptr;
  CU_TRY(tev.mark(0, st), "timing event");
  if ((r = run_route(h, x, n, idx, w, counts, offsets, ws, layer, st)) != ASAP_OK) return r;
  CU_TRY(tev.mark(1, st), "timing event");
  if (h->fp8) {
    void* xq_sh = c.n_shared ? at<void>(ws, L.xq_sh) : nullptr;
    float* xs_sh = c.n_shared ? at<float>(ws, L.xs_sh) : nullptr;
    CU_TRY(asap::launch_dispatch_fp8(x, n, c.hidden, c.top_k, c.n_experts, idx, at<int32_t>(ws, L.chunk_base),
                                     offsets, at<void>(ws, L.xq), at<float>(ws, L.xs), xq_sh, xs_sh, perm_src,
                                     perm_dst, h->status, st),
           "dispatch launch");
    CU_TRY(tev.mark(2, st), "timing event");
    if ((r = run_gate_up_fp8(h, at<void>(ws, L.xq), at<float>(ws, L.xs), offsets, xq_sh, xs_sh, n, at<void>(ws, L.hq),
                             at<float>(ws, L.hs), at<void>(ws, L.hq_sh), at<float>(ws, L.hs_sh), layer, counters,
                             st)) != ASAP_OK)
      return r;
    CU_TRY(tev.mark(3, st), "timing event");
    void* y_perm = at<void>(ws, L.y_perm);
    if ((r = run_down_fp8(h, at<void>(ws, L.hq), at<float>(ws, L.hs), offsets, at<void>(ws, L.hq_sh),
                          at<float>(ws, L.hs_sh), n, y_perm, y_sh, layer, counters + 1, st)) != ASAP_OK)
      return r;
    CU_TRY(tev.mark(4, st), "timing event");
    CU_TRY(asap::launch_combine(y_perm, y_sh, w, perm_dst, n, c.hidden, c.top_k, out, h->status, st),
           "combine launch");
    CU_TRY(tev.mark(5, st), "timing event");
    return ASAP_OK;
  }
  void* x_perm = at<void>(ws, L.x_perm);
  CU_TRY(asap::launch_dispatch(x, n, c.hidden, c.top_k, c.n_experts, idx, at<int32_t>(ws, L.chunk_base), offsets,
                               x_perm, perm_src, perm_dst, h->status, st),
         "dispatch launch");
  CU_TRY(tev.mark(2, st), "timing event");
  // y_perm reuses x_perm's rows: the down GEMM never reads x_perm
  void* hbuf = at<void>(ws, L.h);
  void* hsh = at<void>(ws, L.h_sh);
  if ((r = run_gate_up(h, x_perm, offsets, x, n, hbuf, hsh, layer, counters, st)) != ASAP_OK) return r;
  CU_TRY(tev.mark(3, st), "timing event");
  if (h->combine == ASAP_COMBINE_FUSED) {
    CombineFuse cf;
    cf.cnt = at<int>(ws, L.comb_cnt);
    cf.src = perm_src;
    cf.dst = perm_dst;
    cf.w = w;
    cf.out = out;
    CU_TRY(cudaMemsetAsync(cf.cnt, 0, sizeof(int) * static_cast<size_t>(n) * (c.hidden / asap::kGemmBN), st),
           "slice counters");
    if ((r = run_down(h, hbuf, offsets, hsh, n, x_perm, y_sh, layer, counters + 1, st, nullptr, cf)) != ASAP_OK)
      return r;
    CU_TRY(tev.mark(4, st), "timing event");
    CU_TRY(tev.mark(5, st), "timing event");  // the combine ran inside the down GEMM
    return ASAP_OK;
  }
  if ((r = run_down(h, hbuf, offsets, hsh, n, x_perm, y_sh, layer, counters + 1, st)) != ASAP_OK) return r;
  CU_TRY(tev.mark(4, st), "timing event");
  CU_TRY(asap::launch_combine(x_perm, y_sh, w, perm_dst, n, c.hidden, c.top_k, out, h->status, st),
         "combine launch");
  CU_TRY(tev.mark(5, st), "timing event");
  return ASAP_OK;
}

int run_layer_batched(asap_moe_t h, int32_t count, const void* const* xs, const int32_t* ns, void* const* outs,
                      void* ws, size_t ws_bytes, const int32_t* layer, void* stream) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  if (count < 1 || count > kMaxBatch || !xs || !ns || !outs)
    return fail(ASAP_ERR_INVALID, "count must be in [1, 64] with host arrays xs, ns, outs");
  long long N = 0;
  for (int i = 0; i < count; ++i) {
    if (ns[i] < 0) return fail(ASAP_ERR_INVALID, "negative micro-batch size");
    if (ns[i] > 0 && (!xs[i] || !outs[i] || !aligned16(xs[i]) || !aligned16(outs[i])))
      return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
    N += ns[i];
  }
  if (N > h->cfg.max_tokens)
    return fail(ASAP_ERR_INVALID, "the micro-batches hold " + std::to_string(N) + " tokens, more than max_tokens");
  int r = check_call(h, static_cast<int32_t>(N), ws, ws_bytes, true);
  if (r != ASAP_OK || N == 0) return r;
  const asap_moe_config& c = h->cfg;
  const int n_all = static_cast<int>(N);
  const Layout L = layout(c, n_all);
  cudaStream_t st = S(stream);
  const int k = c.top_k, E = c.n_experts;
  const long long nk = N * k;
  float* logits = at<float>(ws, L.logits);
  int32_t* idx = at<int32_t>(ws, L.idx);
  float* w = at<float>(ws, L.w);
  int32_t* hist = at<int32_t>(ws, L.hist);
  int32_t* base = at<int32_t>(ws, L.chunk_base);
  int32_t* offsets = at<int32_t>(ws, L.offsets);
  int32_t* perm_src = at<int32_t>(ws, L.perm_src);
  int32_t* perm_dst = at<int32_t>(ws, L.perm_dst);
  int32_t* counters = at<int32_t>(ws, L.tile_counters);  // zeroed by the scan kernel
  int chunks_total = 0;
  for (int i = 0; i < count; ++i) chunks_total += asap::ceil_div(ns[i], asap::kChunkTokens);
  // routing: each micro-batch exactly as asap_moe_route would route it alone
  int tok0 = 0, chunk0 = 0;
  for (int i = 0; i < count; ++i) {
    const int n = ns[i];
    if (n > 0 && fused_route(h)) {
      if ((r = run_route_fused(h, xs[i], n, idx + static_cast<long long>(tok0) * k,
                               w + static_cast<long long>(tok0) * k, hist, chunk0, chunks_total, nullptr, nullptr,
                               nullptr, nullptr, nullptr, layer, st)) != ASAP_OK)
        return r;
    } else if (n > 0) {
      const int splits = router_splits(h, n);
      float* lg = logits + static_cast<long long>(asap::kMaxRouterSplits) * tok0 * E;
      if ((r = run_router_logits(h, xs[i], n, lg, splits, layer, st)) != ASAP_OK) return r;
      CU_TRY(asap::launch_gate_seg(lg, splits, n, gate_params(h, layer, at<int32_t>(ws, L.ticket)),
                                   idx + static_cast<long long>(tok0) * k,
                                   w + static_cast<long long>(tok0) * k, hist, chunk0, chunks_total, st),
             "gate launch");
    }
    tok0 += n;
    chunk0 += asap::ceil_div(n, asap::kChunkTokens);
  }
  // one histogram scan over every chunk: expert segments hold the rows of all
  // micro-batches, in (micro-batch, token, slot) order (the scan's ticket is
  // zero at launch: the gate kernels zero it, the fused route does not)
  if (fused_route(h)) CU_TRY(cudaMemsetAsync(at<int32_t>(ws, L.ticket), 0, 4, st), "ticket");
  CU_TRY(asap::launch_scan(hist, chunks_total, E, at<int32_t>(ws, L.counts), offsets, base, at<int32_t>(ws, L.ticket),
                           st, at<int32_t>(ws, L.tile_counters)),
         "scan launch");
  void* y_sh = c.n_shared ? at<void>(ws, L.y_sh) : nullptr;
  tok0 = 0;
  chunk0 = 0;
  for (int i = 0; i < count; ++i) {
    const int n = ns[i];
    if (n > 0) {
      asap::DispatchSeg seg{};
      seg.expert_offsets = offsets;
      seg.chunk0 = chunk0;
      seg.n_chunks_total = chunks_total;
      seg.tok0 = tok0;
      seg.rows_total = nk;
      const int32_t* idx_i = idx + static_cast<long long>(tok0) * k;
      int32_t* pd_i = perm_dst + static_cast<long long>(tok0) * k;
      if (h->fp8) {
        void* xq_sh = c.n_shared ? static_cast<uint8_t*>(at<void>(ws, L.xq_sh)) + static_cast<long long>(tok0) * c.hidden
                                 : nullptr;
        float* xs_sh = c.n_shared ? at<float>(ws, L.xs_sh) + static_cast<long long>(tok0) * (c.hidden / 128) : nullptr;
        CU_TRY(asap::launch_dispatch_fp8_seg(xs[i], n, c.hidden, k, E, idx_i, base, at<void>(ws, L.xq),
                                             at<float>(ws, L.xs), xq_sh, xs_sh, perm_src, pd_i, h->status, seg, st),
               "dispatch launch");
      } else {
        // the shared expert reads the gathered rows from y_sh's region, which
        // its own output overwrites only after the gate/up GEMM
        seg.x_sh = y_sh ? static_cast<uint16_t*>(y_sh) + static_cast<long long>(tok0) * c.hidden : nullptr;
        CU_TRY(asap::launch_dispatch_seg(xs[i], n, c.hidden, k, E, idx_i, base, at<void>(ws, L.x_perm), perm_src, pd_i,
                                         h->status, seg, st),
               "dispatch launch");
      }
    }
    tok0 += n;
    chunk0 += asap::ceil_div(n, asap::kChunkTokens);
  }
  // one grouped GEMM per weight matrix over every micro-batch's rows
  void* y_perm;
  if (h->fp8) {
    void* xq_sh = c.n_shared ? at<void>(ws, L.xq_sh) : nullptr;
    float* xs_sh = c.n_shared ? at<float>(ws, L.xs_sh) : nullptr;
    if ((r = run_gate_up_fp8(h, at<void>(ws, L.xq), at<float>(ws, L.xs), offsets, xq_sh, xs_sh, n_all,
                             at<void>(ws, L.hq), at<float>(ws, L.hs), at<void>(ws, L.hq_sh), at<float>(ws, L.hs_sh),
                             layer, counters, st)) != ASAP_OK)
      return r;
    y_perm = at<void>(ws, L.y_perm);
    if ((r = run_down_fp8(h, at<void>(ws, L.hq), at<float>(ws, L.hs), offsets, at<void>(ws, L.hq_sh),
                          at<float>(ws, L.hs_sh), n_all, y_perm, y_sh, layer, counters + 1, st)) != ASAP_OK)
      return r;
  } else {
    y_perm = at<void>(ws, L.x_perm);
    if ((r = run_gate_up(h, y_perm, offsets, y_sh, n_all, at<void>(ws, L.h), at<void>(ws, L.h_sh), layer, counters,
                         st)) != ASAP_OK)
      return r;
    if ((r = run_down(h, at<void>(ws, L.h), offsets, at<void>(ws, L.h_sh), n_all, y_perm, y_sh, layer, counters + 1,
                      st)) != ASAP_OK)
      return r;
  }
  tok0 = 0;
  for (int i = 0; i < count; ++i) {
    const int n = ns[i];
    if (n > 0) {
      const void* ysh_i = y_sh ? static_cast<const uint16_t*>(y_sh) + static_cast<long long>(tok0) * c.hidden : nullptr;
      CU_TRY(asap::launch_combine(y_perm, ysh_i, w + static_cast<long long>(tok0) * k,
                                  perm_dst + static_cast<long long>(tok0) * k, n, c.hidden, k, outs[i], h->status, st,
                                  nk),
             "combine launch");
    }
    tok0 += n;
  }
  return ASAP_OK;
}

bool valid_layer_ptr(const int32_t* layer) {
  return layer && (reinterpret_cast<uintptr_t>(layer) & 3u) == 0;
}

}  // namespace

ASAP_API int asap_moe_time_layer(int32_t count, void* const* events) {
  if (count < 0 || count > kLayerEvents || (count > 0 && !events))
    return fail(ASAP_ERR_INVALID, "count must be in [0, " + std::to_string(kLayerEvents) + "] with an events array");
  for (int i = 0; i < kLayerEvents; ++i) g_layer_ev[i] = i < count ? static_cast<cudaEvent_t>(events[i]) : nullptr;
  return ASAP_OK;
}

ASAP_API int asap_moe_layer(asap_moe_t h, const void* x, int32_t n, void* out, void* ws, size_t ws_bytes,
                            void* stream) {
  const LayerEvents tev;  // taken by this call whatever its outcome
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  return run_layer(h, x, n, out, ws, ws_bytes, h->layer_ids, stream, tev);
}

ASAP_API int asap_moe_layer_dyn(asap_moe_t h, const int32_t* layer_id, const void* x, int32_t n, void* out,
                                void* ws, size_t ws_bytes, void* stream) {
  const LayerEvents tev;
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  if (!valid_layer_ptr(layer_id)) return fail(ASAP_ERR_INVALID, "layer_id must be a non-NULL 4-byte aligned device pointer");
  return run_layer(h, x, n, out, ws, ws_bytes, layer_id, stream, tev);
}

ASAP_API int asap_moe_layer_batched(asap_moe_t h, int32_t count, const void* const* xs, const int32_t* ns,
                                    void* const* outs, void* ws, size_t ws_bytes, void* stream) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  return run_layer_batched(h, count, xs, ns, outs, ws, ws_bytes, h->layer_ids, stream);
}

ASAP_API int asap_moe_layer_batched_dyn(asap_moe_t h, const int32_t* layer_id, int32_t count, const void* const* xs,
                                        const int32_t* ns, void* const* outs, void* ws, size_t ws_bytes,
                                        void* stream) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  if (!valid_layer_ptr(layer_id)) return fail(ASAP_ERR_INVALID, "layer_id must be a non-NULL 4-byte aligned device pointer");
  return run_layer_batched(h, count, xs, ns, outs, ws, ws_bytes, layer_id, stream);
}

ASAP_API int asap_moe_n_layers(asap_moe_t h, int32_t* n_layers) {
  if (!h || !n_layers) return fail(ASAP_ERR_INVALID, "NULL handle or output");
  *n_layers = static_cast<int32_t>(h->layers.size());
  return ASAP_OK;
}

ASAP_API int asap_moe_set_tiling(asap_moe_t h, int32_t mode) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  if (mode != ASAP_TILING_AUTO && mode != ASAP_TILING_SINGLE && mode != ASAP_TILING_PAIRED)
    return fail(ASAP_ERR_INVALID, "tiling mode must be ASAP_TILING_AUTO, _SINGLE or _PAIRED");
  h->tiling = mode;
  return ASAP_OK;
}

ASAP_API int asap_moe_set_combine(asap_moe_t h, int32_t mode) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  if (mode != ASAP_COMBINE_SEPARATE && mode != ASAP_COMBINE_FUSED)
    return fail(ASAP_ERR_INVALID, "combine mode must be ASAP_COMBINE_SEPARATE or ASAP_COMBINE_FUSED");
  if (mode == ASAP_COMBINE_FUSED && h->fp8)
    return fail(ASAP_ERR_UNSUPPORTED, "the combine is fused into the bf16 down GEMM only");
  h->combine = mode;
  return ASAP_OK;
}

ASAP_API int asap_moe_status(asap_moe_t h, uint32_t* word) {
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(h->device);
  uint32_t v = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(&v, h->status, 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemset(h->status, 0, 4);
  cudaSetDevice(prev);
  if (e != cudaSuccess) return cuda_fail(e, "status read");
  if (word) *word = v;
  if (v != 0) return fail(ASAP_ERR_DEVICE_STATUS, "device status word " + std::to_string(v));
  return ASAP_OK;
}

// ============================================================ mailbox (device-side ready set)
//
// The single-GPU form of ASAP's asynchronous dispatch and combine (Sections
// 3.2.1 and 3.2.2) with ready-set aggregation: DP groups post routed
// micro-batches into slots on their own streams; a service round on the MoE
// stream claims every post that is ready when the round starts (decided on
// the device) and serves all of them with one grouped GEMM pass, so each
// expert's weights stream from HBM once per round instead of once per
// micro-batch.  Host state is only bookkeeping (epochs, events); nothing here
// reads device memory back.

struct asap_moe_mailbox_s {
  asap_moe_t h = nullptr;
  asap::MboxGeom g{};
  const int32_t* layer = nullptr;  // device layer id of posts made without one
  unsigned long long wait_ns = 0;
  Layout L{};                      // server workspace: layout for n_slots * slot_tokens tokens
  void* ws = nullptr;
  asap::MboxSlot* slots = nullptr;
  asap::MboxRound* round = nullptr;
  int32_t* rowmap = nullptr;
  int32_t* log = nullptr;
  unsigned long long* served_host = nullptr;      // host-mapped completion epochs
  unsigned long long* served_host_dev = nullptr;  // its device address
  std::vector<cudaEvent_t> post_ev, served_ev;
  std::vector<unsigned long long> posted, serve_called;  // host view: last post, last serve call per slot
  cudaEvent_t gemm_ev0 = nullptr, gemm_ev1 = nullptr;   // recorded around the next round's GEMMs
  cudaEvent_t round_ev = nullptr;  // end of the last round (rounds share the server workspace)
  bool any_round = false;
  std::mutex mu;
};

namespace {

int mbox_free(asap_moe_mailbox_t m) {
  if (!m) return ASAP_OK;
  int prev = 0;
  cudaGetDevice(&prev);
  if (m->h) cudaSetDevice(m->h->device);
  cudaDeviceSynchronize();
  cudaFree(m->ws);
  cudaFree(m->slots);
  cudaFree(m->round);
  cudaFree(m->rowmap);
  cudaFree(m->log);
  if (m->served_host) cudaFreeHost(m->served_host);
  for (cudaEvent_t e : m->post_ev) cudaEventDestroy(e);
  for (cudaEvent_t e : m->served_ev) cudaEventDestroy(e);
  if (m->round_ev) cudaEventDestroy(m->round_ev);
  cudaSetDevice(prev);
  delete m;
  return ASAP_OK;
}

}  // namespace

ASAP_API int asap_moe_mailbox_create(asap_moe_t h, int32_t n_slots, int32_t slot_tokens, const int32_t* layer_id,
                                     int64_t wait_ns, asap_moe_mailbox_t* out) {
  if (!out) return fail(ASAP_ERR_INVALID, "NULL out");
  *out = nullptr;
  if (!h) return fail(ASAP_ERR_INVALID, "NULL handle");
  const asap_moe_config& c = h->cfg;
  if (n_slots < 1 || n_slots > asap::kMboxMaxSlots)
    return fail(ASAP_ERR_INVALID, "n_slots must be in [1, " + std::to_string(asap::kMboxMaxSlots) + "]");
  if (slot_tokens < 1 || slot_tokens > c.max_tokens)
    return fail(ASAP_ERR_INVALID, "slot_tokens must be in [1, max_tokens]");
  const long long total = static_cast<long long>(n_slots) * slot_tokens;
  if (total * c.top_k >= (1ll << 31)) return fail(ASAP_ERR_INVALID, "n_slots * slot_tokens * top_k must be < 2^31");
  if (layer_id && !valid_layer_ptr(layer_id))
    return fail(ASAP_ERR_INVALID, "layer_id must be NULL or a 4-byte aligned device pointer");
  if (wait_ns <= 0) return fail(ASAP_ERR_INVALID, "wait_ns must be positive");
  asap_moe_mailbox_s* m = new asap_moe_mailbox_s();
  m->h = h;
  m->g.n_slots = n_slots;
  m->g.slot_tokens = slot_tokens;
  m->g.slot_chunks = asap::ceil_div(slot_tokens, asap::kChunkTokens);
  m->g.k = c.top_k;
  m->g.E = c.n_experts;
  m->g.H = c.hidden;
  m->layer = layer_id ? layer_id : h->layer_ids;
  m->wait_ns = static_cast<unsigned long long>(wait_ns);
  m->L = layout(c, total);
  auto bail = [&](int code) {
    mbox_free(m);
    return code;
  };
  int prev = 0;
  cudaGetDevice(&prev);
  cudaError_t e = cudaSetDevice(h->device);
  if (e != cudaSuccess) return bail(cuda_fail(e, "cudaSetDevice"));
  auto restore = [&](int code) {
    cudaSetDevice(prev);
    return code;
  };
  if ((e = cudaMalloc(&m->ws, m->L.total)) != cudaSuccess) return restore(bail(cuda_fail(e, "cudaMalloc mailbox workspace")));
  if ((e = cudaMalloc(&m->slots, sizeof(asap::MboxSlot) * n_slots)) != cudaSuccess ||
      (e = cudaMalloc(&m->round, sizeof(asap::MboxRound))) != cudaSuccess ||
      (e = cudaMalloc(&m->rowmap, sizeof(int32_t) * n_slots * m->g.slot_chunks)) != cudaSuccess ||
      (e = cudaMalloc(&m->log, sizeof(int32_t) * asap::kMboxLog)) != cudaSuccess)
    return restore(bail(cuda_fail(e, "cudaMalloc mailbox state")));
  if ((e = cudaHostAlloc(reinterpret_cast<void**>(&m->served_host), sizeof(unsigned long long) * n_slots,
                         cudaHostAllocMapped)) != cudaSuccess ||
      (e = cudaHostGetDevicePointer(reinterpret_cast<void**>(&m->served_host_dev), m->served_host, 0)) != cudaSuccess)
    return restore(bail(cuda_fail(e, "mapped completion flags")));
  std::memset(m->served_host, 0, sizeof(unsigned long long) * n_slots);
  if ((e = cudaMemset(m->slots, 0, sizeof(asap::MboxSlot) * n_slots)) != cudaSuccess ||
      (e = cudaMemset(m->round, 0, sizeof(asap::MboxRound))) != cudaSuccess ||
      (e = cudaMemset(m->log, 0, sizeof(int32_t) * asap::kMboxLog)) != cudaSuccess)
    return restore(bail(cuda_fail(e, "clear mailbox state")));
  m->post_ev.assign(n_slots, nullptr);
  m->served_ev.assign(n_slots, nullptr);
  for (int i = 0; i < n_slots; ++i)
    if ((e = cudaEventCreateWithFlags(&m->post_ev[i], cudaEventDisableTiming)) != cudaSuccess ||
        (e = cudaEventCreateWithFlags(&m->served_ev[i], cudaEventDisableTiming)) != cudaSuccess)
      return restore(bail(cuda_fail(e, "mailbox events")));
  if ((e = cudaEventCreateWithFlags(&m->round_ev, cudaEventDisableTiming)) != cudaSuccess)
    return restore(bail(cuda_fail(e, "mailbox events")));
  m->posted.assign(n_slots, 0);
  m->serve_called.assign(n_slots, 0);
  if ((e = cudaDeviceSynchronize()) != cudaSuccess) return restore(bail(cuda_fail(e, "mailbox create sync")));
  h->mailboxes.fetch_add(1);
  *out = m;
  return restore(ASAP_OK);
}

ASAP_API int asap_moe_mailbox_destroy(asap_moe_mailbox_t m) {
  if (!m) return ASAP_OK;
  asap_moe_t h = m->h;
  const int r = mbox_free(m);
  h->mailboxes.fetch_sub(1);
  return r;
}

ASAP_API int asap_moe_mailbox_post(asap_moe_mailbox_t m, int32_t slot, const void* x, int32_t n, void* out,
                                   const int32_t* layer_id, void* stream, uint64_t* epoch) {
  if (!m) return fail(ASAP_ERR_INVALID, "NULL mailbox");
  if (layer_id && !valid_layer_ptr(layer_id))
    return fail(ASAP_ERR_INVALID, "layer_id must be NULL or a 4-byte aligned device pointer");
  const int32_t* layer = layer_id ? layer_id : m->layer;
  asap_moe_t h = m->h;
  const asap_moe_config& c = h->cfg;
  if (slot < 0 || slot >= m->g.n_slots) return fail(ASAP_ERR_INVALID, "slot outside [0, n_slots)");
  if (n < 0 || n > m->g.slot_tokens) return fail(ASAP_ERR_INVALID, "n outside [0, slot_tokens]");
  if (n > 0 && (!x || !out || !aligned16(x) || !aligned16(out)))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  std::lock_guard<std::mutex> lock(m->mu);
  if (m->posted[slot] > m->serve_called[slot])
    return fail(ASAP_ERR_INVALID, "slot " + std::to_string(slot) + " still holds post " +
                                      std::to_string(m->posted[slot]) + ", for which no serve call has been made");
  cudaStream_t st = S(stream);
  const unsigned long long ep = m->posted[slot] + 1;
  // backpressure (Section 3.2.1): the round that served the slot's previous
  // post must be done with the slot's region before it is written again
  CU_TRY(cudaStreamWaitEvent(st, m->served_ev[slot], 0), "wait for the slot's previous round");
  const asap::MboxGeom& g = m->g;
  const long long sk = static_cast<long long>(slot) * g.slot_tokens * c.top_k;
  int32_t* idx = at<int32_t>(m->ws, m->L.idx) + sk;
  float* w = at<float>(m->ws, m->L.w) + sk;
  int32_t* hist = at<int32_t>(m->ws, m->L.hist);
  const int chunk0 = slot * g.slot_chunks, chunks_total = g.n_slots * g.slot_chunks;
  int r;
  if (n > 0) {
    // routing exactly as asap_moe_route routes n tokens; the histogram rows
    // are the slot's, scanned later together with the other claimed posts
    if (fused_route(h)) {
      if ((r = run_route_fused(h, x, n, idx, w, hist, chunk0, chunks_total, nullptr, nullptr, nullptr, nullptr,
                               nullptr, layer, st, /*narrow=*/true)) != ASAP_OK)
        return r;
    } else {
      const int splits = router_splits(h, n);
      float* lg = at<float>(m->ws, m->L.logits) +
                  static_cast<long long>(slot) * asap::kMaxRouterSplits * g.slot_tokens * c.n_experts;
      if ((r = run_router_logits(h, x, n, lg, splits, layer, st)) != ASAP_OK) return r;
      CU_TRY(asap::launch_gate_seg(lg, splits, n, gate_params(h, layer, nullptr), idx, w, hist, chunk0,
                                   chunks_total, st),
             "gate launch");
    }
  }
  CU_TRY(asap::launch_mbox_publish(m->slots, slot, x, n, out, layer, ep, h->status, st), "publish launch");
  CU_TRY(cudaEventRecord(m->post_ev[slot], st), "post event");
  m->posted[slot] = ep;
  if (epoch) *epoch = ep;
  return ASAP_OK;
}

namespace {

// One service round on st for the posts (slots[i], epochs[i]) (count >= 1,
// distinct slots, validated by the caller, mailbox lock held): the stream
// waits for each of those posts and for the previous round; the claim waits
// (bounded) for the first one's flag and claims every published, unserved
// post of its layer; each listed slot's served event is recorded after the
// round.
int serve_round(asap_moe_mailbox_t m, int count, const int32_t* slots, const uint64_t* epochs, cudaStream_t st,
                cudaEvent_t gemm_ev0, cudaEvent_t gemm_ev1) {
  asap_moe_t h = m->h;
  const asap_moe_config& c = h->cfg;
  const int32_t slot = slots[0];
  const uint64_t epoch = epochs[0];
  const asap::MboxGeom& g = m->g;
  const Layout& L = m->L;
  void* ws = m->ws;
  const int N = g.n_slots * g.slot_tokens;  // upper bound of the round's tokens
  const bool sh = c.n_shared != 0;
  int32_t* offsets = at<int32_t>(ws, L.offsets);
  int32_t* counters = at<int32_t>(ws, L.tile_counters);
  const int32_t* n_total = &m->round->n_total;
  const int32_t* layer = &m->round->layer;  // the layer of the claimed posts, written by the claim
  int r;
  // the post this round is for was published before the round starts; the
  // previous round (on whatever stream it was served) is done with the
  // server workspace
  for (int i = 0; i < count; ++i) CU_TRY(cudaStreamWaitEvent(st, m->post_ev[slots[i]], 0), "wait for the post");
  if (m->any_round) CU_TRY(cudaStreamWaitEvent(st, m->round_ev, 0), "wait for the previous round");
  CU_TRY(asap::launch_mbox_claim(m->slots, g, slot, epoch, m->wait_ns, m->round, m->rowmap, at<int32_t>(ws, L.ticket),
                                 h->status, st),
         "claim launch");
  CU_TRY(asap::launch_scan_mapped(at<int32_t>(ws, L.hist), m->rowmap, &m->round->chunks_total,
                                  g.n_slots * g.slot_chunks, c.n_experts, at<int32_t>(ws, L.counts), offsets,
                                  at<int32_t>(ws, L.chunk_base), at<int32_t>(ws, L.ticket), counters, st),
         "scan launch");
  const int32_t* idx = at<int32_t>(ws, L.idx);
  int32_t* perm_dst = at<int32_t>(ws, L.perm_dst);
  void* y_sh = sh ? at<void>(ws, L.y_sh) : nullptr;
  void* y_perm;
  if (h->fp8) {
    void* xq_sh = sh ? at<void>(ws, L.xq_sh) : nullptr;
    float* xs_sh = sh ? at<float>(ws, L.xs_sh) : nullptr;
    CU_TRY(asap::launch_dispatch_fp8_mbox(m->round, g, m->rowmap, idx, at<int32_t>(ws, L.chunk_base), offsets,
                                          at<void>(ws, L.xq),
                                          at<float>(ws, L.xs), xq_sh, xs_sh, at<int32_t>(ws, L.perm_src), perm_dst,
                                          h->status, st),
           "dispatch launch");
    if (gemm_ev0) CU_TRY(cudaEventRecord(gemm_ev0, st), "timing event");
    if ((r = run_gate_up_fp8(h, at<void>(ws, L.xq), at<float>(ws, L.xs), offsets, xq_sh, xs_sh, N, at<void>(ws, L.hq),
                             at<float>(ws, L.hs), at<void>(ws, L.hq_sh), at<float>(ws, L.hs_sh), layer, counters,
                             st, n_total)) != ASAP_OK)
      return r;
    y_perm = at<void>(ws, L.y_perm);
    if ((r = run_down_fp8(h, at<void>(ws, L.hq), at<float>(ws, L.hs), offsets, at<void>(ws, L.hq_sh),
                          at<float>(ws, L.hs_sh), N, y_perm, y_sh, layer, counters + 1, st, n_total)) != ASAP_OK)
      return r;
  } else {
    // the shared expert reads the gathered rows from y_sh's region, which its
    // own output overwrites only after the gate/up GEMM
    y_perm = at<void>(ws, L.x_perm);
    CU_TRY(asap::launch_dispatch_mbox(m->round, g, m->rowmap, idx, at<int32_t>(ws, L.chunk_base), offsets, y_perm,
                                      at<int32_t>(ws, L.perm_src), perm_dst, y_sh, h->status, st),
           "dispatch launch");
    if (gemm_ev0) CU_TRY(cudaEventRecord(gemm_ev0, st), "timing event");
    if ((r = run_gate_up(h, y_perm, offsets, y_sh, N, at<void>(ws, L.h), at<void>(ws, L.h_sh), layer, counters, st,
                         n_total)) != ASAP_OK)
      return r;
    if ((r = run_down(h, at<void>(ws, L.h), offsets, at<void>(ws, L.h_sh), N, y_perm, y_sh, layer, counters + 1,
                      st, n_total)) != ASAP_OK)
      return r;
  }
  if (gemm_ev1) CU_TRY(cudaEventRecord(gemm_ev1, st), "timing event");
  CU_TRY(asap::launch_combine_mbox(m->round, g, y_perm, y_sh, at<float>(ws, L.w), perm_dst, h->status, st),
         "combine launch");
  CU_TRY(asap::launch_mbox_finish(m->slots, m->round, m->log, m->served_host_dev, st), "finish launch");
  for (int i = 0; i < count; ++i) {
    CU_TRY(cudaEventRecord(m->served_ev[slots[i]], st), "served event");
    if (epochs[i] > m->serve_called[slots[i]]) m->serve_called[slots[i]] = epochs[i];
  }
  CU_TRY(cudaEventRecord(m->round_ev, st), "round event");
  m->any_round = true;
  return ASAP_OK;
}

}  // namespace

// The mailbox's pending GEMM timing events, taken (the request is cleared)
// by the serve call that starts now, whatever its outcome.  Mailbox lock held.
static std::pair<cudaEvent_t, cudaEvent_t> take_gemm_timing(asap_moe_mailbox_t m) {
  const std::pair<cudaEvent_t, cudaEvent_t> ev{m->gemm_ev0, m->gemm_ev1};
  m->gemm_ev0 = m->gemm_ev1 = nullptr;
  return ev;
}

ASAP_API int asap_moe_mailbox_serve(asap_moe_mailbox_t m, int32_t slot, uint64_t epoch, void* stream) {
  if (!m) return fail(ASAP_ERR_INVALID, "NULL mailbox");
  std::lock_guard<std::mutex> lock(m->mu);
  const auto ev = take_gemm_timing(m);
  if (slot < 0 || slot >= m->g.n_slots) return fail(ASAP_ERR_INVALID, "slot outside [0, n_slots)");
  if (epoch < 1) return fail(ASAP_ERR_INVALID, "epoch must be >= 1 (the value asap_moe_mailbox_post returned)");
  return serve_round(m, 1, &slot, &epoch, S(stream), ev.first, ev.second);
}

ASAP_API int asap_moe_mailbox_serve_many(asap_moe_mailbox_t m, int32_t count, const int32_t* slots,
                                         const uint64_t* epochs, void* stream) {
  if (!m) return fail(ASAP_ERR_INVALID, "NULL mailbox");
  std::lock_guard<std::mutex> lock(m->mu);
  const auto ev = take_gemm_timing(m);
  if (count < 1 || count > m->g.n_slots || !slots || !epochs)
    return fail(ASAP_ERR_INVALID, "count must be in [1, n_slots] with host arrays of count slots and epochs");
  uint64_t seen = 0;
  for (int i = 0; i < count; ++i) {
    const int32_t s = slots[i];
    if (s < 0 || s >= m->g.n_slots) return fail(ASAP_ERR_INVALID, "slot outside [0, n_slots)");
    if (seen & (1ull << s)) return fail(ASAP_ERR_INVALID, "a slot is listed twice");
    seen |= 1ull << s;
    if (epochs[i] < 1 || epochs[i] > m->posted[s])
      return fail(ASAP_ERR_INVALID, "slot " + std::to_string(s) + ": epoch " + std::to_string(epochs[i]) +
                                        " is not a post made to it");
  }
  return serve_round(m, count, slots, epochs, S(stream), ev.first, ev.second);
}

ASAP_API int asap_moe_mailbox_wait(asap_moe_mailbox_t m, int32_t slot, void* stream) {
  if (!m) return fail(ASAP_ERR_INVALID, "NULL mailbox");
  if (slot < 0 || slot >= m->g.n_slots) return fail(ASAP_ERR_INVALID, "slot outside [0, n_slots)");
  std::lock_guard<std::mutex> lock(m->mu);
  if (m->serve_called[slot] < m->posted[slot])
    return fail(ASAP_ERR_INVALID, "no serve call has been made for the slot's last post");
  CU_TRY(cudaStreamWaitEvent(S(stream), m->served_ev[slot], 0), "wait for the slot's round");
  return ASAP_OK;
}

ASAP_API int asap_moe_mailbox_served(asap_moe_mailbox_t m, int32_t slot, uint64_t* epoch) {
  if (!m || !epoch) return fail(ASAP_ERR_INVALID, "NULL mailbox or output");
  if (slot < 0 || slot >= m->g.n_slots) return fail(ASAP_ERR_INVALID, "slot outside [0, n_slots)");
  *epoch = *reinterpret_cast<volatile unsigned long long*>(m->served_host + slot);
  return ASAP_OK;
}

ASAP_API int asap_moe_mailbox_time_gemms(asap_moe_mailbox_t m, void* ev_before, void* ev_after) {
  if (!m) return fail(ASAP_ERR_INVALID, "NULL mailbox");
  std::lock_guard<std::mutex> lock(m->mu);
  m->gemm_ev0 = static_cast<cudaEvent_t>(ev_before);
  m->gemm_ev1 = static_cast<cudaEvent_t>(ev_after);
  return ASAP_OK;
}

ASAP_API int asap_moe_mailbox_rounds(asap_moe_mailbox_t m, int32_t* rounds, int32_t* claimed, int32_t cap) {
  if (!m || !rounds) return fail(ASAP_ERR_INVALID, "NULL mailbox or output");
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(m->h->device);
  cudaError_t e = cudaDeviceSynchronize();
  int32_t cnt = 0;
  if (e == cudaSuccess)
    e = cudaMemcpy(&cnt, &m->round->rounds, sizeof(int32_t), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && claimed && cap > 0)
    e = cudaMemcpy(claimed, m->log, sizeof(int32_t) * std::min(std::min(cap, cnt), asap::kMboxLog),
                   cudaMemcpyDeviceToHost);
  cudaSetDevice(prev);
  if (e != cudaSuccess) return cuda_fail(e, "mailbox rounds read");
  *rounds = cnt;
  return ASAP_OK;
}

// ============================================================ routing without allocation
//
// Some callers cannot allocate device memory when they route a micro-batch:
// a process whose HBM is owned entirely by another allocator (a serving
// framework's caching pool that reserved the device at start-up), or code on
// a path where a cudaMalloc would implicitly synchronise the device or is not
// permitted at all.  asap_moe_route_noalloc gives them the routing step with
// its scratch (router logits, per-chunk histograms, chunk bases) in a
// file-scope device array instead of a caller workspace.  The array holds
// kStaticRouteMaxTokens tokens x 256 experts of up to kMaxRouterSplits logit
// planes and is held by every GPU that loads this library until the process
// exits.

namespace {

constexpr int kStaticRouteMaxTokens = 4096;
// the router's K-slice planes: up to kMaxRouterSplits partial-logit planes of
// [n, E] fp32, as asap_moe_route keeps them in its workspace
constexpr size_t kStaticLogitsBytes = static_cast<size_t>(asap::kMaxRouterSplits) * kStaticRouteMaxTokens *
                                      ASAP_MOE_MAX_EXPERTS * sizeof(float);  // 16 MiB
constexpr size_t kStaticChunkBytes = static_cast<size_t>(kStaticRouteMaxTokens / asap::kChunkTokens) *
                                     ASAP_MOE_MAX_EXPERTS * sizeof(int32_t);                  // 128 KiB
constexpr size_t kStaticRouteBytes = kStaticLogitsBytes + 2 * kStaticChunkBytes + 256;  // + the scan's ticket

constexpr int kStaticMaxDevices = 64;
std::mutex g_static_route_mu;
void* g_static_route_ptr[kStaticMaxDevices] = {};

}  // namespace

// Host code must not use this symbol as a device address: it is a host-side
// stand-in.  The device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_static_route_scratch[kStaticRouteBytes];

namespace {

// Device address of the static scratch on ``device``, looked up once per
// device with that device current.
int static_route_scratch(int device, unsigned char** out) {
  if (device < 0 || device >= kStaticMaxDevices)
    return fail(ASAP_ERR_UNSUPPORTED, "device ordinal beyond the static routing scratch table");
  std::lock_guard<std::mutex> lock(g_static_route_mu);
  if (!g_static_route_ptr[device]) {
    int prev = 0;
    cudaError_t e = cudaGetDevice(&prev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (prev != device && (e = cudaSetDevice(device)) != cudaSuccess) return cuda_fail(e, "cudaSetDevice");
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_route_scratch);
    if (prev != device) cudaSetDevice(prev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the static routing scratch");
    g_static_route_ptr[device] = p;
  }
  *out = static_cast<unsigned char*>(g_static_route_ptr[device]);
  return ASAP_OK;
}

}  // namespace

ASAP_API int asap_moe_route_noalloc(asap_moe_t h, const void* x, int32_t n, int32_t* idx, float* w,
                                    int32_t* counts, int32_t* offsets, void* stream) {
  int r = check_call(h, n, nullptr, 0, false);
  if (r != ASAP_OK || n == 0) return r;
  if (n > kStaticRouteMaxTokens)
    return fail(ASAP_ERR_INVALID, "n = " + std::to_string(n) + " exceeds the " +
                                      std::to_string(kStaticRouteMaxTokens) +
                                      " tokens the static routing scratch holds; use asap_moe_route");
  if (!x || !idx || !w || !counts || !offsets || !aligned16(x)) return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  unsigned char* scratch = nullptr;
  if ((r = static_route_scratch(h->device, &scratch)) != ASAP_OK) return r;
  float* logits = reinterpret_cast<float*>(scratch);
  int32_t* hist = reinterpret_cast<int32_t*>(scratch + kStaticLogitsBytes);
  int32_t* base = reinterpret_cast<int32_t*>(scratch + kStaticLogitsBytes + kStaticChunkBytes);
  cudaStream_t st = S(stream);
  int32_t* ticket = reinterpret_cast<int32_t*>(scratch + kStaticLogitsBytes + 2 * kStaticChunkBytes);
  if (fused_route(h)) {
    // the same single launch as asap_moe_route (same K slices, same bits);
    // its ticket must start at zero, the rest is written before it is read
    CU_TRY(cudaMemsetAsync(ticket, 0, sizeof(int32_t), st), "ticket");
    return run_route_fused(h, x, n, idx, w, hist, 0, asap::ceil_div(n, asap::kChunkTokens), ticket, counts, offsets,
                           base, nullptr, h->layer_ids, st);
  }
  // the router's K slices and their order of addition are those of
  // asap_moe_route, so the bits are the same.  Every scratch element read
  // below is written earlier on the same stream (the logit planes by the
  // router, all E entries of each chunk's histogram and the scan's ticket by
  // the gate kernel), so nothing has to be cleared between calls.
  const int splits = router_splits(h, n);
  if ((r = run_router_logits(h, x, n, logits, splits, h->layer_ids, st)) != ASAP_OK) return r;
  CU_TRY(asap::launch_gate(logits, splits, n, gate_params(h, h->layer_ids, ticket), idx, w, hist, st),
         "gate launch");
  CU_TRY(asap::launch_scan(hist, asap::ceil_div(n, asap::kChunkTokens), h->cfg.n_experts, counts, offsets, base,
                           ticket, st),
         "scan launch");
  return ASAP_OK;
}
