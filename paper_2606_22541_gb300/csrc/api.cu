// C ABI of libasap_moe: argument validation, workspace layout, weight packing
// at handle creation and the launch sequence of every call.  Every call other
// than create / destroy / status only enqueues kernels on the caller's stream.
#include "../../include/asap_moe.h"
#include "common.cuh"
#include "internal.h"

#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#define ASAP_API extern "C" __attribute__((visibility("default")))

struct asap_moe_s {
  asap_moe_config cfg;
  int device = 0;
  int num_sms = 0;
  void* router_w = nullptr;      // [E, H] bf16
  float* router_bias = nullptr;  // [E] fp32 or nullptr
  void* gate_up = nullptr;       // [E][2I, H] bf16, gate/up interleaved per 128 rows
  void* down = nullptr;          // [E][H, I] bf16
  void* sh_gate_up = nullptr;    // [2Is, H]
  void* sh_down = nullptr;       // [H, Is]
  uint32_t* status = nullptr;    // device status word
  bool tc_router = false;        // router GEMM on the tensor core (E == 256)
  CUtensorMap tm_router, tm_gate_up, tm_down, tm_sh_gate_up, tm_sh_down;
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

struct Layout {
  size_t logits, idx, w, hist, chunk_base, counts, offsets, perm_src, perm_dst, x_perm, h, h_sh, y_sh;
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
  const long long nk = n * c.top_k;
  const long long chunks = (n + asap::kChunkTokens - 1) / asap::kChunkTokens;
  L.logits = take(static_cast<size_t>(asap::kMaxRouterSplits) * n * c.n_experts * 4);  // K-slice planes
  L.idx = take(static_cast<size_t>(nk) * 4);
  L.w = take(static_cast<size_t>(nk) * 4);
  L.hist = take(static_cast<size_t>(chunks) * c.n_experts * 4);
  L.chunk_base = take(static_cast<size_t>(chunks) * c.n_experts * 4);
  L.counts = take(static_cast<size_t>(c.n_experts) * 4);
  L.offsets = take(static_cast<size_t>(c.n_experts + 1) * 4);
  L.perm_src = take(static_cast<size_t>(nk) * 4);
  L.perm_dst = take(static_cast<size_t>(nk) * 4);
  L.x_perm = take(static_cast<size_t>(nk) * c.hidden * 2);  // also holds y_perm in asap_moe_layer
  L.h = take(static_cast<size_t>(nk) * c.inter * 2);
  L.h_sh = take(c.n_shared ? static_cast<size_t>(n) * c.shared_inter * 2 : 0);
  L.y_sh = take(c.n_shared ? static_cast<size_t>(n) * c.hidden * 2 : 0);
  L.total = off;
  return L;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

cudaStream_t S(void* s) { return static_cast<cudaStream_t>(s); }

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
// at least 8 k-blocks per slice.
int router_splits(asap_moe_t h, int n) {
  if (!h->tc_router) return 1;
  const int mtiles = asap::ceil_div(n, asap::kGemmBM);
  const int kit = h->cfg.hidden / asap::kGemmBK;
  int s = h->num_sms / std::max(mtiles, 1);
  s = std::min(s, kit / 8);
  s = std::min(s, asap::kMaxRouterSplits);
  return std::max(s, 1);
}

// Router logits as ``splits`` planes of partial sums [splits][n][E] (planes
// are added in order by the consumer); splits == 1 writes the logits.
int run_router_logits(asap_moe_t h, const void* x, int n, float* logits, int splits, cudaStream_t st) {
  const asap_moe_config& c = h->cfg;
  if (h->tc_router) {
    CUtensorMap maps[4];
    std::string err;
    if (!asap::encode_tmap_bf16(&maps[0], x, n, c.hidden, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "x: " + err);
    maps[1] = h->tm_router;
    maps[2] = maps[0];
    maps[3] = maps[1];
    asap::GemmArgs a{};
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
    CU_TRY(asap::gemm_launch(asap::EPI_F32, maps, a, std::min(tiles, h->num_sms), st), "router GEMM launch");
  } else {
    CU_TRY(asap::launch_router_small(x, h->router_w, n, c.hidden, c.n_experts, logits, st), "router launch");
  }
  return ASAP_OK;
}

asap::GateParams gate_params(asap_moe_t h) {
  const asap_moe_config& c = h->cfg;
  asap::GateParams p{};
  p.n_experts = c.n_experts;
  p.top_k = c.top_k;
  p.gating = c.gating;
  p.n_groups = c.gating == ASAP_GATE_SIGMOID_GROUPED ? c.n_groups : 1;
  p.topk_groups = c.gating == ASAP_GATE_SIGMOID_GROUPED ? c.topk_groups : 1;
  p.route_scale = c.route_scale;
  p.bias = h->router_bias;
  return p;
}

int run_gate_scan(asap_moe_t h, const float* logits, int splits, int n, int32_t* idx, float* w, int32_t* counts,
                  int32_t* offsets, void* ws, cudaStream_t st) {
  const Layout L = layout(h->cfg, n);
  int32_t* hist = at<int32_t>(ws, L.hist);
  int32_t* base = at<int32_t>(ws, L.chunk_base);
  CU_TRY(asap::launch_gate(logits, splits, n, gate_params(h), idx, w, hist, st), "gate launch");
  CU_TRY(asap::launch_scan(hist, asap::ceil_div(n, asap::kChunkTokens), h->cfg.n_experts, counts, offsets, base,
                           st),
         "scan launch");
  return ASAP_OK;
}

int ub_mtiles(const asap_moe_config& c, long long nk) {
  return asap::ceil_div(nk, asap::kGemmBM) + static_cast<int>(std::min<long long>(c.n_experts, nk));
}

// GEMM1: h = silu(X Wg^T) * (X Wu^T) on the routed segments, plus the shared
// expert on x (problem 1 of the same launch).
int run_gate_up(asap_moe_t h, const void* x_perm, const int32_t* offsets, const void* x, int n, void* hbuf,
                void* hsh, cudaStream_t st) {
  const asap_moe_config& c = h->cfg;
  const long long nk = static_cast<long long>(n) * c.top_k;
  const bool sh = c.n_shared != 0;
  std::string err;
  CUtensorMap maps[4];
  if (!asap::encode_tmap_bf16(&maps[0], x_perm, nk, c.hidden, asap::kGemmBM, &err))
    return fail(ASAP_ERR_INVALID, "x_perm: " + err);
  maps[1] = h->tm_gate_up;
  if (sh) {
    if (!asap::encode_tmap_bf16(&maps[2], x, n, c.hidden, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "x: " + err);
    maps[3] = h->tm_sh_gate_up;
  } else {
    maps[2] = maps[0];
    maps[3] = maps[1];
  }
  asap::GemmArgs a{};
  a.offsets = offsets;
  a.groups = c.n_experts;
  a.m0 = static_cast<int>(nk);
  a.b_stride0 = 2 * c.inter;
  a.n_tiles0 = c.inter / 128;
  a.k_iters0 = c.hidden / asap::kGemmBK;
  a.out0 = hbuf;
  a.ldo0 = c.inter;
  a.m1 = sh ? n : 0;
  a.n_tiles1 = sh ? c.shared_inter / 128 : 0;
  a.k_iters1 = c.hidden / asap::kGemmBK;
  a.out1 = hsh;
  a.ldo1 = c.shared_inter;
  a.status = h->status;
  a.hint_a = 2;
  a.hint_b = 1;
  a.k_splits = 1;
  const long long tiles = static_cast<long long>(ub_mtiles(c, nk)) * a.n_tiles0 +
                          (sh ? static_cast<long long>(asap::ceil_div(n, asap::kGemmBM)) * a.n_tiles1 : 0);
  CU_TRY(asap::gemm_launch(asap::EPI_SWIGLU, maps, a, static_cast<int>(std::min<long long>(tiles, h->num_sms)), st),
         "gate/up GEMM launch");
  return ASAP_OK;
}

// GEMM2: y = h Wd^T on the routed segments, plus the shared expert.
int run_down(asap_moe_t h, const void* hbuf, const int32_t* offsets, const void* hsh, int n, void* y_perm,
             void* y_sh, cudaStream_t st) {
  const asap_moe_config& c = h->cfg;
  const long long nk = static_cast<long long>(n) * c.top_k;
  const bool sh = c.n_shared != 0;
  std::string err;
  CUtensorMap maps[4];
  if (!asap::encode_tmap_bf16(&maps[0], hbuf, nk, c.inter, asap::kGemmBM, &err))
    return fail(ASAP_ERR_INVALID, "h: " + err);
  maps[1] = h->tm_down;
  if (sh) {
    if (!asap::encode_tmap_bf16(&maps[2], hsh, n, c.shared_inter, asap::kGemmBM, &err))
      return fail(ASAP_ERR_INVALID, "h_shared: " + err);
    maps[3] = h->tm_sh_down;
  } else {
    maps[2] = maps[0];
    maps[3] = maps[1];
  }
  asap::GemmArgs a{};
  a.offsets = offsets;
  a.groups = c.n_experts;
  a.m0 = static_cast<int>(nk);
  a.b_stride0 = c.hidden;
  a.n_tiles0 = c.hidden / asap::kGemmBN;
  a.k_iters0 = c.inter / asap::kGemmBK;
  a.out0 = y_perm;
  a.ldo0 = c.hidden;
  a.m1 = sh ? n : 0;
  a.n_tiles1 = sh ? c.hidden / asap::kGemmBN : 0;
  a.k_iters1 = sh ? c.shared_inter / asap::kGemmBK : 0;
  a.out1 = y_sh;
  a.ldo1 = c.hidden;
  a.status = h->status;
  a.hint_a = 2;
  a.hint_b = 1;
  a.k_splits = 1;
  const long long tiles = static_cast<long long>(ub_mtiles(c, nk)) * a.n_tiles0 +
                          (sh ? static_cast<long long>(asap::ceil_div(n, asap::kGemmBM)) * a.n_tiles1 : 0);
  CU_TRY(asap::gemm_launch(asap::EPI_BF16, maps, a, static_cast<int>(std::min<long long>(tiles, h->num_sms)), st),
         "down GEMM launch");
  return ASAP_OK;
}

int run_expert_ffn(asap_moe_t h, const void* x_perm, const int32_t* offsets, const void* x, int n,
                   void* y_perm, void* y_sh, void* hbuf, void* hsh, cudaStream_t st) {
  int r = run_gate_up(h, x_perm, offsets, x, n, hbuf, hsh, st);
  if (r != ASAP_OK) return r;
  return run_down(h, hbuf, offsets, hsh, n, y_perm, y_sh, st);
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
  if (c->dtype == ASAP_FP8_E4M3_BLOCK128)
    return fail(ASAP_ERR_UNSUPPORTED, "the FP8 configuration is not built yet");
  if (c->dtype != ASAP_BF16) return fail(ASAP_ERR_INVALID, "unknown dtype");
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
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  cudaFree(h->router_w);
  cudaFree(h->router_bias);
  cudaFree(h->gate_up);
  cudaFree(h->down);
  cudaFree(h->sh_gate_up);
  cudaFree(h->sh_down);
  cudaFree(h->status);
  cudaSetDevice(prev);
  delete h;
  return ASAP_OK;
}

ASAP_API int asap_moe_create(const asap_moe_config* cfg, const asap_moe_weights* wts, asap_moe_t* out) {
  if (!out) return fail(ASAP_ERR_INVALID, "NULL out");
  *out = nullptr;
  int r = asap_moe_check_config(cfg);
  if (r != ASAP_OK) return r;
  if (!wts || !wts->router_w || !wts->w_gate || !wts->w_up || !wts->w_down)
    return fail(ASAP_ERR_INVALID, "router and expert weights are required");
  if (cfg->n_shared && (!wts->sh_gate || !wts->sh_up || !wts->sh_down))
    return fail(ASAP_ERR_INVALID, "shared-expert weights are required when n_shared == 1");
  const asap_moe_config& c = *cfg;
  asap_moe_s* h = new asap_moe_s();
  h->cfg = c;
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
  if (e != cudaSuccess) return bail(cuda_fail(e, "GEMM attributes"));
  e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking);
  if (e != cudaSuccess) return bail(cuda_fail(e, "stream"));

  const size_t H = c.hidden, E = c.n_experts, I = c.inter, Is = c.shared_inter;
  const size_t router_bytes = E * H * 2, gu_bytes = E * 2 * I * H * 2, down_bytes = E * H * I * 2;
  if ((e = cudaMalloc(&h->status, 256)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc status"));
  if ((e = cudaMemsetAsync(h->status, 0, 256, st)) != cudaSuccess) return bail(cuda_fail(e, "memset"));
  if ((e = cudaMalloc(&h->router_w, router_bytes)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc router"));
  if ((e = cudaMemcpyAsync(h->router_w, wts->router_w, router_bytes, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
    return bail(cuda_fail(e, "copy router"));
  if (wts->router_bias) {
    if ((e = cudaMalloc(&h->router_bias, E * 4)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc bias"));
    if ((e = cudaMemcpyAsync(h->router_bias, wts->router_bias, E * 4, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
      return bail(cuda_fail(e, "copy bias"));
  }
  if ((e = cudaMalloc(&h->gate_up, gu_bytes)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc gate/up"));
  if ((e = asap::launch_pack_gate_up(wts->w_gate, wts->w_up, static_cast<int>(E), static_cast<int>(I),
                                     static_cast<int>(H), h->gate_up, st)) != cudaSuccess)
    return bail(cuda_fail(e, "pack gate/up"));
  if ((e = cudaMalloc(&h->down, down_bytes)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc down"));
  if ((e = cudaMemcpyAsync(h->down, wts->w_down, down_bytes, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
    return bail(cuda_fail(e, "copy down"));
  if (c.n_shared) {
    if ((e = cudaMalloc(&h->sh_gate_up, 2 * Is * H * 2)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc shared"));
    if ((e = asap::launch_pack_gate_up(wts->sh_gate, wts->sh_up, 1, static_cast<int>(Is), static_cast<int>(H),
                                       h->sh_gate_up, st)) != cudaSuccess)
      return bail(cuda_fail(e, "pack shared"));
    if ((e = cudaMalloc(&h->sh_down, H * Is * 2)) != cudaSuccess) return bail(cuda_fail(e, "cudaMalloc shared down"));
    if ((e = cudaMemcpyAsync(h->sh_down, wts->sh_down, H * Is * 2, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
      return bail(cuda_fail(e, "copy shared down"));
  }
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return bail(cuda_fail(e, "create sync"));
  cudaStreamDestroy(st);
  st = nullptr;

  std::string err;
  h->tc_router = (c.n_experts == asap::kGemmBN);
  if (h->tc_router && !asap::encode_tmap_bf16(&h->tm_router, h->router_w, E, H, asap::kGemmBN, &err))
    return bail(fail(ASAP_ERR_CUDA, "router map: " + err));
  if (!asap::encode_tmap_bf16(&h->tm_gate_up, h->gate_up, E * 2 * I, H, asap::kGemmBN, &err))
    return bail(fail(ASAP_ERR_CUDA, "gate/up map: " + err));
  if (!asap::encode_tmap_bf16(&h->tm_down, h->down, E * H, I, asap::kGemmBN, &err))
    return bail(fail(ASAP_ERR_CUDA, "down map: " + err));
  if (c.n_shared) {
    if (!asap::encode_tmap_bf16(&h->tm_sh_gate_up, h->sh_gate_up, 2 * Is, H, asap::kGemmBN, &err))
      return bail(fail(ASAP_ERR_CUDA, "shared gate/up map: " + err));
    if (!asap::encode_tmap_bf16(&h->tm_sh_down, h->sh_down, H, Is, asap::kGemmBN, &err))
      return bail(fail(ASAP_ERR_CUDA, "shared down map: " + err));
  }
  *out = h;
  return ASAP_OK;
}

ASAP_API int asap_moe_router_logits(asap_moe_t h, const void* x, int32_t n, float* logits, void* ws,
                                    size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !logits || !aligned16(x) || !aligned16(logits))
    return fail(ASAP_ERR_INVALID, "x and logits must be non-NULL and 16-byte aligned");
  const int splits = router_splits(h, n);
  if (splits == 1) return run_router_logits(h, x, n, logits, 1, S(stream));
  // the same K slices and the same order of addition as asap_moe_route
  float* parts = at<float>(ws, layout(h->cfg, n).logits);
  if ((r = run_router_logits(h, x, n, parts, splits, S(stream))) != ASAP_OK) return r;
  CU_TRY(asap::launch_reduce_splits(parts, splits, static_cast<long long>(n) * h->cfg.n_experts, logits, S(stream)),
         "logit reduction launch");
  return ASAP_OK;
}

ASAP_API int asap_moe_route_logits(asap_moe_t h, const float* logits, int32_t n, int32_t* idx, float* w,
                                   int32_t* counts, int32_t* offsets, void* ws, size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!logits || !idx || !w || !counts || !offsets) return fail(ASAP_ERR_INVALID, "NULL tensor");
  return run_gate_scan(h, logits, 1, n, idx, w, counts, offsets, ws, S(stream));
}

ASAP_API int asap_moe_route(asap_moe_t h, const void* x, int32_t n, int32_t* idx, float* w, int32_t* counts,
                            int32_t* offsets, void* ws, size_t ws_bytes, void* stream) {
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !idx || !w || !counts || !offsets || !aligned16(x)) return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  float* logits = at<float>(ws, layout(h->cfg, n).logits);
  const int splits = router_splits(h, n);
  r = run_router_logits(h, x, n, logits, splits, S(stream));
  if (r != ASAP_OK) return r;
  return run_gate_scan(h, logits, splits, n, idx, w, counts, offsets, ws, S(stream));
}

ASAP_API int asap_moe_dispatch(asap_moe_t h, const void* x, int32_t n, const int32_t* idx, void* x_perm,
                               float* x_perm_scales, int32_t* perm_src, int32_t* perm_dst, void* ws,
                               size_t ws_bytes, void* stream) {
  (void)x_perm_scales;
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x || !idx || !x_perm || !perm_src || !perm_dst || !aligned16(x) || !aligned16(x_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  const asap_moe_config& c = h->cfg;
  const Layout L = layout(c, n);
  const int chunks = asap::ceil_div(n, asap::kChunkTokens);
  cudaStream_t st = S(stream);
  int32_t* hist = at<int32_t>(ws, L.hist);
  int32_t* base = at<int32_t>(ws, L.chunk_base);
  CU_TRY(asap::launch_hist(idx, n, c.top_k, c.n_experts, hist, h->status, st), "hist launch");
  CU_TRY(asap::launch_scan(hist, chunks, c.n_experts, at<int32_t>(ws, L.counts), at<int32_t>(ws, L.offsets), base, st),
         "scan launch");
  CU_TRY(asap::launch_dispatch(x, n, c.hidden, c.top_k, c.n_experts, idx, base, x_perm, perm_src, perm_dst, h->status,
                               st),
         "dispatch launch");
  return ASAP_OK;
}

ASAP_API int asap_moe_expert_ffn(asap_moe_t h, const void* x_perm, const float* x_perm_scales,
                                 const int32_t* offsets, const void* x, int32_t n, void* y_perm, void* y_shared,
                                 void* ws, size_t ws_bytes, void* stream) {
  (void)x_perm_scales;
  int r = check_call(h, n, ws, ws_bytes, true);
  if (r != ASAP_OK || n == 0) return r;
  if (!x_perm || !offsets || !y_perm || !aligned16(x_perm) || !aligned16(y_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->cfg.n_shared && (!x || !y_shared || !aligned16(x) || !aligned16(y_shared)))
    return fail(ASAP_ERR_INVALID, "x and y_shared are required for the shared expert");
  const Layout L = layout(h->cfg, n);
  return run_expert_ffn(h, x_perm, offsets, x, n, y_perm, y_shared, at<void>(ws, L.h), at<void>(ws, L.h_sh),
                        S(stream));
}

ASAP_API int asap_moe_expert_gate_up(asap_moe_t h, const void* x_perm, const float* x_perm_scales,
                                     const int32_t* offsets, const void* x, int32_t n, void* h_perm,
                                     void* h_shared, void* stream) {
  (void)x_perm_scales;
  int r = check_call(h, n, nullptr, 0, false);
  if (r != ASAP_OK || n == 0) return r;
  if (!x_perm || !offsets || !h_perm || !aligned16(x_perm) || !aligned16(h_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->cfg.n_shared && (!x || !h_shared || !aligned16(x) || !aligned16(h_shared)))
    return fail(ASAP_ERR_INVALID, "x and h_shared are required for the shared expert");
  return run_gate_up(h, x_perm, offsets, x, n, h_perm, h_shared, S(stream));
}

ASAP_API int asap_moe_expert_down(asap_moe_t h, const void* h_perm, const float* h_perm_scales,
                                  const int32_t* offsets, const void* h_shared, int32_t n, void* y_perm,
                                  void* y_shared, void* stream) {
  (void)h_perm_scales;
  int r = check_call(h, n, nullptr, 0, false);
  if (r != ASAP_OK || n == 0) return r;
  if (!h_perm || !offsets || !y_perm || !aligned16(h_perm) || !aligned16(y_perm))
    return fail(ASAP_ERR_INVALID, "NULL or unaligned tensor");
  if (h->cfg.n_shared && (!h_shared || !y_shared || !aligned16(h_shared) || !aligned16(y_shared)))
    return fail(ASAP_ERR_INVALID, "h_shared and y_shared are required for the shared expert");
  return run_down(h, h_perm, offsets, h_shared, n, y_perm, y_shared, S(stream));
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

ASAP_API int asap_moe_layer(asap_moe_t h, const void* x, int32_t n, void* out, void* ws, size_t ws_bytes,
                            void* stream) {
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
  void* x_perm = at<void>(ws, L.x_perm);
  void* y_sh = c.n_shared ? at<void>(ws, L.y_sh) : nullptr;
  const int splits = router_splits(h, n);
  if ((r = run_router_logits(h, x, n, logits, splits, st)) != ASAP_OK) return r;
  if ((r = run_gate_scan(h, logits, splits, n, idx, w, counts, offsets, ws, st)) != ASAP_OK) return r;
  CU_TRY(asap::launch_dispatch(x, n, c.hidden, c.top_k, c.n_experts, idx, at<int32_t>(ws, L.chunk_base), x_perm,
                               perm_src, perm_dst, h->status, st),
         "dispatch launch");
  // y_perm reuses x_perm's rows: the down GEMM never reads x_perm
  if ((r = run_expert_ffn(h, x_perm, offsets, x, n, x_perm, y_sh, at<void>(ws, L.h), at<void>(ws, L.h_sh), st)) !=
      ASAP_OK)
    return r;
  CU_TRY(asap::launch_combine(x_perm, y_sh, w, perm_dst, n, c.hidden, c.top_k, out, h->status, st),
         "combine launch");
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

// ============================================================ routing without allocation
//
// Some callers cannot allocate device memory when they route a micro-batch:
// a process whose HBM is owned entirely by another allocator (a serving
// framework's caching pool that reserved the device at start-up), or code on
// a path where a cudaMalloc would implicitly synchronise the device or is not
// permitted at all.  asap_moe_route_noalloc gives them the routing step with
// its scratch (router logits, per-chunk histograms, chunk bases) in a
// file-scope device array instead of a caller workspace.  The array is
// kStaticRouteMaxTokens tokens x 256 experts and is held by every GPU that
// loads this library until the process exits.

namespace {

constexpr int kStaticRouteMaxTokens = 4096;
constexpr size_t kStaticLogitsBytes =
    static_cast<size_t>(kStaticRouteMaxTokens) * ASAP_MOE_MAX_EXPERTS * sizeof(float);   // 4 MiB
constexpr size_t kStaticChunkBytes = static_cast<size_t>(kStaticRouteMaxTokens / asap::kChunkTokens) *
                                     ASAP_MOE_MAX_EXPERTS * sizeof(int32_t);                  // 128 KiB
constexpr size_t kStaticRouteBytes = kStaticLogitsBytes + 2 * kStaticChunkBytes;

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
  // every scratch element read below is written earlier on the same stream
  // (logits by the router, all E entries of each chunk's histogram by the
  // gate kernel), so nothing has to be cleared between calls
  if ((r = run_router_logits(h, x, n, logits, 1, st)) != ASAP_OK) return r;
  CU_TRY(asap::launch_gate(logits, 1, n, gate_params(h), idx, w, hist, st), "gate launch");
  CU_TRY(asap::launch_scan(hist, asap::ceil_div(n, asap::kChunkTokens), h->cfg.n_experts, counts, offsets, base, st),
         "scan launch");
  return ASAP_OK;
}
