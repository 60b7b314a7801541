// Routing kernels: router logits on CUDA cores (small expert counts), top-k
// gating with a fixed tie-break, per-chunk expert histograms and their
// deterministic prefix scan into per-expert counts and offsets.
//
// The MoE side of ASAP receives, for every micro-batch, the number of tokens
// per expert as its metadata (Section 3.2.1); here those counts and their
// exclusive prefix sums are produced on the device, from per-chunk histograms,
// so the position of every (token, slot) in its expert's segment is a pure
// function of the routing: increasing (t, j) inside each segment.
#include "common.cuh"
#include "internal.h"

#include <math_constants.h>

#include <algorithm>

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;

// ------------------------------------------------------------ router logits
// One warp per token; logits[t, e] = sum_h x[t, h] Wr[e, h] in fp32 with a
// fixed reduction order (per-lane strided partial sums, then a butterfly).
constexpr int kRouterEB = 16;  // experts per pass

__global__ void __launch_bounds__(256) router_small_kernel(const uint4* __restrict__ x, LayerRef lref,
                                                           uint32_t* status, int n, int V, int E,
                                                           float* __restrict__ logits) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * 8 + warp;
  if (t >= n) return;
  const uint4* __restrict__ wr = static_cast<const uint4*>(
      lref.table[load_layer(lref.layer, lref.n_layers, status, t == 0 && lane == 0)].router_w);
  const uint4* xr = x + static_cast<long long>(t) * V;
  for (int e0 = 0; e0 < E; e0 += kRouterEB) {
    float acc[kRouterEB];
#pragma unroll
    for (int i = 0; i < kRouterEB; ++i) acc[i] = 0.f;
    for (int v = lane; v < V; v += 32) {
      const uint4 xv = __ldg(xr + v);
      const float xf[8] = {bf16_lo(xv.x), bf16_hi(xv.x), bf16_lo(xv.y), bf16_hi(xv.y),
                           bf16_lo(xv.z), bf16_hi(xv.z), bf16_lo(xv.w), bf16_hi(xv.w)};
#pragma unroll
      for (int i = 0; i < kRouterEB; ++i) {
        if (e0 + i < E) {
          const uint4 wv = __ldg(wr + static_cast<long long>(e0 + i) * V + v);
          const float wf[8] = {bf16_lo(wv.x), bf16_hi(wv.x), bf16_lo(wv.y), bf16_hi(wv.y),
                               bf16_lo(wv.z), bf16_hi(wv.z), bf16_lo(wv.w), bf16_hi(wv.w)};
          float a = acc[i];
#pragma unroll
          for (int q = 0; q < 8; ++q) a = fmaf(xf[q], wf[q], a);
          acc[i] = a;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < kRouterEB; ++i) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc[i] += __shfl_xor_sync(kFull, acc[i], o);
    }
    float mine = 0.f;
#pragma unroll
    for (int i = 0; i < kRouterEB; ++i)
      if (lane == i) mine = acc[i];
    if (lane < kRouterEB && e0 + lane < E) logits[static_cast<long long>(t) * E + e0 + lane] = mine;
  }
}

// ------------------------------------------------------------ gating
// Warp-wide argmax over (key, expert) with the fixed order: larger key first,
// lower expert index on equal keys.  Every lane returns the same winner.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(kFull, v, o);
    const int oi = __shfl_xor_sync(kFull, i, o);
    if (ov > v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
}

constexpr int kGateWarps = kChunkTokens;  // one warp per token of the chunk

// One CTA per chunk of kChunkTokens tokens, one warp per token.  The logits
// arrive as ``splits`` partial planes (K slices of the router GEMM) that are
// added in slice order.  Lane l holds experts l, l+32, ..., so expert order
// and (i, lane) order agree.  The chunk's expert histogram is written
// transposed: hist[e * n_chunks + chunk].
__global__ void __launch_bounds__(kGateWarps * 32) gate_kernel(const float* __restrict__ logits, int splits,
                                                               long long plane, int n, GateParams p,
                                                               int32_t* __restrict__ idx,
                                                               float* __restrict__ wout,
                                                               int32_t* __restrict__ hist, int n_chunks,
                                                               int chunk0) {
  __shared__ int shist[kMaxExperts];
  __shared__ float ssel[kGateWarps][kMaxExperts];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = p.n_experts, k = p.top_k;
  for (int e = threadIdx.x; e < E; e += blockDim.x) shist[e] = 0;
  __syncthreads();

  const int t0 = blockIdx.x * kChunkTokens;
  const int t1 = min(n, t0 + kChunkTokens);
  const bool grouped = p.gating == 2;
  const int gsz = grouped ? E / p.n_groups : E;
  // selection bias of this launch's layer
  const float* __restrict__ bias =
      grouped ? p.lref.table[load_layer(p.lref.layer, p.lref.n_layers, p.status, threadIdx.x == 0 && blockIdx.x == 0)]
                    .router_bias
              : nullptr;

  for (int t = t0 + warp; t < t1; t += kGateWarps) {
    const float* lrow = logits + static_cast<long long>(t) * E;
    float key[8], sv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = lane + 32 * i;
      float l = -CUDART_INF_F;
      if (e < E) {
        l = lrow[e];
        for (int s2 = 1; s2 < splits; ++s2) l += lrow[s2 * plane + e];
      }
      if (grouped) {
        const float s = 1.0f / (1.0f + expf(-l));
        sv[i] = s;
        key[i] = e < E ? s + (bias ? bias[e] : 0.0f) : -CUDART_INF_F;
      } else {
        sv[i] = l;
        key[i] = l;
      }
    }
    uint32_t eligible = 0xffu;
    if (grouped) {
      // group score = sum of the two largest selection scores in the group
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = lane + 32 * i;
        if (e < E) ssel[warp][e] = key[i];
      }
      __syncwarp();
      float gscore = -CUDART_INF_F;
      if (lane < p.n_groups) {
        float m1 = -CUDART_INF_F, m2 = -CUDART_INF_F;
        for (int j = 0; j < gsz; ++j) {
          const float v = ssel[warp][lane * gsz + j];
          if (v > m1) {
            m2 = m1;
            m1 = v;
          } else if (v > m2) {
            m2 = v;
          }
        }
        gscore = m1 + m2;
      }
      __syncwarp();
      uint32_t kept = 0;
      for (int r = 0; r < p.topk_groups; ++r) {
        float v = (kept >> lane) & 1u ? -CUDART_INF_F : gscore;
        int gi = lane < p.n_groups && !((kept >> lane) & 1u) ? lane : 0x7fffffff;
        if (gi == 0x7fffffff) v = -CUDART_INF_F;
        warp_argmax(v, gi);
        if (gi < 32) kept |= 1u << gi;
      }
      eligible = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = lane + 32 * i;
        if (e < E && ((kept >> (e / gsz)) & 1u)) eligible |= 1u << i;
      }
    }

    int sel_e[kMaxTopK];
    float sel_v[kMaxTopK], sel_s[kMaxTopK];
    uint32_t taken = 0;
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) {
      sel_e[j] = 0x7fffffff;
      sel_v[j] = -CUDART_INF_F;
      sel_s[j] = 0.f;
      if (j < k) {
        float bv = -CUDART_INF_F;
        int bi = 0x7fffffff;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int e = lane + 32 * i;
          if (e < E && ((eligible >> i) & 1u) && !((taken >> i) & 1u) && (key[i] > bv || bi == 0x7fffffff)) {
            bv = key[i];
            bi = e;
          }
        }
        warp_argmax(bv, bi);
        float mine = 0.f;
        if (bi != 0x7fffffff && (bi & 31) == lane) {
          const int ii = bi >> 5;
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (i == ii) {
              mine = sv[i];
              taken |= 1u << i;
            }
        }
        sel_e[j] = bi;
        sel_v[j] = bv;
        sel_s[j] = __shfl_sync(kFull, mine, bi != 0x7fffffff ? (bi & 31) : 0);
      }
    }

    float wj[kMaxTopK];
    if (grouped) {
      float sum = 0.f;
#pragma unroll
      for (int j = 0; j < kMaxTopK; ++j)
        if (j < k) sum += sel_s[j];
#pragma unroll
      for (int j = 0; j < kMaxTopK; ++j) wj[j] = sel_s[j] / sum * p.route_scale;
    } else {
      const float m = sel_v[0];  // the first pick is the largest logit
      float z = 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int e = lane + 32 * i;
        if (e < E) z += expf(key[i] - m);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(kFull, z, o);
      float ex[kMaxTopK];
      float zsel = 0.f;
#pragma unroll
      for (int j = 0; j < kMaxTopK; ++j) {
        ex[j] = j < k ? expf(sel_v[j] - m) : 0.f;
        zsel += ex[j];
      }
      const float den = p.gating == 1 ? zsel : z;
#pragma unroll
      for (int j = 0; j < kMaxTopK; ++j) wj[j] = ex[j] / den;
    }

    int my_e = 0;
    float my_w = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j)
      if (lane == j) {
        my_e = sel_e[j];
        my_w = wj[j];
      }
    if (lane < k) {
      idx[static_cast<long long>(t) * k + lane] = my_e;
      wout[static_cast<long long>(t) * k + lane] = my_w;
      if (my_e >= 0 && my_e < E) atomicAdd(&shist[my_e], 1);
    }
  }
  __syncthreads();
  if (hist)
    for (int e = threadIdx.x; e < E; e += blockDim.x)
      hist[static_cast<long long>(e) * n_chunks + chunk0 + blockIdx.x] = shist[e];
}

// ------------------------------------------------------------ histogram only
__global__ void __launch_bounds__(256) hist_kernel(const int32_t* __restrict__ idx, int n, int k, int E,
                                                   int32_t* __restrict__ hist, int n_chunks, uint32_t* status) {
  __shared__ int shist[kMaxExperts];
  for (int e = threadIdx.x; e < E; e += blockDim.x) shist[e] = 0;
  __syncthreads();
  const int t0 = blockIdx.x * kChunkTokens;
  const int ne = (min(n, t0 + kChunkTokens) - t0) * k;
  for (int i = threadIdx.x; i < ne; i += blockDim.x) {
    const int e = idx[static_cast<long long>(t0) * k + i];
    if (e >= 0 && e < E) atomicAdd(&shist[e], 1);
    else record_status(status, ST_BAD_EXPERT_INDEX);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[static_cast<long long>(e) * n_chunks + blockIdx.x] = shist[e];
}

// ------------------------------------------------------------ scan
// One CTA.  hist and chunk_base are stored expert-major ([E][n_chunks]), so
// warp w scans experts w, w+32, ... over 32 consecutive chunks per coalesced
// load, giving each (expert, chunk) the number of earlier entries of that
// expert; then counts, the exclusive offsets, and the absolute chunk bases.
__global__ void __launch_bounds__(1024) scan_kernel(const int32_t* __restrict__ hist, int n_chunks, int E,
                                                    int32_t* __restrict__ counts,
                                                    int32_t* __restrict__ offsets,
                                                    int32_t* __restrict__ chunk_base,
                                                    int32_t* __restrict__ tile_counters) {
  __shared__ int scount[kMaxExperts];
  __shared__ int soff[kMaxExperts + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the grouped GEMMs that follow on this stream claim tiles from these
  if (tile_counters && threadIdx.x < kTileCounters) tile_counters[threadIdx.x] = 0;
  for (int e = warp; e < E; e += 32) {
    const int32_t* hrow = hist + static_cast<long long>(e) * n_chunks;
    int32_t* brow = chunk_base + static_cast<long long>(e) * n_chunks;
    int run = 0;
    for (int c0 = 0; c0 < n_chunks; c0 += 32) {
      const int c = c0 + lane;
      const int v = c < n_chunks ? hrow[c] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += u;
      }
      if (c < n_chunks) brow[c] = run + incl - v;
      run += __shfl_sync(kFull, incl, 31);
    }
    if (lane == 0) scount[e] = run;
  }
  __syncthreads();
  if (warp == 0) {
    int loc[8];
    int local = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = lane * 8 + i;
      loc[i] = e < E ? scount[e] : 0;
      local += loc[i];
    }
    int incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += u;
    }
    int run = incl - local;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = lane * 8 + i;
      if (e < E) soff[e] = run;
      run += loc[i];
    }
    if (lane == 31) soff[E] = incl;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    counts[e] = scount[e];
    offsets[e] = soff[e];
  }
  if (threadIdx.x == 0) offsets[E] = soff[E];
  for (int e = warp; e < E; e += 32) {
    int32_t* brow = chunk_base + static_cast<long long>(e) * n_chunks;
    const int base = soff[e];
    for (int c = lane; c < n_chunks; c += 32) brow[c] += base;
  }
}

// Sum of the K-slice planes of the router GEMM, added in slice order.
__global__ void reduce_splits_kernel(const float* __restrict__ parts, int splits, long long plane,
                                     float* __restrict__ out) {
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < plane;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    float v = parts[i];
    for (int s2 = 1; s2 < splits; ++s2) v += parts[s2 * plane + i];
    out[i] = v;
  }
}

}  // namespace

cudaError_t launch_router_small(const void* x, const LayerRef& lref, int n, int H, int E, float* logits,
                                uint32_t* status, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  router_small_kernel<<<ceil_div(n, 8), 256, 0, s>>>(static_cast<const uint4*>(x), lref, status, n, H / 8, E,
                                                       logits);
  return cudaGetLastError();
}

cudaError_t launch_gate(const float* logits, int splits, int n, const GateParams& p, int32_t* idx, float* w,
                        int32_t* hist, cudaStream_t s) {
  return launch_gate_seg(logits, splits, n, p, idx, w, hist, 0, ceil_div(n, kChunkTokens), s);
}

cudaError_t launch_gate_seg(const float* logits, int splits, int n, const GateParams& p, int32_t* idx, float* w,
                            int32_t* hist, int chunk0, int n_chunks_total, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int chunks = ceil_div(n, kChunkTokens);
  gate_kernel<<<chunks, kGateWarps * 32, 0, s>>>(logits, splits, static_cast<long long>(n) * p.n_experts, n, p,
                                                  idx, w, hist, n_chunks_total, chunk0);
  return cudaGetLastError();
}

cudaError_t launch_hist(const int32_t* idx, int n, int k, int E, int32_t* hist, uint32_t* status,
                        cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int chunks = ceil_div(n, kChunkTokens);
  hist_kernel<<<chunks, 256, 0, s>>>(idx, n, k, E, hist, chunks, status);
  return cudaGetLastError();
}

cudaError_t launch_reduce_splits(const float* parts, int splits, long long plane, float* out, cudaStream_t s) {
  if (plane <= 0) return cudaSuccess;
  const int blocks = static_cast<int>(std::min<long long>((plane + 255) / 256, 4096));
  reduce_splits_kernel<<<blocks, 256, 0, s>>>(parts, splits, plane, out);
  return cudaGetLastError();
}

cudaError_t launch_scan(const int32_t* hist, int n_chunks, int E, int32_t* counts, int32_t* offsets,
                        int32_t* chunk_base, cudaStream_t s, int32_t* tile_counters) {
  scan_kernel<<<1, 1024, 0, s>>>(hist, n_chunks, E, counts, offsets, chunk_base, tile_counters);
  return cudaGetLastError();
}

}  // namespace asap
