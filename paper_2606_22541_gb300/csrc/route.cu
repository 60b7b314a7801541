// Routing kernels: router logits for expert counts below 256 (mma.sync, or
// CUDA cores for shapes it does not cover), top-k
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
// fixed reduction order (per-lane strided partial sums in increasing h, then
// a butterfly).  Each lane loads kRouterAhead of its 16-byte pieces of the
// token row before using them, so their HBM latencies overlap.
constexpr int kRouterEB = 16;    // experts per pass
constexpr int kRouterAhead = 8;  // row pieces in flight per lane

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
    for (int v0 = lane; v0 < V; v0 += 32 * kRouterAhead) {
      uint4 xv[kRouterAhead];
#pragma unroll
      for (int u = 0; u < kRouterAhead; ++u) {
        const int v = v0 + 32 * u;
        xv[u] = v < V ? __ldg(xr + v) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < kRouterAhead; ++u) {
        const int v = v0 + 32 * u;
        if (v < V) {
          const float xf[8] = {bf16_lo(xv[u].x), bf16_hi(xv[u].x), bf16_lo(xv[u].y), bf16_hi(xv[u].y),
                               bf16_lo(xv[u].z), bf16_hi(xv[u].z), bf16_lo(xv[u].w), bf16_hi(xv[u].w)};
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

// Router logits on the tensor core for 8, 16, 32 or 64 experts (mma.sync
// m16n8k16, bf16 in, fp32 accumulate; the partials of 64 experts fill 32 KB
// of shared memory, the static limit is 48 KB): the contraction
// has only E columns, too narrow for a 128 x 256 tcgen05 tile.  A CTA takes
// 16 tokens; its 8 warps split K, warp w taking the 32-wide K chunks w, w + 8,
// ...; the partial sums are added in warp order in shared memory.
//
// Fragments are loaded straight from global memory with a permutation of K
// that A and B share (the dot product does not depend on the order of K):
// thread (g = lane / 4, q = lane % 4) loads 16 bytes (8 bf16) of token rows g
// and g + 8 and of expert rows 8 j + g at K offset 8 q of the chunk, and feeds
// bf16 pairs 0, 1 to the chunk's first MMA and pairs 2, 3 to the second: in
// the first MMA, K slots 2q, 2q+1 are K offsets 8q, 8q+1 and slots 2q+8,
// 2q+9 are 8q+2, 8q+3, for A and for B alike.
constexpr int kRmmaWarps = 8;
constexpr int kRmmaTokens = 16;

__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <int NB>  // E = 8 NB experts
__global__ void __launch_bounds__(kRmmaWarps * 32) router_mma_kernel(const uint4* __restrict__ x, LayerRef lref,
                                                                     uint32_t* status, int n, int V,
                                                                     float* __restrict__ logits) {
  constexpr int E = 8 * NB;
  __shared__ float part[kRmmaWarps][kRmmaTokens][E];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, q = lane & 3;
  const int t0 = blockIdx.x * kRmmaTokens;
  const uint4* __restrict__ wr = static_cast<const uint4*>(
      lref.table[load_layer(lref.layer, lref.n_layers, status, blockIdx.x == 0 && threadIdx.x == 0)].router_w);
  // token rows g and g + 8 (rows past n read as zero and are not stored)
  const bool in0 = t0 + g < n, in1 = t0 + g + 8 < n;
  const uint4* x0 = x + static_cast<long long>(in0 ? t0 + g : 0) * V;
  const uint4* x1 = x + static_cast<long long>(in1 ? t0 + g + 8 : 0) * V;
  float c[NB][4];
#pragma unroll
  for (int j = 0; j < NB; ++j) c[j][0] = c[j][1] = c[j][2] = c[j][3] = 0.f;
  const uint4 zero = make_uint4(0, 0, 0, 0);
  // chunk ch covers 16-byte vectors 4 ch .. 4 ch + 3 of every row
  for (int ch = warp; ch < V / 4; ch += kRmmaWarps) {
    const int v = 4 * ch + q;
    const uint4 a = in0 ? __ldg(x0 + v) : zero;
    const uint4 b = in1 ? __ldg(x1 + v) : zero;
#pragma unroll
    for (int j = 0; j < NB; ++j) {
      const uint4 w = __ldg(wr + static_cast<long long>(8 * j + g) * V + v);
      mma_bf16_16816(c[j], a.x, b.x, a.y, b.y, w.x, w.y);
      mma_bf16_16816(c[j], a.z, b.z, a.w, b.w, w.z, w.w);
    }
  }
  // c[j]: (token g, experts 8j + 2q, 8j + 2q + 1) and (token g + 8, the same experts)
#pragma unroll
  for (int j = 0; j < NB; ++j) {
    part[warp][g][8 * j + 2 * q] = c[j][0];
    part[warp][g][8 * j + 2 * q + 1] = c[j][1];
    part[warp][g + 8][8 * j + 2 * q] = c[j][2];
    part[warp][g + 8][8 * j + 2 * q + 1] = c[j][3];
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kRmmaTokens * E; i += blockDim.x) {
    const int tl = i / E, e = i % E;
    if (t0 + tl >= n) continue;
    float sum = part[0][tl][e];
#pragma unroll
    for (int w = 1; w < kRmmaWarps; ++w) sum += part[w][tl][e];
    logits[static_cast<long long>(t0 + tl) * E + e] = sum;
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
// chunk-major: hist[chunk * E + e].
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

  if (p.ticket && blockIdx.x == 0 && threadIdx.x == 0) *p.ticket = 0;  // for the scan that follows
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
        const float s = gate_sigmoid(l);
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
      hist[static_cast<long long>(chunk0 + blockIdx.x) * E + e] = shist[e];
}

// ------------------------------------------------------------ gating, a team of lanes per token
// The same rules as gate_kernel for the common shapes (E = T S experts, T =
// min(32, E) lanes per token, S in {1, 2, 4, 8}; n_groups a power of two up
// to 32 for the grouped rule).  Lane q of a team holds experts [q S, (q+1) S)
// in registers (16-byte loads of the K-slice planes, added in slice order).
//  - Group scores: a group of gsz = E / G experts spans R = gsz / S lanes of
//    the team (G <= T), whose local top-2 keys merge over the R lanes.
//  - Groups are kept by rank: a group's rank is the number of groups with a
//    larger score, or an equal score and a lower index.
//  - Each of the k rounds takes every lane's best remaining eligible
//    expert, keeps the team's best (a butterfly, ties to the lower expert)
//    and marks it taken in its owner lane.
// Weights as in gate_kernel; the softmax sum adds each lane's slice in expert
// order, then the lanes in a butterfly.  Selection keys, group scores and the
// tie-breaks are those of gate_kernel, so both give the same experts.  One
// CTA per chunk of kChunkTokens tokens (32 T threads).

template <int T>
__device__ __forceinline__ void team_argmax(float& v, int& i, float& x) {
#pragma unroll
  for (int o = T / 2; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(kFull, v, o);
    const int oi = __shfl_xor_sync(kFull, i, o);
    const float ox = __shfl_xor_sync(kFull, x, o);
    if (ov > v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
      x = ox;
    }
  }
}

template <int T, int S>
__global__ void __launch_bounds__(kChunkTokens * T) gate_team_kernel(const float* __restrict__ logits, int splits,
                                                                 long long plane, int n, GateParams p,
                                                                 int32_t* __restrict__ idx,
                                                                 float* __restrict__ wout,
                                                                 int32_t* __restrict__ hist, int n_chunks,
                                                                 int chunk0) {
  static_assert(T * S <= kMaxExperts && (T == 8 || T == 16 || T == 32) && S <= 8, "team shape");
  __shared__ int shist[kMaxExperts];
  const int lane = threadIdx.x & 31;
  const int q = lane & (T - 1);  // lane in team
  const int E = T * S, k = p.top_k;
  for (int e = threadIdx.x; e < E; e += blockDim.x) shist[e] = 0;
  if (p.ticket && blockIdx.x == 0 && threadIdx.x == 0) *p.ticket = 0;  // for the scan that follows
  __syncthreads();
  const bool grouped = p.gating == 2;
  const float* __restrict__ bias =
      grouped ? p.lref.table[load_layer(p.lref.layer, p.lref.n_layers, p.status, threadIdx.x == 0 && blockIdx.x == 0)]
                    .router_bias
              : nullptr;
  const int t = blockIdx.x * kChunkTokens + threadIdx.x / T;
  const bool valid = t < n;
  const int e0 = q * S;
  float key[S], val[S];
  {
    const float* row = logits + static_cast<long long>(valid ? t : 0) * E + e0;
    float l[S];
    if constexpr (S % 4 == 0) {
#pragma unroll
      for (int v = 0; v < S / 4; ++v) {
        const float4 a = __ldg(reinterpret_cast<const float4*>(row) + v);
        l[4 * v] = a.x;
        l[4 * v + 1] = a.y;
        l[4 * v + 2] = a.z;
        l[4 * v + 3] = a.w;
      }
#pragma unroll 1
      for (int s2 = 1; s2 < splits; ++s2) {
#pragma unroll
        for (int v = 0; v < S / 4; ++v) {
          const float4 a = __ldg(reinterpret_cast<const float4*>(row + s2 * plane) + v);
          l[4 * v] += a.x;
          l[4 * v + 1] += a.y;
          l[4 * v + 2] += a.z;
          l[4 * v + 3] += a.w;
        }
      }
    } else {
#pragma unroll
      for (int j = 0; j < S; ++j) {
        float a = __ldg(row + j);
        for (int s2 = 1; s2 < splits; ++s2) a += __ldg(row + s2 * plane + j);
        l[j] = a;
      }
    }
#pragma unroll
    for (int j = 0; j < S; ++j) {
      if (!valid) l[j] = 0.f;
      if (grouped) {
        const float sg = gate_sigmoid(l[j]);
        val[j] = sg;
        key[j] = sg + (bias ? bias[e0 + j] : 0.0f);
      } else {
        val[j] = l[j];
        key[j] = l[j];
      }
    }
  }
  uint32_t eligible = (1u << S) - 1u;  // bit j: expert e0 + j may be chosen (S <= 8)
  if (grouped) {
    const int G = p.n_groups;  // <= T (checked at launch)
    uint32_t kept = 0;  // this lane's group is kept
    {
      const int R = (E / G) / S;  // lanes per group
      const int g = q / R;
      float m1 = -CUDART_INF_F, m2 = -CUDART_INF_F;
#pragma unroll
      for (int j = 0; j < S; ++j) {
        if (key[j] > m1) {
          m2 = m1;
          m1 = key[j];
        } else if (key[j] > m2) {
          m2 = key[j];
        }
      }
      for (int o = 1; o < R; o <<= 1) {
        const float a1 = __shfl_xor_sync(kFull, m1, o);
        const float a2 = __shfl_xor_sync(kFull, m2, o);
        const float hi = fmaxf(m1, a1);  // top two of {m1, m2, a1, a2}
        const float lo = fmaxf(fminf(m1, a1), fmaxf(m2, a2));
        m1 = hi;
        m2 = lo;
      }
      const float gs = m1 + m2;
      // rank of this lane's group among all G: groups with a larger score,
      // or an equal score and a lower index, come first (score of group gg
      // read from its first lane, gg R)
      int rank = 0;
#pragma unroll 1
      for (int gg = 0; gg < G; ++gg) {
        const float o = __shfl_sync(kFull, gs, (lane & ~(T - 1)) + gg * R);
        rank += (o > gs || (o == gs && gg < g)) ? 1 : 0;
      }
      kept = rank < p.topk_groups ? 1u : 0u;
      if (!kept) eligible = 0;
    }
  }
  // softmax: the sum of exp(l - max l) over all experts
  float z = 0.f, lmax = -CUDART_INF_F;
  if (p.gating == 0) {
#pragma unroll
    for (int j = 0; j < S; ++j) lmax = fmaxf(lmax, key[j]);
#pragma unroll
    for (int o = 1; o < T; o <<= 1) lmax = fmaxf(lmax, __shfl_xor_sync(kFull, lmax, o));
#pragma unroll
    for (int j = 0; j < S; ++j) z += expf(key[j] - lmax);
#pragma unroll
    for (int o = 1; o < T; o <<= 1) z += __shfl_xor_sync(kFull, z, o);
  }
  // k rounds: every lane offers its best remaining eligible expert (larger
  // key, then lower expert), the team keeps the best offer, and its owner
  // marks it taken
  int e_mine = 0x7fffffff;
  float x_mine = 0.f, sum = 0.f, m = 0.f, zsel = 0.f;
  uint32_t avail = eligible;
#pragma unroll 1
  for (int r = 0; r < k; ++r) {
    float v = -CUDART_INF_F, x = 0.f;
    int ei = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < S; ++j) {
      if (((avail >> j) & 1u) && (ei == 0x7fffffff || key[j] > v)) {
        v = key[j];
        x = val[j];
        ei = e0 + j;
      }
    }
    team_argmax<T>(v, ei, x);
    if (ei >= e0 && ei < e0 + S) avail &= ~(1u << (ei - e0));
    if (grouped) {
      sum += x;
      if (r == q) {
        e_mine = ei;
        x_mine = x;
      }
    } else {
      if (r == 0) m = v;  // the largest logit
      const float ex = expf(v - m);
      zsel += ex;
      if (r == q) {
        e_mine = ei;
        x_mine = ex;
      }
    }
  }
  float w_mine;
  if (grouped) {
    w_mine = x_mine / sum * p.route_scale;
  } else {
    w_mine = x_mine / (p.gating == 0 ? z : zsel);
  }
  if (valid && q < k) {
    idx[static_cast<long long>(t) * k + q] = e_mine;
    wout[static_cast<long long>(t) * k + q] = w_mine;
    if (e_mine >= 0 && e_mine < E) atomicAdd(&shist[e_mine], 1);
  }
  __syncthreads();
  if (hist)
    for (int e = threadIdx.x; e < E; e += blockDim.x)
      hist[static_cast<long long>(chunk0 + blockIdx.x) * E + e] = shist[e];
}

// ------------------------------------------------------------ histogram only
__global__ void __launch_bounds__(256) hist_kernel(const int32_t* __restrict__ idx, int n, int k, int E,
                                                   int32_t* __restrict__ hist, int n_chunks, uint32_t* status,
                                                   int32_t* ticket) {
  __shared__ int shist[kMaxExperts];
  if (blockIdx.x == 0 && threadIdx.x == 0) *ticket = 0;  // for the scan that follows
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
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[static_cast<long long>(blockIdx.x) * E + e] = shist[e];
}

// ------------------------------------------------------------ scan
// hist and chunk_base are chunk-major ([n_chunks][E]).  CTA g handles experts
// 32g .. 32g+31 (lane = expert) and its 8 warps consecutive ranges of chunks:
// each warp sums its range (128-byte rows), the warps' sums are combined in
// shared memory, then each warp writes chunk_base[c][e] = the entries of
// expert e in chunks before c (relative to the expert's offset, which
// dispatch adds) over its range.  The last CTA to finish (ticket counter,
// zero at launch, reset here) scans the counts into the exclusive offsets and
// clears the grouped GEMMs' tile counters.
constexpr int kScanThreads = 256;
constexpr int kScanWarps = kScanThreads / 32;

__device__ __forceinline__ int block_exclusive_scan(int v, int* swarp, int& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int u = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) swarp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    int w = lane < nw ? swarp[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(kFull, wi, o);
      if (lane >= o) wi += u;
    }
    if (lane < nw) swarp[lane] = wi - w;
    if (lane == nw - 1) swarp[32] = wi;
  }
  __syncthreads();
  total = swarp[32];
  const int r = swarp[warp] + incl - v;
  __syncthreads();  // swarp may be reused by the caller
  return r;
}

// MAPPED (a mailbox round): the rows scanned are rowmap[0 .. *n_chunks_dev)
// of hist, in that order (n_chunks is then rowmap's length), and chunk_base
// is written at the same rows.
template <bool MAPPED>
__global__ void __launch_bounds__(kScanThreads) scan_kernel(const int32_t* __restrict__ hist, int n_chunks, int E,
                                                            int32_t* __restrict__ counts,
                                                            int32_t* __restrict__ offsets,
                                                            int32_t* __restrict__ chunk_base,
                                                            int32_t* __restrict__ tile_counters,
                                                            int32_t* __restrict__ ticket,
                                                            const int32_t* __restrict__ rowmap,
                                                            const int32_t* __restrict__ n_chunks_dev) {
  __shared__ int part[kScanWarps][32];
  __shared__ int swarp[33];
  __shared__ bool last;
  if constexpr (MAPPED) n_chunks = max(0, min(*n_chunks_dev, n_chunks));  // n_chunks: rowmap's length
  auto row = [&](int c) -> long long { return MAPPED ? rowmap[c] : c; };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e = blockIdx.x * 32 + lane;
  const bool ve = e < E;
  const int per = (n_chunks + kScanWarps - 1) / kScanWarps;
  const int c0 = min(n_chunks, warp * per), c1 = min(n_chunks, c0 + per);
  int sum = 0;
  if (ve) {
#pragma unroll 8
    for (int c = c0; c < c1; ++c) sum += hist[row(c) * E + e];
  }
  part[warp][lane] = sum;
  __syncthreads();
  int run = 0, total = 0;
#pragma unroll
  for (int w = 0; w < kScanWarps; ++w) {
    const int v = part[w][lane];
    if (w < warp) run += v;
    total += v;
  }
  if (ve) {
#pragma unroll 8
    for (int c = c0; c < c1; ++c) {
      const long long o = row(c) * E + e;
      const int v = hist[o];
      chunk_base[o] = run;
      run += v;
    }
    if (warp == 0) counts[e] = total;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(ticket, 1) == static_cast<int>(gridDim.x) - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  int base = 0;
  for (int e0 = 0; e0 < E; e0 += kScanThreads) {
    const int ee = e0 + threadIdx.x;
    const int v = ee < E ? __ldcg(counts + ee) : 0;
    int tot = 0;
    const int ex = block_exclusive_scan(v, swarp, tot);
    if (ee < E) offsets[ee] = base + ex;
    base += tot;
  }
  if (threadIdx.x == 0) {
    offsets[E] = base;
    *ticket = 0;
  }
  // the grouped GEMMs that follow on this stream claim tiles from these
  if (tile_counters && threadIdx.x < kTileCounters) tile_counters[threadIdx.x] = 0;
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
  if (H % 32 == 0) {
    const int grid = ceil_div(n, kRmmaTokens);
    const uint4* xv = static_cast<const uint4*>(x);
#define ASAP_ROUTER_MMA(NBV)                                                                                  \
  if (E == 8 * NBV) {                                                                                         \
    router_mma_kernel<NBV><<<grid, kRmmaWarps * 32, 0, s>>>(xv, lref, status, n, H / 8, logits);              \
    return cudaGetLastError();                                                                                \
  }
    ASAP_ROUTER_MMA(1)
    ASAP_ROUTER_MMA(2)
    ASAP_ROUTER_MMA(4)
    ASAP_ROUTER_MMA(8)
#undef ASAP_ROUTER_MMA
  }
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
  const long long plane = static_cast<long long>(n) * p.n_experts;
  // a team of T = min(32, E) lanes per token when the shape allows it
  const int E = p.n_experts;
  const int T = E >= 32 ? 32 : E;
  const int S = E / T;
  const int G = p.gating == 2 ? p.n_groups : 1;
  // (16-byte vector loads of the logits rows need a 16-byte aligned base)
  const bool team = (T == 8 || T == 16 || T == 32) && E % T == 0 && (S == 1 || S == 2 || S == 4 || S == 8) &&
                    (G & (G - 1)) == 0 && G <= T && (S < 4 || (reinterpret_cast<uintptr_t>(logits) & 15u) == 0);
  if (team) {
#define ASAP_GATE_TEAM(TV, SV)                                                                                  \
  if (T == TV && S == SV) {                                                                                     \
    gate_team_kernel<TV, SV><<<chunks, kChunkTokens * TV, 0, s>>>(logits, splits, plane, n, p, idx, w, hist,    \
                                                                  n_chunks_total, chunk0);                      \
    return cudaGetLastError();                                                                                  \
  }
    ASAP_GATE_TEAM(32, 8)
    ASAP_GATE_TEAM(32, 4)
    ASAP_GATE_TEAM(32, 2)
    ASAP_GATE_TEAM(32, 1)
    ASAP_GATE_TEAM(16, 1)
    ASAP_GATE_TEAM(8, 1)
#undef ASAP_GATE_TEAM
  }
  gate_kernel<<<chunks, kGateWarps * 32, 0, s>>>(logits, splits, plane, n, p, idx, w, hist, n_chunks_total, chunk0);
  return cudaGetLastError();
}

cudaError_t launch_hist(const int32_t* idx, int n, int k, int E, int32_t* hist, uint32_t* status, int32_t* ticket,
                        cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int chunks = ceil_div(n, kChunkTokens);
  hist_kernel<<<chunks, 256, 0, s>>>(idx, n, k, E, hist, chunks, status, ticket);
  return cudaGetLastError();
}

cudaError_t launch_reduce_splits(const float* parts, int splits, long long plane, float* out, cudaStream_t s) {
  if (plane <= 0) return cudaSuccess;
  const int blocks = static_cast<int>(std::min<long long>((plane + 255) / 256, 4096));
  reduce_splits_kernel<<<blocks, 256, 0, s>>>(parts, splits, plane, out);
  return cudaGetLastError();
}

cudaError_t launch_scan(const int32_t* hist, int n_chunks, int E, int32_t* counts, int32_t* offsets,
                        int32_t* chunk_base, int32_t* ticket, cudaStream_t s, int32_t* tile_counters) {
  scan_kernel<false><<<ceil_div(E, 32), kScanThreads, 0, s>>>(hist, n_chunks, E, counts, offsets, chunk_base,
                                                             tile_counters, ticket, nullptr, nullptr);
  return cudaGetLastError();
}

cudaError_t launch_scan_mapped(const int32_t* hist, const int32_t* rowmap, const int32_t* n_chunks, int max_chunks,
                               int E, int32_t* counts, int32_t* offsets, int32_t* chunk_base, int32_t* ticket,
                               int32_t* tile_counters, cudaStream_t s) {
  scan_kernel<true><<<ceil_div(E, 32), kScanThreads, 0, s>>>(hist, max_chunks, E, counts, offsets, chunk_base,
                                                            tile_counters, ticket, rowmap, n_chunks);
  return cudaGetLastError();
}

}  // namespace asap
