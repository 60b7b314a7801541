// Data movement of the MoE layer: dispatch (token rows into per-expert
// segments), combine (weighted gather-reduce back to tokens) and the one-off
// gate/up weight packing done at handle creation.
//
// Dispatch is the single-GPU form of the token payload the MoE side receives
// grouped for its experts (ASAP Section 3.2.1); combine returns each expert's
// result to its token through the expert IDs (Section 3.2.2).  Both move rows
// as 16-byte vectors with every lane of a warp on consecutive vectors of the
// same row, so each warp-wide access is 512 contiguous bytes.
#include "common.cuh"
#include "internal.h"

#include <cuda_fp8.h>

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;
// The bf16 dispatch splits a chunk's row copies over two CTAs (every one
// ranks the chunk's entries, the first writes the permutation), so 4096
// tokens run 256 CTAs, more than the 152 SMs (measured on GB300: 112 -> 107
// us; four CTAs per chunk: 111 us); the FP8 dispatch, which also quantises,
// is faster with one CTA per chunk (85 us vs 100 us).
#ifndef ASAP_DISPATCH_PARTS
#define ASAP_DISPATCH_PARTS 2
#endif
template <bool FP8>
__host__ __device__ constexpr int dispatch_parts() { return FP8 ? 1 : ASAP_DISPATCH_PARTS; }
constexpr int kRankWarps = kChunkTokens * kMaxTopK / 32;  // warps that rank the chunk's entries
template <bool FP8>
__host__ __device__ constexpr int dispatch_warps() {
  return kChunkTokens / dispatch_parts<FP8>() > kRankWarps ? kChunkTokens / dispatch_parts<FP8>() : kRankWarps;
}

// One CTA per chunk of kChunkTokens tokens.  Entry i = t_local * k + j is
// ranked by thread i, so warp order and lane order follow (t, j); the rank of
// an entry inside its expert is (entries of that expert in earlier chunks)
// + (in earlier warps of this chunk) + (in earlier lanes of this warp):
// positions increase with (t, j) inside every segment.  chunk_base is
// chunk-major, relative to the expert's offset: the entries of expert e in
// chunks before ``chunk`` are offsets[e] + chunk_base[chunk * E + e].
// Then one warp per token
// reads its row once and writes it to its k positions.
// Quantise 8 consecutive values of a 128-channel block held by 16 lanes
// (lanes 0-15 one block, 16-31 the next): scale = amax / 448 over the block,
// q = e4m3(v / scale) with round-to-nearest-even and saturation; the
// quotient is taken as v * (1 / scale) in fp32, which can differ from the
// exact quotient by an ulp before the e4m3 rounding.
__device__ __forceinline__ uint2 quantize8(uint4 v, float& scale) {
  float f[8] = {bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y),
                bf16_lo(v.z), bf16_hi(v.z), bf16_lo(v.w), bf16_hi(v.w)};
  float am = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) am = fmaxf(am, fabsf(f[i]));
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
  scale = am > 0.f ? am / 448.0f : 1.0f;
  const float inv = 1.0f / scale;  // one division; the quotients below are products
  uint32_t w[2];
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const __nv_fp8x2_storage_t lo =
        __nv_cvt_float2_to_fp8x2(make_float2(f[4 * u] * inv, f[4 * u + 1] * inv), __NV_SATFINITE, __NV_E4M3);
    const __nv_fp8x2_storage_t hi =
        __nv_cvt_float2_to_fp8x2(make_float2(f[4 * u + 2] * inv, f[4 * u + 3] * inv), __NV_SATFINITE, __NV_E4M3);
    w[u] = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
  }
  return make_uint2(w[0], w[1]);
}

// Chunk c (part ``part`` of its row copies) of one micro-batch; the body of
// the dispatch kernels (one CTA per chunk and part).
template <bool FP8>
__device__ __forceinline__ void dispatch_chunk(int c, int part, const uint4* __restrict__ x, int n, int V, int k,
                                               int E, const int32_t* __restrict__ idx,
                                               const int32_t* __restrict__ chunk_base, void* __restrict__ x_perm_v,
                                               float* __restrict__ xs, uint2* __restrict__ xq_sh,
                                               float* __restrict__ xs_sh, int32_t* __restrict__ perm_src,
                                               int32_t* __restrict__ perm_dst, uint32_t* status,
                                               const DispatchSeg& seg) {
  __shared__ int wcnt[kRankWarps][kMaxExperts];
  __shared__ int spos[kChunkTokens * kMaxTopK];
  constexpr int kParts = dispatch_parts<FP8>();
  const int t0 = c * kChunkTokens;
  const int nt = min(kChunkTokens, n - t0);
  const int ne = nt * k;
  const long long nk = seg.rows_total;  // positions of every micro-batch of the call
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < kRankWarps * E; i += blockDim.x) wcnt[i / E][i % E] = 0;
  __syncthreads();

  const int i = threadIdx.x;
  int e = -1, rank = 0;
  if (warp < kRankWarps) {
    if (i < ne) {
      e = idx[static_cast<long long>(t0) * k + i];
      if (e < 0 || e >= E) {
        record_status(status, ST_BAD_EXPERT_INDEX);
        e = -1;
      }
    }
    const unsigned peers = __match_any_sync(kFull, e);
    rank = __popc(peers & ((1u << lane) - 1u));
    if (e >= 0 && lane == __ffs(peers) - 1) wcnt[warp][e] = __popc(peers);
  }
  __syncthreads();
  for (int ee = threadIdx.x; ee < E; ee += blockDim.x) {
    int run = seg.expert_offsets[ee] + chunk_base[static_cast<long long>(seg.chunk0 + c) * E + ee];
#pragma unroll
    for (int w = 0; w < kRankWarps; ++w) {
      const int v = wcnt[w][ee];
      wcnt[w][ee] = run;
      run += v;
    }
  }
  __syncthreads();
  if (i < ne) {
    int pos = -1;
    if (e >= 0) {
      pos = wcnt[warp][e] + rank;
      if (pos < 0 || pos >= nk) {
        record_status(status, ST_BAD_POSITION);
        pos = -1;
      }
    }
    spos[i] = pos;
    if (part == 0) {
      perm_dst[static_cast<long long>(t0) * k + i] = pos;
      if (pos >= 0) perm_src[pos] = seg.tok0 + t0 + i / k;
    }
  }
  __syncthreads();
  // row copies: one warp per token of this CTA's part, read once, write k times
  const int tl = part * (kChunkTokens / kParts) + warp;  // token of the chunk
  if (warp < kChunkTokens / kParts && tl < nt) {
    const uint4* src = x + static_cast<long long>(t0 + tl) * V;
    int p[kMaxTopK];
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) p[j] = j < k ? spos[tl * k + j] : -1;
    if constexpr (!FP8) {
      uint4* x_perm = static_cast<uint4*>(x_perm_v);
      // optional copy of the row for the shared expert (calls that serve
      // several micro-batches gather their tokens into one matrix)
      uint4* sh = seg.x_sh ? static_cast<uint4*>(seg.x_sh) + static_cast<long long>(t0 + tl) * V : nullptr;
      int v = lane;
      for (; v + 32 < V; v += 64) {
        const uint4 a = __ldg(src + v);
        const uint4 b = __ldg(src + v + 32);
#pragma unroll
        for (int j = 0; j < kMaxTopK; ++j)
          if (p[j] >= 0) {
            uint4* d = x_perm + static_cast<long long>(p[j]) * V;
            d[v] = a;
            d[v + 32] = b;
          }
        if (sh) {
          sh[v] = a;
          sh[v + 32] = b;
        }
      }
      for (; v < V; v += 32) {
        const uint4 a = __ldg(src + v);
#pragma unroll
        for (int j = 0; j < kMaxTopK; ++j)
          if (p[j] >= 0) x_perm[static_cast<long long>(p[j]) * V + v] = a;
        if (sh) sh[v] = a;
      }
    } else {
      // e4m3 rows: V vectors of 8 values -> V 8-byte words; one scale per 16
      // vectors (128 channels); a warp covers two blocks per step
      uint2* xq = static_cast<uint2*>(x_perm_v);
      const int nb = V / 16;
      const long long t = t0 + tl;
      for (int v = lane; v < V; v += 32) {
        float scale;
        const uint2 q = quantize8(__ldg(src + v), scale);
        const int blk = v >> 4;
        const bool head = (lane & 15) == 0;
#pragma unroll
        for (int j = 0; j < kMaxTopK; ++j)
          if (p[j] >= 0) {
            xq[static_cast<long long>(p[j]) * V + v] = q;
            if (head) xs[static_cast<long long>(p[j]) * nb + blk] = scale;
          }
        if (xq_sh) {
          xq_sh[t * V + v] = q;
          if (head) xs_sh[t * nb + blk] = scale;
        }
      }
    }
  }
}

template <bool FP8>
__global__ void __launch_bounds__(dispatch_warps<FP8>() * 32)
    dispatch_kernel(const uint4* __restrict__ x, int n, int V, int k, int E,
                    const int32_t* __restrict__ idx, const int32_t* __restrict__ chunk_base, int n_chunks,
                    void* __restrict__ x_perm_v, float* __restrict__ xs, uint2* __restrict__ xq_sh,
                    float* __restrict__ xs_sh, int32_t* __restrict__ perm_src,
                    int32_t* __restrict__ perm_dst, uint32_t* status, const DispatchSeg seg) {
  constexpr int kParts = dispatch_parts<FP8>();
  dispatch_chunk<FP8>(blockIdx.x / kParts, blockIdx.x % kParts, x, n, V, k, E, idx, chunk_base, x_perm_v, xs, xq_sh,
                      xs_sh, perm_src, perm_dst, status, seg);
}

// One work item of a mailbox round's dispatch: part ``part`` of the round's
// chunk vc (see dispatch_mbox_kernel).
template <bool FP8>
__device__ __forceinline__ void dispatch_mbox_item(int vc, int part, const MboxRound* __restrict__ r,
                                                   const MboxGeom& g, const int32_t* __restrict__ rowmap,
                                                   const int32_t* __restrict__ idx,
                                                   const int32_t* __restrict__ chunk_base,
                                                   const int32_t* __restrict__ offsets, void* __restrict__ x_perm_v,
                                                   float* __restrict__ xs, void* __restrict__ x_sh,
                                                   float* __restrict__ xs_sh, int32_t* __restrict__ perm_src,
                                                   int32_t* __restrict__ perm_dst, uint32_t* status) {
  const int row = rowmap[vc];
  const int slot = row / g.slot_chunks;
  const int c = row - slot * g.slot_chunks;
  const int i = r->index_of[slot];
  const int n = r->n[i];
  const long long tok0 = r->tok0[i];
  const int V = g.H / 8;
  DispatchSeg seg{};
  seg.expert_offsets = offsets;
  seg.chunk0 = slot * g.slot_chunks;
  seg.n_chunks_total = g.n_slots * g.slot_chunks;
  seg.tok0 = static_cast<int>(tok0);
  seg.rows_total = static_cast<long long>(r->n_total) * g.k;
  uint2* xq_sh = nullptr;
  float* xs_sh_i = nullptr;
  if constexpr (FP8) {
    if (x_sh) {
      xq_sh = static_cast<uint2*>(x_sh) + tok0 * V;
      xs_sh_i = xs_sh + tok0 * (V / 16);
    }
  } else {
    seg.x_sh = x_sh ? static_cast<void*>(static_cast<uint4*>(x_sh) + tok0 * V) : nullptr;
  }
  const long long sidx = static_cast<long long>(slot) * g.slot_tokens * g.k;
  dispatch_chunk<FP8>(c, part, static_cast<const uint4*>(r->x[i]), n, V, g.k, g.E, idx + sidx, chunk_base, x_perm_v,
                      xs, xq_sh, xs_sh_i, perm_src, perm_dst + sidx, status, seg);
}

// Dispatch of a mailbox round: work item q is part q % kParts of the
// round's chunk q / kParts in the scan's order (the row map lists the claimed
// posts' histogram rows, post after post); CTA b takes items b, b + gridDim.x,
// ...  The chunk's post comes at r->tok0[i] in the combined token order, its
// histogram row and chunk bases are its slot's, its idx / perm_dst entries
// its slot's region.
template <bool FP8>
__global__ void __launch_bounds__(dispatch_warps<FP8>() * 32)
    dispatch_mbox_kernel(const MboxRound* __restrict__ r, const MboxGeom g, const int32_t* __restrict__ rowmap,
                         const int32_t* __restrict__ idx, const int32_t* __restrict__ chunk_base,
                         const int32_t* __restrict__ offsets, void* __restrict__ x_perm_v, float* __restrict__ xs,
                         void* __restrict__ x_sh, float* __restrict__ xs_sh, int32_t* __restrict__ perm_src,
                         int32_t* __restrict__ perm_dst, uint32_t* status) {
  constexpr int kParts = dispatch_parts<FP8>();
  const int items = r->chunks_total * kParts;
  for (int q = blockIdx.x; q < items; q += gridDim.x) {
    dispatch_mbox_item<FP8>(q / kParts, q % kParts, r, g, rowmap, idx, chunk_base, offsets, x_perm_v, xs, x_sh,
                            xs_sh, perm_src, perm_dst, status);
    __syncthreads();  // the chunk's shared rank tables are rewritten by the next item
  }
}

// Rows of bf16 to e4m3 with a scale per 128 channels; one warp per row.
__global__ void __launch_bounds__(256) quantize_rows_kernel(const uint4* __restrict__ x, int rows, int V,
                                                            uint2* __restrict__ q, float* __restrict__ s) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long r = static_cast<long long>(blockIdx.x) * 8 + warp;
  if (r >= rows) return;
  const int nb = V / 16;
  for (int v = lane; v < V; v += 32) {
    float scale;
    const uint2 w = quantize8(__ldg(x + r * V + v), scale);
    q[r * V + v] = w;
    if ((lane & 15) == 0) s[r * nb + (v >> 4)] = scale;
  }
}

constexpr int kCombineWarps = 8;

// One warp per token: out[t] = sum_j w[t,j] y_perm[perm_dst[t,j]] (+ y_sh[t]),
// fp32 fused multiply-adds in slot order, then the shared row, then bf16.
// The body for one token: w_t, pd_t its k weights and positions, y_sh_t its
// shared-expert row (nullable), out_t its output row.
__device__ __forceinline__ void combine_token(const uint4* __restrict__ y_perm, const uint4* __restrict__ y_sh_t,
                                              const float* __restrict__ w_t, const int32_t* __restrict__ pd_t, int V,
                                              int k, uint4* __restrict__ out_t, uint32_t* status, long long nk,
                                              int lane) {
  int p[kMaxTopK];
  float wj[kMaxTopK];
#pragma unroll
  for (int j = 0; j < kMaxTopK; ++j) {
    p[j] = -1;
    wj[j] = 0.f;
    if (j < k) {
      p[j] = pd_t[j];
      wj[j] = w_t[j];
      if (p[j] < 0 || p[j] >= nk) {
        if (lane == 0) record_status(status, ST_BAD_POSITION);
        p[j] = -1;
      }
    }
  }
#pragma unroll 2
  for (int v = lane; v < V; v += 32) {
    uint4 yv[kMaxTopK];
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j)
      if (p[j] >= 0) yv[j] = __ldg(y_perm + static_cast<long long>(p[j]) * V + v);
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) {
      if (p[j] >= 0) {
        const float a = wj[j];
        acc[0] = fmaf(a, bf16_lo(yv[j].x), acc[0]);
        acc[1] = fmaf(a, bf16_hi(yv[j].x), acc[1]);
        acc[2] = fmaf(a, bf16_lo(yv[j].y), acc[2]);
        acc[3] = fmaf(a, bf16_hi(yv[j].y), acc[3]);
        acc[4] = fmaf(a, bf16_lo(yv[j].z), acc[4]);
        acc[5] = fmaf(a, bf16_hi(yv[j].z), acc[5]);
        acc[6] = fmaf(a, bf16_lo(yv[j].w), acc[6]);
        acc[7] = fmaf(a, bf16_hi(yv[j].w), acc[7]);
      }
    }
    if (y_sh_t) {
      const uint4 s = __ldg(y_sh_t + v);
      acc[0] += bf16_lo(s.x);
      acc[1] += bf16_hi(s.x);
      acc[2] += bf16_lo(s.y);
      acc[3] += bf16_hi(s.y);
      acc[4] += bf16_lo(s.z);
      acc[5] += bf16_hi(s.z);
      acc[6] += bf16_lo(s.w);
      acc[7] += bf16_hi(s.w);
    }
    out_t[v] = make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                          pack_bf16x2(acc[6], acc[7]));
  }
}

__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_kernel(const uint4* __restrict__ y_perm, const uint4* __restrict__ y_sh,
                   const float* __restrict__ w, const int32_t* __restrict__ perm_dst, int n, int V,
                   int k, uint4* __restrict__ out, uint32_t* status, long long nk) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kCombineWarps + warp;
  if (t >= n) return;
  const long long tk = static_cast<long long>(t) * k, tv = static_cast<long long>(t) * V;
  combine_token(y_perm, y_sh ? y_sh + tv : nullptr, w + tk, perm_dst + tk, V, k, out + tv, status, nk, lane);
}

// Combine of a mailbox round: warp w of CTA b combines the tokens
// (b + j gridDim.x) * kCombineWarps + w of the round's combined token order
// (the claimed posts one after the other).  A token's post i (the last with
// r->tok0[i] <= it) writes into its own output; its weights and positions are
// in its slot's region, its shared-expert row at its place in the combined
// order.
__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_mbox_kernel(const MboxRound* __restrict__ r, const MboxGeom g, const uint4* __restrict__ y_perm,
                        const uint4* __restrict__ y_sh, const float* __restrict__ w,
                        const int32_t* __restrict__ perm_dst, uint32_t* status) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_total = r->n_total, count = r->count;
  const int V = g.H / 8;
  const long long nk = static_cast<long long>(n_total) * g.k;
  for (int tg = blockIdx.x * kCombineWarps + warp; tg < n_total; tg += gridDim.x * kCombineWarps) {
    int lo = 0, hi = count;  // the last claimed post starting at or before tg
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (r->tok0[mid] <= tg) lo = mid; else hi = mid;
    }
    const int i = lo;
    const int t = tg - r->tok0[i];
    if (t >= r->n[i]) continue;
    const long long tk = (static_cast<long long>(r->slot[i]) * g.slot_tokens + t) * g.k;
    combine_token(y_perm, y_sh ? y_sh + (static_cast<long long>(r->tok0[i]) + t) * V : nullptr, w + tk,
                  perm_dst + tk, V, g.k, static_cast<uint4*>(r->out[i]) + static_cast<long long>(t) * V, status, nk,
                  lane);
  }
}

// packed[e][b*256 + r] = gate[e][b*128 + r] for r < 128, up[e][b*128 + r - 128]
// otherwise, so one 256-row weight tile holds 128 gate rows and the matching
// 128 up rows.
// Tile-contiguous weights: 128-byte row pieces grouped per GEMM box.
// dst box (e, nt, kb) = 256 consecutive rows of 128 B: rows nt*256 .. of
// expert e's packed matrix, bytes [kb*128, kb*128 + 128) of each row; one box
// is one contiguous 32 KB read from HBM.  gate_up: packed row r of tile nt is
// gate row nt*128 + r (r < 128) or up row nt*128 + r - 128; else row nt*256 + r
// of a.  R: packed rows per expert; V: 16-byte units per row.
__global__ void retile_kernel(const uint4* __restrict__ a, const uint4* __restrict__ b, int E, int R, int V,
                              bool gate_up, uint4* __restrict__ dst) {
  const int KB = V / 8, NT = R / 256;
  const long long total = static_cast<long long>(E) * R * V;
  for (long long q = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; q < total;
       q += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int v8 = static_cast<int>(q & 7);
    long long t = q >> 3;
    const int r = static_cast<int>(t & 255);
    t >>= 8;
    const int kb = static_cast<int>(t % KB);
    t /= KB;
    const int nt = static_cast<int>(t % NT);
    const long long e = t / NT;
    const uint4* src;
    if (gate_up)
      src = (r < 128 ? a : b) + (e * (R / 2) + nt * 128 + (r & 127)) * V;
    else
      src = a + (e * R + nt * 256 + r) * V;
    dst[q] = src[kb * 8 + v8];
  }
}

}  // namespace

cudaError_t launch_dispatch(const void* x, int n, int H, int k, int E, const int32_t* idx,
                            const int32_t* chunk_base, const int32_t* offsets, void* x_perm, int32_t* perm_src,
                            int32_t* perm_dst, uint32_t* status, cudaStream_t s) {
  DispatchSeg seg{};
  seg.expert_offsets = offsets;
  seg.n_chunks_total = ceil_div(n, kChunkTokens);
  seg.rows_total = static_cast<long long>(n) * k;
  return launch_dispatch_seg(x, n, H, k, E, idx, chunk_base, x_perm, perm_src, perm_dst, status, seg, s);
}

cudaError_t launch_dispatch_seg(const void* x, int n, int H, int k, int E, const int32_t* idx,
                                const int32_t* chunk_base, void* x_perm, int32_t* perm_src, int32_t* perm_dst,
                                uint32_t* status, const DispatchSeg& seg, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int chunks = ceil_div(n, kChunkTokens);
  dispatch_kernel<false><<<chunks * dispatch_parts<false>(), dispatch_warps<false>() * 32, 0, s>>>(static_cast<const uint4*>(x), n, H / 8, k, E, idx,
                                                                chunk_base, seg.n_chunks_total, x_perm, nullptr,
                                                                nullptr, nullptr, perm_src, perm_dst, status, seg);
  return cudaGetLastError();
}

cudaError_t launch_dispatch_fp8(const void* x, int n, int H, int k, int E, const int32_t* idx,
                                const int32_t* chunk_base, const int32_t* offsets, void* xq, float* xs,
                                void* xq_sh, float* xs_sh, int32_t* perm_src, int32_t* perm_dst, uint32_t* status,
                                cudaStream_t s) {
  DispatchSeg seg{};
  seg.expert_offsets = offsets;
  seg.n_chunks_total = ceil_div(n, kChunkTokens);
  seg.rows_total = static_cast<long long>(n) * k;
  return launch_dispatch_fp8_seg(x, n, H, k, E, idx, chunk_base, xq, xs, xq_sh, xs_sh, perm_src, perm_dst, status,
                                 seg, s);
}

cudaError_t launch_dispatch_fp8_seg(const void* x, int n, int H, int k, int E, const int32_t* idx,
                                    const int32_t* chunk_base, void* xq, float* xs, void* xq_sh, float* xs_sh,
                                    int32_t* perm_src, int32_t* perm_dst, uint32_t* status, const DispatchSeg& seg,
                                    cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int chunks = ceil_div(n, kChunkTokens);
  dispatch_kernel<true><<<chunks * dispatch_parts<true>(), dispatch_warps<true>() * 32, 0, s>>>(static_cast<const uint4*>(x), n, H / 8, k, E, idx,
                                                               chunk_base, seg.n_chunks_total, xq, xs,
                                                               static_cast<uint2*>(xq_sh), xs_sh, perm_src, perm_dst,
                                                               status, seg);
  return cudaGetLastError();
}

cudaError_t launch_quantize_rows(const void* x, int rows, int cols, void* q, float* s, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  quantize_rows_kernel<<<ceil_div(rows, 8), 256, 0, st>>>(static_cast<const uint4*>(x), rows, cols / 8,
                                                          static_cast<uint2*>(q), s);
  return cudaGetLastError();
}

cudaError_t launch_combine(const void* y_perm, const void* y_shared, const float* w,
                           const int32_t* perm_dst, int n, int H, int k, void* out, uint32_t* status,
                           cudaStream_t s, long long rows_total) {
  if (n <= 0) return cudaSuccess;
  combine_kernel<<<ceil_div(n, kCombineWarps), kCombineWarps * 32, 0, s>>>(
      static_cast<const uint4*>(y_perm), static_cast<const uint4*>(y_shared), w, perm_dst, n, H / 8, k,
      static_cast<uint4*>(out), status, rows_total > 0 ? rows_total : static_cast<long long>(n) * k);
  return cudaGetLastError();
}

cudaError_t launch_dispatch_mbox(const MboxRound* r, MboxGeom g, const int32_t* rowmap, const int32_t* idx,
                                 const int32_t* chunk_base, const int32_t* offsets, void* x_perm, int32_t* perm_src,
                                 int32_t* perm_dst, void* x_sh, uint32_t* status, cudaStream_t s) {
  const int grid = g.slot_chunks * dispatch_parts<false>();  // one post's work items; more loop
  dispatch_mbox_kernel<false><<<grid, dispatch_warps<false>() * 32, 0, s>>>(r, g, rowmap, idx, chunk_base, offsets,
                                                                            x_perm, nullptr, x_sh, nullptr, perm_src,
                                                                            perm_dst, status);
  return cudaGetLastError();
}

cudaError_t launch_dispatch_fp8_mbox(const MboxRound* r, MboxGeom g, const int32_t* rowmap, const int32_t* idx,
                                     const int32_t* chunk_base, const int32_t* offsets, void* xq, float* xs,
                                     void* xq_sh, float* xs_sh, int32_t* perm_src, int32_t* perm_dst,
                                     uint32_t* status, cudaStream_t s) {
  const int grid = g.slot_chunks * dispatch_parts<true>();  // one post's work items; more loop
  dispatch_mbox_kernel<true><<<grid, dispatch_warps<true>() * 32, 0, s>>>(r, g, rowmap, idx, chunk_base, offsets, xq,
                                                                          xs, xq_sh, xs_sh, perm_src, perm_dst,
                                                                          status);
  return cudaGetLastError();
}

cudaError_t launch_combine_mbox(const MboxRound* r, MboxGeom g, const void* y_perm, const void* y_shared,
                                const float* w, const int32_t* perm_dst, uint32_t* status, cudaStream_t s) {
  const int grid = ceil_div(g.slot_tokens, kCombineWarps);  // one post's tokens; more loop
  combine_mbox_kernel<<<grid, kCombineWarps * 32, 0, s>>>(r, g, static_cast<const uint4*>(y_perm),
                                                          static_cast<const uint4*>(y_shared), w, perm_dst, status);
  return cudaGetLastError();
}

cudaError_t launch_retile(const void* a, const void* b, int E, int R, long long row_bytes, bool gate_up, void* dst,
                          cudaStream_t s) {
  if (R % 256 != 0 || row_bytes % 128 != 0) return cudaErrorInvalidValue;
  retile_kernel<<<4096, 256, 0, s>>>(static_cast<const uint4*>(a), static_cast<const uint4*>(b), E, R,
                                     static_cast<int>(row_bytes / 16), gate_up, static_cast<uint4*>(dst));
  return cudaGetLastError();
}

}  // namespace asap
