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

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kDispatchWarps = kChunkTokens;  // one warp per token for the copies
constexpr int kRankWarps = kChunkTokens * kMaxTopK / 32;  // warps that rank the chunk's entries

// One CTA per chunk of kChunkTokens tokens.  Entry i = t_local * k + j is
// ranked by thread i, so warp order and lane order follow (t, j); the rank of
// an entry inside its expert is (entries of that expert in earlier chunks)
// + (in earlier warps of this chunk) + (in earlier lanes of this warp):
// positions increase with (t, j) inside every segment.  chunk_base is
// expert-major: chunk_base[e * n_chunks + chunk].  Then one warp per token
// reads its row once and writes it to its k positions.
__global__ void __launch_bounds__(kDispatchWarps * 32)
    dispatch_kernel(const uint4* __restrict__ x, int n, int V, int k, int E,
                    const int32_t* __restrict__ idx, const int32_t* __restrict__ chunk_base, int n_chunks,
                    uint4* __restrict__ x_perm, int32_t* __restrict__ perm_src,
                    int32_t* __restrict__ perm_dst, uint32_t* status) {
  __shared__ int wcnt[kRankWarps][kMaxExperts];
  __shared__ int spos[kChunkTokens * kMaxTopK];
  const int c = blockIdx.x;
  const int t0 = c * kChunkTokens;
  const int nt = min(kChunkTokens, n - t0);
  const int ne = nt * k;
  const int nk = n * k;
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
    int run = chunk_base[static_cast<long long>(ee) * n_chunks + c];
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
    perm_dst[static_cast<long long>(t0) * k + i] = pos;
    if (pos >= 0) perm_src[pos] = t0 + i / k;
  }
  __syncthreads();
  // row copies: one warp per token, read once, write k times
  if (warp < nt) {
    const uint4* src = x + static_cast<long long>(t0 + warp) * V;
    int p[kMaxTopK];
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) p[j] = j < k ? spos[warp * k + j] : -1;
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
    }
    for (; v < V; v += 32) {
      const uint4 a = __ldg(src + v);
#pragma unroll
      for (int j = 0; j < kMaxTopK; ++j)
        if (p[j] >= 0) x_perm[static_cast<long long>(p[j]) * V + v] = a;
    }
  }
}

constexpr int kCombineWarps = 8;

// One warp per token: out[t] = sum_j w[t,j] y_perm[perm_dst[t,j]] (+ y_sh[t]),
// fp32 fused multiply-adds in slot order, then the shared row, then bf16.
__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_kernel(const uint4* __restrict__ y_perm, const uint4* __restrict__ y_sh,
                   const float* __restrict__ w, const int32_t* __restrict__ perm_dst, int n, int V,
                   int k, uint4* __restrict__ out, uint32_t* status) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kCombineWarps + warp;
  if (t >= n) return;
  const long long nk = static_cast<long long>(n) * k;
  int p[kMaxTopK];
  float wj[kMaxTopK];
#pragma unroll
  for (int j = 0; j < kMaxTopK; ++j) {
    p[j] = -1;
    wj[j] = 0.f;
    if (j < k) {
      p[j] = perm_dst[static_cast<long long>(t) * k + j];
      wj[j] = w[static_cast<long long>(t) * k + j];
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
    if (y_sh) {
      const uint4 s = __ldg(y_sh + static_cast<long long>(t) * V + v);
      acc[0] += bf16_lo(s.x);
      acc[1] += bf16_hi(s.x);
      acc[2] += bf16_lo(s.y);
      acc[3] += bf16_hi(s.y);
      acc[4] += bf16_lo(s.z);
      acc[5] += bf16_hi(s.z);
      acc[6] += bf16_lo(s.w);
      acc[7] += bf16_hi(s.w);
    }
    out[static_cast<long long>(t) * V + v] =
        make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                   pack_bf16x2(acc[6], acc[7]));
  }
}

// packed[e][b*256 + r] = gate[e][b*128 + r] for r < 128, up[e][b*128 + r - 128]
// otherwise, so one 256-row weight tile holds 128 gate rows and the matching
// 128 up rows.
__global__ void pack_gate_up_kernel(const uint4* __restrict__ gate, const uint4* __restrict__ up, int E,
                                    int I, int V, uint4* __restrict__ packed) {
  const long long total = static_cast<long long>(E) * 2 * I * V;
  for (long long q = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; q < total;
       q += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int v = static_cast<int>(q % V);
    const long long rowq = q / V;
    const int r = static_cast<int>(rowq % (2 * I));
    const long long e = rowq / (2 * I);
    const int b = r / 256, rr = r % 256;
    const int src_row = b * 128 + (rr & 127);
    const uint4* src = rr < 128 ? gate : up;
    packed[q] = src[(e * I + src_row) * V + v];
  }
}

}  // namespace

cudaError_t launch_dispatch(const void* x, int n, int H, int k, int E, const int32_t* idx,
                            const int32_t* chunk_base, void* x_perm, int32_t* perm_src,
                            int32_t* perm_dst, uint32_t* status, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int chunks = ceil_div(n, kChunkTokens);
  dispatch_kernel<<<chunks, kDispatchWarps * 32, 0, s>>>(static_cast<const uint4*>(x), n, H / 8, k, E, idx,
                                                         chunk_base, chunks, static_cast<uint4*>(x_perm), perm_src,
                                                         perm_dst, status);
  return cudaGetLastError();
}

cudaError_t launch_combine(const void* y_perm, const void* y_shared, const float* w,
                           const int32_t* perm_dst, int n, int H, int k, void* out, uint32_t* status,
                           cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  combine_kernel<<<ceil_div(n, kCombineWarps), kCombineWarps * 32, 0, s>>>(
      static_cast<const uint4*>(y_perm), static_cast<const uint4*>(y_shared), w, perm_dst, n, H / 8, k,
      static_cast<uint4*>(out), status);
  return cudaGetLastError();
}

cudaError_t launch_pack_gate_up(const void* gate, const void* up, int E, int I, int H, void* packed,
                                cudaStream_t s) {
  pack_gate_up_kernel<<<4096, 256, 0, s>>>(static_cast<const uint4*>(gate), static_cast<const uint4*>(up), E, I,
                                           H / 8, static_cast<uint4*>(packed));
  return cudaGetLastError();
}

}  // namespace asap
