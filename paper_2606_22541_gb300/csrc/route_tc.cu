// Routing of a micro-batch in one launch on the sm_103a tensor core: router
// logits, grouped sigmoid gating with top-k, the expert histogram and its
// scan into per-expert counts and offsets (the metadata the MoE side of ASAP
// receives per DP group, Section 3.2.1; Table 1: top-K of E_total = 256).
//
// Design (one 128-token tile per thread-block cluster):
//  - The cluster has ``splits`` CTAs (1, 2 or 4); CTA r computes the partial
//    logits of the tile over K slice r (the same slices as the standalone
//    router GEMM): TMA rings of x [128 x 64] and router-weight [256 x 64]
//    boxes, tcgen05.mma kind::f16 M=128 N=256 into one TMEM accumulator.
//  - Or (seq_slices > 1, no cluster) one CTA computes the slices one after
//    the other: slice 0 into TMEM columns 0.., each later slice into columns
//    256.., which the epilogue warps add into the first buffer (TMEM load,
//    fp32 add, TMEM store) while the next slice streams -- the same sum in
//    the same order, so the same logits, on a quarter of the SMs.  Several
//    micro-batches routed at once then run side by side in one wave.
//  - Each 32-token quarter q of the tile is gated by CTA q % splits.  The
//    epilogue warps read their quarter from TMEM and store it into the owning
//    CTA's shared memory through distributed shared memory, one slot per K
//    slice; the owner adds the slots in slice order, so the logits are
//    bit-identical to the K-slice planes added in order.
//  - Gating of a quarter: warp b holds experts 32b .. 32b+31 of every token
//    (lane = token): sigmoid scores (kept in shared memory), selection keys
//    (score + bias), each block's top-2 keys, group scores (sum of the
//    group's top-2 keys) and the groups kept by rank.  Each eligible block
//    (in a kept group) holds at least two keys >= its second key, so when
//    the eligible blocks hold at least k such keys, the smallest second key T
//    of the eligible blocks is a lower bound of the token's k-th selected
//    key: only eligible keys >= T can be selected.  One thread per token
//    then inserts just those candidates, in increasing expert order, into its
//    top-k by (key desc, expert asc).  Same scores, keys, tie-breaks and
//    weight arithmetic as the gate kernels, so the same experts and weights.
//  - Per-chunk histograms go to hist[chunk][e]; the last CTA to finish
//    (ticket counter, zero at launch) scans them into chunk bases, counts and
//    offsets, one thread per expert.
// The shared memory of the operand rings is reused for the partial-logit
// slots and the gate's scratch once every CTA of the cluster is done with its
// rings (cluster barrier).  Every wait is bounded; on a timeout the CTA still
// takes part in both cluster barriers, so no CTA leaves while a peer may
// still write to its shared memory.
#include "common.cuh"
#include "gemm_config.h"
#include "internal.h"

#include <math_constants.h>

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kRA = ASAP_RING_RT_A, kRB = ASAP_RING_RT_B;
constexpr int kABytes = kGemmBM * kGemmBK * 2;  // x box
constexpr int kBBytes = kGemmBN * kGemmBK * 2;  // router-weight box
constexpr int kRingBytes = kRA * kABytes + kRB * kBBytes;
constexpr int kThreads = 256;  // warp 0 B producer, 1 MMA, 2-5 epilogue, 6 A producer, 7 gate only
constexpr int kBlocks = 8;     // 32-expert blocks of the 256 experts (one warp each in the gate)
constexpr int kSlotFloat4 = 32 * kRouteExperts / 4;       // one 32-token partial slot
constexpr int kRecvBytes = 4 * kSlotFloat4 * 16;          // (4 / splits) quarters x splits slots
constexpr int kSigPitch = 33;                                   // floats per expert row (bank spread)
constexpr int kSigOff = kRecvBytes;                             // sigmoid scores [expert][token]
constexpr int kTopOff = kSigOff + kRouteExperts * kSigPitch * 4;  // per block: top-2 keys per token
constexpr int kMaskOff = kTopOff + 2 * kBlocks * 32 * 4;        // per block: candidate bits per token
constexpr int kHistOff = kMaskOff + kBlocks * 32 * 4;           // chunk histogram
constexpr int kWarpSumOff = kHistOff + kRouteExperts * 4;       // the scan's warp totals
constexpr int kScratchEnd = kWarpSumOff + 40 * 4;
static_assert(kScratchEnd <= kRingBytes, "the gate's scratch overlays the operand rings");
static_assert(kThreads == kRouteExperts, "the scan gives one thread per expert");
constexpr int kBarOff = kRingBytes;
// mbarriers fullA[kRA], emptyA[kRA], fullB[kRB], emptyB[kRB], tfull, drain,
// bfree; then the TMEM address, abort flag, last-CTA flag and the bias pointer
constexpr int kNumBars = 2 * kRA + 2 * kRB + 3;
constexpr int kBarBytes = 8 * kNumBars + 32;
constexpr size_t kSmem = kRingBytes + kBarBytes;
constexpr uint32_t kIdesc = idesc_bf16_f32(kGemmBM, kGemmBN);

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Shared-memory address of the same offset in CTA ``rank`` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(addr), "r"(rank));
  return d;
}
__device__ __forceinline__ void st_cluster_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared::cluster.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
// All threads of every CTA of the cluster; orders shared and global memory
// (release on arrive, acquire on wait).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
}

// 32 lanes x 16 consecutive 32-bit columns from registers into TMEM (the
// warp's own lane quarter).
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ int warp_inclusive_scan(int v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int u = __shfl_up_sync(kFull, v, o);
    if (lane >= o) v += u;
  }
  return v;
}

__global__ void __launch_bounds__(kThreads, 1)
    route_fused_kernel(const __grid_constant__ CUtensorMap tmX, const RouteFusedArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const uint32_t base = smem_u32(smem);
  const bool aligned = (base & 1023u) == 0;  // the 128-byte swizzle needs it; uniform for the CTA
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int splits = a.splits;
  const uint32_t rank = cluster_ctarank();
  const int tile = blockIdx.x / splits;
  const int row0 = tile * kGemmBM;
  // K slice of this CTA: the bounds the standalone router GEMM uses
  const int kb0 = static_cast<int>(static_cast<long long>(a.k_iters) * rank / splits);
  const int kb1 = static_cast<int>(static_cast<long long>(a.k_iters) * (rank + 1) / splits);
  const uint32_t sA = base, sB = base + kRA * kABytes;
  uint8_t* bar_area = smem + kBarOff;
  const uint32_t bar0 = smem_u32(bar_area);
  auto fullA = [&](int s) { return bar0 + 8u * s; };
  auto emptyA = [&](int s) { return bar0 + 8u * (kRA + s); };
  auto fullB = [&](int s) { return bar0 + 8u * (2 * kRA + s); };
  auto emptyB = [&](int s) { return bar0 + 8u * (2 * kRA + kRB + s); };
  const uint32_t tfull = bar0 + 8u * (2 * kRA + 2 * kRB);
  const uint32_t drain = tfull + 8u;
  const uint32_t bfree = drain + 8u;  // sequential slices: the second TMEM buffer was added in
  // K slices computed one after the other by this CTA (1 with a cluster)
  const int nseq = splits == 1 ? max(a.seq_slices, 1) : 1;
  const uint32_t tmem_cols = nseq > 1 ? 2 * kGemmBN : kGemmBN;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_area + 8 * kNumBars);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);
  volatile int* acc_bad = reinterpret_cast<volatile int*>(tmem_slot + 3);
  const float** bias_slot = reinterpret_cast<const float**>(tmem_slot + 4);
  const CUtensorMap* tmW = nullptr;

  if (warp == 0) {
    if (lane == 0) {
      const LayerEntry& le =
          a.lref.table[load_layer(a.lref.layer, a.lref.n_layers, a.status, blockIdx.x == 0)];
      tmW = &le.map[MAP_ROUTER];
      *bias_slot = le.router_bias;
      tensormap_acquire(tmW);
      for (int s = 0; s < kRA; ++s) {
        mbar_init(fullA(s), 1);
        mbar_init(emptyA(s), 1);
      }
      for (int s = 0; s < kRB; ++s) {
        mbar_init(fullB(s), 1);
        mbar_init(emptyB(s), 1);
      }
      mbar_init(tfull, 1);
      mbar_init(drain, 1);
      mbar_init(bfree, 128);  // the four epilogue warps
      *abort_flag = 0;
      *last_flag = 0;
      *acc_bad = aligned ? 0 : 1;
      fence_barrier_init();
      tma_prefetch_desc(&tmX);
      tma_prefetch_desc(tmW);
      if (!aligned) record_status(a.status, ST_SMEM_ALIGN);
    }
  } else if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  bool ok = aligned;  // epilogue warps: the accumulator is complete
  if (aligned && (warp == 0 || warp == 6) && lane == 0) {
    // ------------------------------------------------------------ producers
    const bool isB = warp == 0;
    const int nst = isB ? kRB : kRA;
    const uint32_t bytes = isB ? kBBytes : kABytes;
    const uint32_t ring = isB ? sB : sA;
    const uint64_t pol = l2_policy(isB ? 2 : 0);  // router weights are re-read by every tile
    const CUtensorMap* m = isB ? tmW : &tmX;
    const int row = isB ? 0 : row0;
    int stage = 0;
    uint32_t phase = 0, pending = 0, issued_phase = 0;
    bool good = true;
    for (int kb = kb0; kb < kb1; ++kb) {
      if (!mbar_wait(isB ? emptyB(stage) : emptyA(stage), phase ^ 1u, abort_flag)) {
        good = false;
        break;
      }
      const uint32_t full = isB ? fullB(stage) : fullA(stage);
      mbar_arrive_expect_tx(full, bytes);
      tma_load_2d(ring + stage * bytes, m, full, kb * kGemmBK, row, pol);
      pending |= 1u << stage;
      issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
      if (++stage == nst) {
        stage = 0;
        phase ^= 1u;
      }
    }
    if (!good) {
      *abort_flag = 1;
      record_status(a.status, ST_WAIT_TIMEOUT);
      int dummy = 0;
      for (int s = 0; s < nst; ++s)
        if (pending & (1u << s)) mbar_wait(isB ? fullB(s) : fullA(s), (issued_phase >> s) & 1u, &dummy);
    }
  } else if (aligned && warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    int sa = 0, sb = 0;
    uint32_t pa = 0, pb = 0;
    bool good = true, issued = false;
    // slice q of nseq covers k-blocks [k_iters q / nseq, k_iters (q + 1) / nseq)
    // (the bounds of a cluster's CTAs); slice 0 accumulates into TMEM columns
    // 0.., the later ones into columns 256.., which the epilogue warps add into
    // the first buffer before the next slice may start there
    int q = 0, q_start = kb0;
    int q_end = nseq > 1 ? static_cast<int>(static_cast<long long>(a.k_iters) / nseq) : kb1;
    for (int kb = kb0; kb < kb1; ++kb) {
      if (kb == q_start && q >= 2 && !mbar_wait(bfree, (q - 2) & 1, abort_flag)) {
        good = false;
        break;
      }
      if (!mbar_wait(fullA(sa), pa, abort_flag) || !mbar_wait(fullB(sb), pb, abort_flag)) {
        good = false;
        break;
      }
      tc_fence_after();
      const uint32_t a_addr = sA + sa * kABytes, b_addr = sB + sb * kBBytes;
      const uint32_t d = tmem_base + (q == 0 ? 0u : static_cast<uint32_t>(kGemmBN));
#pragma unroll
      for (int kk = 0; kk < kGemmBK / 16; ++kk)
        tc_mma_bf16(d, smem_desc_sw128(a_addr + kk * 32), smem_desc_sw128(b_addr + kk * 32), kIdesc,
                    (kb > q_start || kk > 0) ? 1u : 0u);
      issued = true;
      tc_commit(emptyA(sa));
      tc_commit(emptyB(sb));
      if (++sa == kRA) {
        sa = 0;
        pa ^= 1u;
      }
      if (++sb == kRB) {
        sb = 0;
        pb ^= 1u;
      }
      if (kb + 1 == q_end && q + 1 < nseq) {
        tc_commit(tfull);  // slice q complete
        ++q;
        q_start = kb + 1;
        q_end = static_cast<int>(static_cast<long long>(a.k_iters) * (q + 1) / nseq);
      }
    }
    if (good) {
      tc_commit(tfull);
    } else {
      *abort_flag = 1;
      record_status(a.status, ST_WAIT_TIMEOUT);
      if (issued) {
        int dummy = 0;
        tc_commit(drain);
        mbar_wait(drain, 0, &dummy);
      }
    }
  } else if (warp >= 2 && warp <= 5) {
    if (aligned) {
      ok = __all_sync(kFull, mbar_wait(tfull, 0, abort_flag));
      // sequential slices: add slice q (columns 256..) into the sum of the
      // slices before it (columns 0..), in slice order, each warp its 32 lanes
      const uint32_t lanes = tmem_base + (static_cast<uint32_t>((warp & 3) * 32) << 16);
      for (int qs = 1; ok && qs < nseq; ++qs) {
        ok = __all_sync(kFull, mbar_wait(tfull, qs & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kGemmBN; c += 16) {
          uint32_t acc[16], part[16];
          tmem_ld16(lanes + c, acc);
          tmem_ld16(lanes + kGemmBN + c, part);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[i] = __float_as_uint(__uint_as_float(acc[i]) + __uint_as_float(part[i]));
          tmem_st16(lanes + c, acc);
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(bfree);
      }
      if (!ok && lane == 0) {
        *abort_flag = 1;
        *acc_bad = 1;
        record_status(a.status, ST_WAIT_TIMEOUT);
      }
    }
  }
  __syncwarp();
  tc_fence_before();
  // (1) every CTA of the cluster is done with its rings: they may now receive
  cluster_sync_all();

  if (!*acc_bad) {
    // ------------------------------------------------------------ partial logits to the owner
    // warp w reads TMEM lanes 32 (w % 4) .. (the tokens of quarter w % 4),
    // columns 128 (w / 4) .. + 127
    tc_fence_after();
    const int q = warp & 3;
    const int c_lo = (warp >> 2) * (kGemmBN / 2);
    const uint32_t owner = static_cast<uint32_t>(q % splits);
    const int j = q / splits;
    const uint32_t local = base + static_cast<uint32_t>((j * splits + static_cast<int>(rank)) * kSlotFloat4 * 16);
    const bool remote = owner != rank;  // the own quarter stays in this CTA
    const uint32_t slot = remote ? mapa_shared(local, owner) : local;
    const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    // all 128 columns in flight before one wait, then the stores
    uint32_t v[4][32];
#pragma unroll
    for (int u = 0; u < 4; ++u) tmem_ld32(taddr + c_lo + 32 * u, v[u]);
    tmem_ld_wait();
#pragma unroll
    for (int u = 0; u < 4; ++u) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        // float4 (experts 4f .. 4f+3) of this token: (f * 32 + token) in the slot
        const uint32_t ad = slot + static_cast<uint32_t>((((c_lo + 32 * u) / 4 + i) * 32 + lane) * 16);
        if (remote)
          st_cluster_v4(ad, v[u][4 * i], v[u][4 * i + 1], v[u][4 * i + 2], v[u][4 * i + 3]);
        else
          st_shared_v4(ad, v[u][4 * i], v[u][4 * i + 1], v[u][4 * i + 2], v[u][4 * i + 3]);
      }
    }
  }
  tc_fence_before();
  // (2) the slots are complete; no CTA touches another's memory after this
  cluster_sync_all();

  // ------------------------------------------------------------ gating
  const float4* recv = reinterpret_cast<const float4*>(smem);
  float* sig = reinterpret_cast<float*>(smem + kSigOff);
  float* top1 = reinterpret_cast<float*>(smem + kTopOff);
  float* top2 = top1 + kBlocks * 32;
  uint32_t* cmask = reinterpret_cast<uint32_t*>(smem + kMaskOff);
  int* shist = reinterpret_cast<int*>(smem + kHistOff);
  const float* bias = *bias_slot;
  const int G = a.n_groups;  // 1, 2, 4 or 8: a group is 8 / G blocks
  const int bpg = kBlocks / G;
  const int k = a.top_k;
  const int n_chunks = (a.n + kChunkTokens - 1) / kChunkTokens;
  shist[threadIdx.x] = 0;
  __syncthreads();
#pragma unroll 1
  for (int j = 0; j < 4 / splits; ++j) {
    const int qq = j * splits + static_cast<int>(rank);  // quarter of the tile gated here
    const int t0 = row0 + 32 * qq;
    if (t0 >= a.n) continue;  // the same for the whole CTA
    const int t = t0 + lane;
    float key[32];
    {
      const float4* s0 = recv + j * splits * kSlotFloat4;
#pragma unroll
      for (int c4 = 0; c4 < 8; ++c4) {
        const int f = (8 * warp + c4) * 32 + lane;
        float4 v = s0[f];
        for (int r = 1; r < splits; ++r) {  // K slices in order
          const float4 u = s0[r * kSlotFloat4 + f];
          v.x += u.x;
          v.y += u.y;
          v.z += u.z;
          v.w += u.w;
        }
        key[4 * c4] = v.x;
        key[4 * c4 + 1] = v.y;
        key[4 * c4 + 2] = v.z;
        key[4 * c4 + 3] = v.w;
      }
    }
    float m1 = -CUDART_INF_F, m2 = -CUDART_INF_F;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const float sg = gate_sigmoid(key[i]);
      sig[(32 * warp + i) * kSigPitch + lane] = sg;
      key[i] = sg + (bias ? __ldg(bias + 32 * warp + i) : 0.0f);
      // the two largest keys (an equal key becomes the second)
      m2 = fmaxf(m2, fminf(m1, key[i]));
      m1 = fmaxf(m1, key[i]);
    }
    top1[warp * 32 + lane] = m1;
    top2[warp * 32 + lane] = m2;
    __syncthreads();
    // group scores: the two largest keys of each group's blocks, summed; a
    // group is kept when fewer than topk_groups groups come before it (larger
    // score, or an equal score and a lower index)
    float gsv[kBlocks];
#pragma unroll
    for (int g = 0; g < kBlocks; ++g) {
      float h1 = -CUDART_INF_F, h2 = -CUDART_INF_F;
      if (g < G) {
        h1 = top1[g * bpg * 32 + lane];
        h2 = top2[g * bpg * 32 + lane];
        for (int b = g * bpg + 1; b < (g + 1) * bpg; ++b) {
          const float a1 = top1[b * 32 + lane], a2 = top2[b * 32 + lane];
          const float hi = fmaxf(h1, a1);
          const float lo = fmaxf(fminf(h1, a1), fmaxf(h2, a2));
          h1 = hi;
          h2 = lo;
        }
      }
      gsv[g] = h1 + h2;
    }
    uint32_t kept = 0;  // bit g: group g is kept
#pragma unroll
    for (int g = 0; g < kBlocks; ++g) {
      int grank = 0;
#pragma unroll
      for (int g2 = 0; g2 < kBlocks; ++g2)
        if (g2 < G) grank += (gsv[g2] > gsv[g] || (gsv[g2] == gsv[g] && g2 < g)) ? 1 : 0;
      if (g < G && grank < a.topk_groups) kept |= 1u << g;
    }
    // T: the smallest second key of the eligible blocks, when they hold at
    // least k keys >= it (two per block); else every eligible key is a
    // candidate
    float T = CUDART_INF_F;
    int nel = 0;
#pragma unroll
    for (int b = 0; b < kBlocks; ++b)
      if ((kept >> (b / bpg)) & 1u) {
        T = fminf(T, top2[b * 32 + lane]);
        ++nel;
      }
    if (2 * nel < k) T = -CUDART_INF_F;
    uint32_t bits = 0;
    if (t < a.n && ((kept >> (warp / bpg)) & 1u)) {  // (rows past the end are zero-filled)
#pragma unroll
      for (int i = 0; i < 32; ++i) bits |= (key[i] >= T ? 1u : 0u) << i;
    }
    cmask[warp * 32 + lane] = bits;
    __syncthreads();
    {
      // the token's top-k: lanes 8u .. 8u+7 of warp w serve token 4w + u of
      // the quarter, one lane per block.  Each lane keeps its block's top 8
      // candidates by (key desc, expert asc); they arrive in increasing
      // expert order, so an equal key never passes one already held.  Then k
      // rounds: the best head of the 8 lanes (butterfly; larger key, then
      // lower expert) is the next pick and its lane pops it.
      const int tt = 4 * warp + (lane >> 3);
      const int b = lane & 7;
      float lk[kMaxTopK], lv[kMaxTopK];
      int le[kMaxTopK];
#pragma unroll
      for (int s = 0; s < kMaxTopK; ++s) {
        lk[s] = -CUDART_INF_F;
        lv[s] = 0.f;
        le[s] = 0x7fffffff;
      }
      uint32_t m = cmask[b * 32 + tt];
      while (m) {
        const int i = __ffs(m) - 1;
        m &= m - 1;
        const int e = 32 * b + i;
        const float x = sig[e * kSigPitch + tt];
        const float v = x + (bias ? __ldg(bias + e) : 0.0f);
#pragma unroll
        for (int s = kMaxTopK - 1; s >= 1; --s) {  // selects, from the old entries
          const bool up = v > lk[s - 1], here = v > lk[s];
          lk[s] = up ? lk[s - 1] : (here ? v : lk[s]);
          le[s] = up ? le[s - 1] : (here ? e : le[s]);
          lv[s] = up ? lv[s - 1] : (here ? x : lv[s]);
        }
        const bool top = v > lk[0];
        lk[0] = top ? v : lk[0];
        le[0] = top ? e : le[0];
        lv[0] = top ? x : lv[0];
      }
      int es[kMaxTopK];
      float xs[kMaxTopK];
      float sum = 0.f;
#pragma unroll
      for (int r = 0; r < kMaxTopK; ++r) {
        es[r] = 0x7fffffff;
        xs[r] = 0.f;
        if (r < k) {
          float v = lk[0], x = lv[0];
          int e = le[0];
#pragma unroll
          for (int o = 1; o < 8; o <<= 1) {
            const float ov = __shfl_xor_sync(kFull, v, o);
            const int oe = __shfl_xor_sync(kFull, e, o);
            const float ox = __shfl_xor_sync(kFull, x, o);
            if (ov > v || (ov == v && oe < e)) {
              v = ov;
              e = oe;
              x = ox;
            }
          }
          const bool pop = le[0] == e;
#pragma unroll
          for (int s = 0; s < kMaxTopK - 1; ++s) {
            lk[s] = pop ? lk[s + 1] : lk[s];
            le[s] = pop ? le[s + 1] : le[s];
            lv[s] = pop ? lv[s + 1] : lv[s];
          }
          lk[kMaxTopK - 1] = pop ? -CUDART_INF_F : lk[kMaxTopK - 1];
          le[kMaxTopK - 1] = pop ? 0x7fffffff : le[kMaxTopK - 1];
          es[r] = e;
          xs[r] = x;
          sum += x;
        }
      }
      const int tg = t0 + tt;
      if (b == 0 && tg < a.n) {
#pragma unroll
        for (int r = 0; r < kMaxTopK; ++r) {
          if (r < k) {
            a.idx[static_cast<long long>(tg) * k + r] = es[r];
            a.w[static_cast<long long>(tg) * k + r] = xs[r] / sum * a.route_scale;
            if (es[r] >= 0 && es[r] < kRouteExperts) atomicAdd(&shist[es[r]], 1);
          }
        }
      }
    }
    __syncthreads();
    const int chunk = tile * 4 + qq;
    if (chunk < n_chunks)
      a.hist[static_cast<long long>(a.chunk0 + chunk) * kRouteExperts + threadIdx.x] = shist[threadIdx.x];
    shist[threadIdx.x] = 0;
    __syncthreads();
  }

  // ------------------------------------------------------------ scan (last CTA)
  if (a.ticket) {
    __threadfence();  // this thread's histogram stores before the ticket
    __syncthreads();
    if (threadIdx.x == 0) *last_flag = atomicAdd(a.ticket, 1) == static_cast<int>(gridDim.x) - 1 ? 1 : 0;
    __syncthreads();
    if (*last_flag) {
      __threadfence();
      // thread e: expert e's column of the chunk-major histogram, 64 rows in
      // flight at a time
      const int e = threadIdx.x;
      const int nct = a.n_chunks_total;
      int run = 0;
#pragma unroll 1
      for (int c0 = 0; c0 < nct; c0 += 64) {
        int v[64];
#pragma unroll
        for (int u = 0; u < 64; ++u)
          v[u] = c0 + u < nct ? __ldcg(a.hist + static_cast<long long>(c0 + u) * kRouteExperts + e) : 0;
#pragma unroll
        for (int u = 0; u < 64; ++u) {
          if (c0 + u < nct) a.chunk_base[static_cast<long long>(c0 + u) * kRouteExperts + e] = run;
          run += v[u];
        }
      }
      // offsets: exclusive scan of the counts, one thread per expert
      int* swarp = reinterpret_cast<int*>(smem + kWarpSumOff);
      const int incl = warp_inclusive_scan(run);
      if (lane == 31) swarp[warp] = incl;
      __syncthreads();
      int before = 0;
      for (int w2 = 0; w2 < warp; ++w2) before += swarp[w2];
      a.counts[e] = run;
      a.offsets[e] = before + incl - run;
      if (e == kRouteExperts - 1) a.offsets[kRouteExperts] = before + incl;
      // the grouped GEMMs that follow on this stream claim tiles from these
      if (a.tile_counters && threadIdx.x < kTileCounters) a.tile_counters[threadIdx.x] = 0;
      if (threadIdx.x == 0) *a.ticket = 0;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, tmem_cols);
  }
}

}  // namespace

cudaError_t route_fused_set_attributes() {
  return cudaFuncSetAttribute(route_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kSmem));
}

cudaError_t launch_route_fused(const CUtensorMap& tmX, const RouteFusedArgs& a, cudaStream_t s) {
  if (a.n <= 0) return cudaSuccess;
  if (!(a.splits == 1 || a.splits == 2 || a.splits == 4) || !(a.n_groups == 1 || a.n_groups == 2 ||
                                                              a.n_groups == 4 || a.n_groups == 8) ||
      a.top_k < 1 || a.top_k > kMaxTopK || a.k_iters < a.splits ||
      !(a.seq_slices <= 1 || (a.splits == 1 && (a.seq_slices == 2 || a.seq_slices == 4) && a.k_iters >= a.seq_slices)))
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(ceil_div(a.n, kGemmBM) * a.splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(a.splits);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, route_fused_kernel, tmX, a);
}

}  // namespace asap
