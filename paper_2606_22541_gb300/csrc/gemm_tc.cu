// Grouped GEMM on the sm_103a tensor core (tcgen05 + TMEM), fed by TMA.
//
// This is the expert computation of the MoE layer: a grouped matrix
// multiplication with the token hidden states on the left and one layer's
// expert weights on the right (ASAP Section 3.4.2).  Each expert e owns the
// row segment [offsets[e], offsets[e+1]) of the grouped activations; the tile
// list is derived on the device from those offsets, so the host never reads
// the per-expert counts back (the bubble-free principle of Section 3.4.2).
//
// Design (one CTA per SM, persistent, warp-specialised; 224 threads, 352 with
// paired m-tiles):
//   warp 0   : weight producer.  B boxes [256 rows, 64 K] into its ring; the
//              weights are stored tile-contiguous (one 32 KB read per box).
//   last warp: activation producer.  A boxes [128 rows, 64 K] (two per stage
//              for a paired tile) into its ring.  Ring depths per launch kind
//              in gemm_config.h; 128-byte swizzle.
//   warp 1   : TMEM allocator and MMA issuer (one thread): per stage 4 x
//              tcgen05.mma.cta_group::1.kind::f16 (M=128, N=256, K=16), twice
//              for a paired tile; fp32 accumulators in TMEM (2 x 256 columns:
//              ping-pong accumulators for single m-tiles, the two halves of a
//              paired tile).
//   epilogue : warps 2-5 (2-9 paired).  tcgen05.ld 32x32b (warp w reads TMEM
//              lanes 32*(w%4) ...), fused SwiGLU (gate and up columns of a
//              tile are the two 128-column halves), bf16 stores staged through
//              shared memory so each store writes whole 128-byte row pieces
//              (fp32 router logits are stored directly).
// Weights: the B descriptors come from the layer table (one entry per layer,
// in global memory) at the layer id the kernel loads when it starts, so one
// launch sequence serves any layer (the MoE Super Kernel of Section 3.4.2).
// Tile order: expert-major; inside an expert the m-tiles of one n-tile are
// adjacent so CTAs running at the same time share the weight tile through L2.
// Rows of a tile past the segment end belong to the next expert (or are
// zero-filled by TMA past the tensor end) and are masked at the store.
#include "common.cuh"
#include "gemm_config.h"
#include "gemm_sched.cuh"
#include "internal.h"

#include <mutex>

namespace asap {

namespace {

// Shape of one launch kind.  PAIR: a tile is two 128-row m-tiles of the same
// expert and n-tile that share every weight box (two M = 128 MMAs per K
// step into the two halves of TMEM); each weight box then feeds twice the MMA
// work, so the same ring bytes cover twice the load latency.  The last tile
// of a segment whose remaining rows fit one m-tile is a half tile: one A box
// and one MMA per K step, so a segment pays for at most 127 padding rows, as
// without PAIR.  Without PAIR a tile is one 128-row m-tile and the two TMEM
// halves are ping-pong accumulators (the epilogue of one tile overlaps the
// main loop of the next).  Ring depths per launch kind in gemm_config.h.
template <int EPI, bool PAIR>
struct Gemm {
  static constexpr int BMT = PAIR ? 2 * kGemmBM : kGemmBM;  // rows per tile
  static constexpr int SA = PAIR ? ASAP_RING_PAIR_A
                                 : EPI == EPI_BF16 ? ASAP_RING_DN_A : EPI == EPI_SWIGLU ? ASAP_RING_GU_A : ASAP_RING_RT_A;
  static constexpr int SB = PAIR ? ASAP_RING_PAIR_B
                                 : EPI == EPI_BF16 ? ASAP_RING_DN_B : EPI == EPI_SWIGLU ? ASAP_RING_GU_B : ASAP_RING_RT_B;
  static constexpr int A_BYTES = BMT * kGemmBK * 2;
  static constexpr int EPI_WARPS = PAIR ? 8 : 4;        // two per TMEM lane quarter with PAIR (one per half)
  static constexpr int kThreads = 32 * (3 + EPI_WARPS);  // warp 0 B producer, 1 MMA, epilogue, last A producer
  static constexpr int kAProdWarp = 2 + EPI_WARPS;
};
constexpr int BM = kGemmBM, BN = kGemmBN, BK = kGemmBK;


constexpr int B_BYTES = BN * BK * 2;
constexpr uint32_t kTmemCols = 2 * BN;
constexpr uint32_t kIdesc = idesc_bf16_f32(BM, BN);
// A 128-row half of an expert tile that holds at most 64 rows (a segment's
// tail) takes one M = 64 MMA instead of an M = 128 one: rows are padded to 64
// instead of 128, which removes about half of the padding work (at 8192 tokens
// of the DeepSeek-V3 shape 26 % more MMA rows than routed rows with 128-row
// granularity, 13 % with 64-row tails).  Its accumulator rows sit in TMEM
// lanes 0-15 of each 32-lane quarter (row 16 q + i in lane 32 q + i).  Expert
// GEMMs only; the router keeps M = 128 (its logits must match the one-launch
// route bit for bit).
constexpr uint32_t kIdesc64 = idesc_bf16_f32(64, BN);
constexpr int kTailRows = 64;

constexpr int kBarBytes = 384;  // 2*SA + 2*SB + 5 + 2*kTileQ mbarriers, tmem slot, abort flag, tile ids
// bf16 epilogues stage their stores through 4 KB of shared memory per warp
// (32 rows x 8 chunks of 16 bytes)
constexpr int kStageWarpBytes = 32 * 8 * 16;
template <int EPI, bool PAIR>
__host__ __device__ constexpr int stage_bytes() {
  return EPI == EPI_F32 ? 0 : Gemm<EPI, PAIR>::EPI_WARPS * kStageWarpBytes;
}
// Dynamic shared memory: rings (1024-byte aligned for the 128-byte swizzle,
// the alignment the kernel declares and checks), barriers, store staging,
// schedule table.
template <int EPI, bool PAIR>
__host__ __device__ constexpr size_t smem_bytes() {
  return Gemm<EPI, PAIR>::SA * Gemm<EPI, PAIR>::A_BYTES + Gemm<EPI, PAIR>::SB * B_BYTES + kBarBytes +
         stage_bytes<EPI, PAIR>() + sizeof(Sched);
}


// One round of a warp's stores: lane l holds 8 chunks of 16 bytes (pk, 32
// words) of its row l.  Every lane writes them to the warp's 4 KB staging
// buffer, chunk j of row r at slot j ^ (r % 8): the layout of a [32 rows, 64
// columns] bf16 box under the 128-byte swizzle (the buffer is 1024-byte
// aligned).  A warp whose 32 rows all belong to the tile (valid_rows == 32)
// stores the buffer with one TMA store of that box (tm, column x, row y);
// otherwise lanes 8u .. 8u+7 store the 8 chunks of rows u, u + 4, ... below
// valid_rows, each store instruction four rows x 128 contiguous bytes (out:
// the warp's first row at the round's first column).  The buffer is rewritten
// only after the previous round's TMA store has read it.
__device__ __forceinline__ void store_round(const uint32_t* pk, uint4* stage, int lane, uint16_t* out, long long ldo,
                                            int valid_rows, const CUtensorMap* tm, int x, int y) {
  if (lane == 0) bulk_wait_group_read0();
  __syncwarp();
#pragma unroll
  for (int j = 0; j < 8; ++j)
    stage[lane * 8 + (j ^ (lane & 7))] = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
  if (valid_rows == 32 && tm) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tm, smem_u32(stage), x, y);
      bulk_commit_group();
    }
    return;
  }
  __syncwarp();
  const int ru = lane >> 3, cu = lane & 7;
  uint16_t* dst = out + ru * ldo + cu * 8;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int r = ru + 4 * k;
    const uint4 v = stage[r * 8 + (cu ^ (r & 7))];
    if (r < valid_rows) *reinterpret_cast<uint4*>(dst + 4 * k * ldo) = v;
  }
  __syncwarp();
}

// TMEM -> packed bf16 for 64 output columns starting at output column c0:
// SwiGLU tiles read gate columns c0 .. c0 + 63 and the matching up columns
// BN / 2 further and form silu(g) u; plain tiles read columns c0 .. c0 + 63.
// (16 columns per TMEM wait: 32 or 64 per wait measured the same.)
template <int EPI>
__device__ __forceinline__ void tmem_to_bf16_64(uint32_t taddr, int c0, uint32_t* pk) {
#pragma unroll
  for (int c = 0; c < 64; c += 16) {
    uint32_t g[16];
    tmem_ld16(taddr + c0 + c, g);
    if constexpr (EPI == EPI_SWIGLU) {
      uint32_t u[16];
      tmem_ld16(taddr + BN / 2 + c0 + c, u);
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
        const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
        // silu(g) u with the fast exponential and divide (within a few
        // fp32 ulp, far below h's bf16 rounding)
        pk[c / 2 + i] = pack_bf16x2(__fdividef(g0, 1.0f + __expf(-g0)) * u0, __fdividef(g1, 1.0f + __expf(-g1)) * u1);
      }
    } else {
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 8; ++i) pk[c / 2 + i] = pack_bf16x2(__uint_as_float(g[2 * i]), __uint_as_float(g[2 * i + 1]));
    }
  }
}

// Combine fused into the down GEMM: after a warp has stored its rows of a
// tile (plain stores, so that a fence orders them before the arrivals), each
// stored row adds one arrival to its token slice (token t, 256-column
// n-tile); the arrival that completes a slice (its k routed rows and the
// shared row) has the warp sum it, out[t, slice] = sum_j w[t,j]
// y_perm[perm_dst[t,j], slice] in slot order, then + y_sh[t, slice], rounded
// to bf16: the combine kernel's arithmetic, so the output bits are the
// same.  No wait: the last arrival does the work.
__device__ __forceinline__ void combine_slices(const Tile& T, const GemmArgs& a, long long r0, int lane,
                                               int valid_rows) {
  const int V = static_cast<int>(a.ldo0 / 8);  // 16-byte vectors per row
  const int NT = V / 32;                        // 256-column slices per row
  const int need = a.comb_k + (a.m1 > 0 ? 1 : 0);
  int t = -1;
  if (lane < valid_rows) {
    const long long r = r0 + lane;
    t = T.p1 ? static_cast<int>(r) : __ldg(a.comb_src + r);
    if (t < 0 || t >= a.comb_n) {
      record_status(a.status, ST_BAD_POSITION);
      t = -1;
    }
  }
  __threadfence();  // the warp's row stores (after its last __syncwarp) before the arrivals
  bool last = false;
  if (t >= 0) last = atomicAdd(a.comb_cnt + static_cast<long long>(t) * NT + T.n_tile, 1) == need - 1;
  unsigned m = __ballot_sync(0xffffffffu, last);
  if (!m) return;
  __threadfence();  // the other rows of the completed slices, stored by other CTAs
  const uint4* y = static_cast<const uint4*>(a.out0);
  const uint4* ysh = static_cast<const uint4*>(a.out1);
  uint4* out = static_cast<uint4*>(a.comb_out);
  const int v = T.n_tile * 32 + lane;
  while (m) {
    const int src = __ffs(m) - 1;
    m &= m - 1;
    const int tt = __shfl_sync(0xffffffffu, t, src);
    const long long tk = static_cast<long long>(tt) * a.comb_k;
    int p[kMaxTopK];
    float wj[kMaxTopK];
    uint4 yv[kMaxTopK];
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) {
      p[j] = -1;
      wj[j] = 0.f;
      if (j < a.comb_k) {
        p[j] = __ldcg(a.comb_dst + tk + j);
        wj[j] = __ldg(a.comb_w + tk + j);
        if (p[j] < 0 || p[j] >= a.m0) {
          if (lane == 0) record_status(a.status, ST_BAD_POSITION);
          p[j] = -1;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j)
      if (p[j] >= 0) yv[j] = __ldcg(y + static_cast<long long>(p[j]) * V + v);
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) {
      if (p[j] >= 0) {
        const float w = wj[j];
        acc[0] = fmaf(w, bf16_lo(yv[j].x), acc[0]);
        acc[1] = fmaf(w, bf16_hi(yv[j].x), acc[1]);
        acc[2] = fmaf(w, bf16_lo(yv[j].y), acc[2]);
        acc[3] = fmaf(w, bf16_hi(yv[j].y), acc[3]);
        acc[4] = fmaf(w, bf16_lo(yv[j].z), acc[4]);
        acc[5] = fmaf(w, bf16_hi(yv[j].z), acc[5]);
        acc[6] = fmaf(w, bf16_lo(yv[j].w), acc[6]);
        acc[7] = fmaf(w, bf16_hi(yv[j].w), acc[7]);
      }
    }
    if (a.m1 > 0) {
      const uint4 sv = __ldcg(ysh + static_cast<long long>(tt) * V + v);
      acc[0] += bf16_lo(sv.x);
      acc[1] += bf16_hi(sv.x);
      acc[2] += bf16_lo(sv.y);
      acc[3] += bf16_hi(sv.y);
      acc[4] += bf16_lo(sv.z);
      acc[5] += bf16_hi(sv.z);
      acc[6] += bf16_lo(sv.w);
      acc[7] += bf16_hi(sv.w);
    }
    out[static_cast<long long>(tt) * V + v] = make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]),
                                                         pack_bf16x2(acc[4], acc[5]), pack_bf16x2(acc[6], acc[7]));
  }
}

// Epilogue of one tile for the thread owning TMEM lane ``row`` (taddr: that
// lane, the accumulator's first column); it arrives on ``tempty`` once the
// accumulator has been read.  lanes: the warp's lanes that hold rows (16 for
// an M = 64 accumulator, whose row 16 q + i the thread of lane i reads).  bf16 outputs (SwiGLU: BN / 2 columns, plain: BN)
// are stored in rounds of 64 columns through the warp's staging buffer.
// EARLY (down GEMM with paired tiles, whose accumulator is all of TMEM): the
// whole row is read into registers (packed bf16) and the accumulator handed
// back before any store, so the stores overlap the next tile's main loop
// (measured 1-2 % faster; for the gate/up GEMM it measured no faster and
// spilled).  Otherwise rows are read and stored round by round (single
// m-tiles' two accumulators already overlap the epilogue with the next main
// loop).  The fp32 epilogue (router logits) stores as it reads.  COMB: the
// combine is fused (combine_slices after the tile's stores, which are plain
// stores: tm is nullptr).
template <int EPI, bool EARLY, bool COMB>
__device__ __forceinline__ void epilogue_tile(const Tile& T, const GemmArgs& a, uint32_t taddr, int row,
                                              uint32_t tempty, uint4* stage, int lane, int lanes,
                                              const CUtensorMap* tm) {
  // output row of the tile's row 0; split-K slices of problem 0 write separate planes
  const long long orow_t = static_cast<long long>(T.a_row) + (T.p1 ? 0 : T.split * a.split_rows0);
  if constexpr (EPI == EPI_F32) {
    const bool valid = row < T.rows;
    float* out = static_cast<float*>(T.p1 ? a.out1 : a.out0);
    const long long ldo = T.p1 ? a.ldo1 : a.ldo0;
    float* dst = out + (orow_t + row) * ldo + static_cast<long long>(T.n_tile) * BN;
#pragma unroll 1
    for (int c = 0; c < BN; c += 16) {
      uint32_t v[16];
      tmem_ld16(taddr + c, v);
      tmem_ld_wait();
      if (valid) {
        uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
        for (int i = 0; i < 4; ++i) d4[i] = make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    }
    tc_fence_before();
    mbar_arrive(tempty);
  } else {
    constexpr int kOutCols = EPI == EPI_SWIGLU ? BN / 2 : BN;
    constexpr int kRounds = kOutCols / 64;
    const int wrow0 = row - lane;                      // the warp's first row in the tile
    const int valid_rows = min(T.rows - wrow0, lanes);  // rows of the warp that are stored
    uint16_t* out = static_cast<uint16_t*>(T.p1 ? a.out1 : a.out0);
    const long long ldo = T.p1 ? a.ldo1 : a.ldo0;
    uint16_t* out_w = out + (orow_t + wrow0) * ldo + static_cast<long long>(T.n_tile) * kOutCols;
    // the warp's box origin for the TMA stores: column of the round, row
    const int bx = T.n_tile * kOutCols, by = static_cast<int>(orow_t + wrow0);
    if constexpr (EARLY) {
      uint32_t pk[kRounds * 32];
#pragma unroll
      for (int rd = 0; rd < kRounds; ++rd) tmem_to_bf16_64<EPI>(taddr, 64 * rd, pk + 32 * rd);
      tc_fence_before();
      mbar_arrive(tempty);
#pragma unroll
      for (int rd = 0; rd < kRounds; ++rd)
        store_round(pk + 32 * rd, stage, lane, out_w + 64 * rd, ldo, valid_rows, tm, bx + 64 * rd, by);
      if constexpr (COMB) combine_slices(T, a, orow_t + wrow0, lane, valid_rows);
    } else {
#pragma unroll 1
      for (int rd = 0; rd < kRounds; ++rd) {
        uint32_t pk[32];
        tmem_to_bf16_64<EPI>(taddr, 64 * rd, pk);
        store_round(pk, stage, lane, out_w + 64 * rd, ldo, valid_rows, tm, bx + 64 * rd, by);
      }
      tc_fence_before();
      mbar_arrive(tempty);
      if constexpr (COMB) combine_slices(T, a, orow_t + wrow0, lane, valid_rows);
    }
  }
}

template <int EPI, bool PAIR, bool COMB>
__global__ void __launch_bounds__(Gemm<EPI, PAIR>::kThreads, 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                        const __grid_constant__ CUtensorMap tmO0, const __grid_constant__ CUtensorMap tmO1,
                        const GemmArgs args) {
  using C = Gemm<EPI, PAIR>;
  constexpr int SA = C::SA, SB = C::SB, A_BYTES = C::A_BYTES, BMT = C::BMT;
  static_assert(8 * (2 * SA + 2 * SB + 5) + kTileQBytes + 8 <= kBarBytes, "barrier area");
  static_assert(smem_bytes<EPI, PAIR>() <= 227 * 1024, "shared memory budget");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  if (base & 1023u) {  // uniform for the CTA: nothing is initialised yet
    if (threadIdx.x == 0) record_status(args.status, ST_SMEM_ALIGN);
    return;
  }
  uint8_t* gbase = smem_raw;
  const uint32_t sA = base;
  const uint32_t sB = base + SA * A_BYTES;
  // bf16 store staging, kStageWarpBytes per epilogue warp, right after the
  // rings so that every warp's buffer is 1024-byte aligned (the 128-byte
  // swizzle of its TMA stores); then the barriers and the schedule table
  uint4* stage_all = reinterpret_cast<uint4*>(gbase + SA * A_BYTES + SB * B_BYTES);
  uint8_t* bar_area = gbase + SA * A_BYTES + SB * B_BYTES + stage_bytes<EPI, PAIR>();
  const uint32_t bar0 = smem_u32(bar_area);
  // mbarriers (8 bytes each): fullA[SA], emptyA[SA], fullB[SB], emptyB[SB],
  // tfull[2], tempty[2], drain, tile queue full[kTileQ], empty[kTileQ]
  auto fullA = [&](int s) { return bar0 + 8u * s; };
  auto emptyA = [&](int s) { return bar0 + 8u * (SA + s); };
  auto fullB = [&](int s) { return bar0 + 8u * (2 * SA + s); };
  auto emptyB = [&](int s) { return bar0 + 8u * (2 * SA + SB + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * SA + 2 * SB + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * SA + 2 * SB + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * SA + 2 * SB + 4);
  const uint32_t tq_base = bar0 + 8u * (2 * SA + 2 * SB + 5);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_area + 8 * (2 * SA + 2 * SB + 5) + kTileQBytes);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  Sched* sch = reinterpret_cast<Sched*>(bar_area + kBarBytes);
  // consumers of each queued tile id: A producer, MMA issuer, the epilogue warps
  constexpr int kTileQConsumers = 2 + C::EPI_WARPS;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int G = args.offsets ? args.groups : 1;
  // weight descriptors of this launch's layer (only the B producer reads them)
  const CUtensorMap* tmB0 = nullptr;
  const CUtensorMap* tmB1 = nullptr;

  if (warp == 0) {
    if (lane == 0) {
      const LayerEntry& le =
          args.lref.table[load_layer(args.lref.layer, args.lref.n_layers, args.status, blockIdx.x == 0)];
      tmB0 = &le.map[args.bmap0];
      tmB1 = &le.map[args.bmap1];
      tensormap_acquire(tmB0);
      if (args.m1 > 0) tensormap_acquire(tmB1);
      for (int s = 0; s < SA; ++s) {
        mbar_init(fullA(s), 1);
        mbar_init(emptyA(s), 1);
      }
      for (int s = 0; s < SB; ++s) {
        mbar_init(fullB(s), 1);
        mbar_init(emptyB(s), 1);
      }
      for (int a = 0; a < 2; ++a) {
        mbar_init(tfull_bar(a), 1);
        mbar_init(tempty_bar(a), 32 * C::EPI_WARPS);
      }
      mbar_init(drain_bar, 1);
      TileQueue{tq_base}.init(kTileQConsumers);
      *abort_flag = 0;
      fence_barrier_init();
      tma_prefetch_desc(&tmA0);
      tma_prefetch_desc(tmB0);
      if (args.m1 > 0) {
        tma_prefetch_desc(&tmA1);
        tma_prefetch_desc(tmB1);
      }
    }
    build_schedule<BMT>(args, sch, G, lane);
  } else if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total0 = sch->tile_start[G];
  const int total = total0 + (sch->m1 > 0 ? ((sch->m1 + BMT - 1) / BMT) * args.n_tiles1 : 0);
  TileQueue tq{tq_base};

  if ((warp == 0 || warp == C::kAProdWarp) && lane == 0) {
    // ------------------------------------------------------------ producers
    // warp 0 claims the tiles and streams their weight boxes (B) into its
    // ring, warp 6 the activation boxes (A) into its own; the MMA issuer joins
    // them per k-step.
    const bool isB = warp == 0;
    const int nst = isB ? SB : SA;
    const uint32_t bytes = isB ? B_BYTES : A_BYTES;  // stage stride
    const uint32_t ring = isB ? sB : sA;
    const uint64_t pol = l2_policy(isB ? args.hint_b : args.hint_a);
    int stage = 0;
    uint32_t phase = 0;
    uint32_t pending = 0, issued_phase = 0;  // bit s: stage s has a load in flight
    bool ok = true;
    int t = blockIdx.x;
    while (ok) {
      int cur;
      if (isB) {
        cur = t < total ? t : -1;
        if (!tq.push(cur, abort_flag)) {
          ok = false;
          break;
        }
        if (cur >= 0) t = next_tile(args, cur);  // claimed now, used after this tile's loads
      } else if (!tq.pop(cur, abort_flag, true)) {
        ok = false;
        break;
      }
      if (cur < 0) break;
      Tile T;
      decode_tile<BMT>(cur, sch, G, total0, args, T);
      const CUtensorMap* m = isB ? (T.p1 ? tmB1 : tmB0) : (T.p1 ? &tmA1 : &tmA0);
      const int row = isB ? T.b_row : T.a_row;
      // tile-contiguous weights: box (b_row / BN, kb) is rows ((b_row / BN) k_iters + kb) BN
      const bool tiled = isB && args.b_tiled;
      const long long tile_row0 = static_cast<long long>(row / BN) * (T.p1 ? args.k_iters1 : args.k_iters0);
      // A boxes are 128 rows: a paired tile loads two (rows 128 .. 255 land
      // 128 x 128 bytes further, the layout of one 256-row box), a half tile one
      const bool two = PAIR && !isB && T.rows > BM;
      const uint32_t tx = isB ? B_BYTES : two ? A_BYTES : static_cast<uint32_t>(BM * BK * 2);
      for (int kb = T.kb0; kb < T.kb1; ++kb) {
        const uint32_t full = isB ? fullB(stage) : fullA(stage);
        if (!mbar_wait(isB ? emptyB(stage) : emptyA(stage), phase ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(full, tx);
        if (tiled)
          tma_load_2d(ring + stage * bytes, m, full, 0, static_cast<int>((tile_row0 + kb) * BN), pol);
        else
          tma_load_2d(ring + stage * bytes, m, full, kb * BK, row, pol);
        if (two) tma_load_2d(ring + stage * bytes + BM * BK * 2, m, full, kb * BK, row + BM, pol);
        pending |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == nst) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok) {
      *abort_flag = 1;
      record_status(args.status, ST_WAIT_TIMEOUT);
      // let the copies already issued land before the CTA's memory goes away
      int dummy = 0;
      for (int s = 0; s < nst; ++s)
        if (pending & (1u << s)) mbar_wait(isB ? fullB(s) : fullA(s), (issued_phase >> s) & 1u, &dummy);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    int sa = 0, sb = 0;
    uint32_t pa = 0, pb = 0;
    bool ok = true, issued = false;
    for (int it = 0; ok; ++it) {
      int t;
      if (!tq.pop(t, abort_flag, true)) {
        ok = false;
        break;
      }
      if (t < 0) break;
      Tile T;
      decode_tile<BMT>(t, sch, G, total0, args, T);
      // PAIR: one tile accumulator (both TMEM halves); else ping-pong halves
      const int acc = PAIR ? 0 : (it & 1);
      const uint32_t acc_phase = PAIR ? (it & 1) : ((it >> 1) & 1);
      if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem_base + acc * BN;
      const bool two = PAIR && T.rows > BM;  // else a half tile: the upper MMA is skipped
      // M = 64 for a 128-row half holding at most 64 rows (expert GEMMs)
      const uint32_t id_lo = (EPI != EPI_F32 && T.rows <= kTailRows) ? kIdesc64 : kIdesc;
      const uint32_t id_hi = (EPI != EPI_F32 && T.rows - BM <= kTailRows) ? kIdesc64 : kIdesc;
      for (int kb = T.kb0; kb < T.kb1; ++kb) {
        if (!mbar_wait(fullA(sa), pa, abort_flag) || !mbar_wait(fullB(sb), pb, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_addr = sA + sa * A_BYTES;
        const uint32_t b_addr = sB + sb * B_BYTES;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t adesc = BK == 64 ? smem_desc_sw128(a_addr + kk * 32) : smem_desc_sw64(a_addr + kk * 32);
          const uint64_t bdesc = BK == 64 ? smem_desc_sw128(b_addr + kk * 32) : smem_desc_sw64(b_addr + kk * 32);
          tc_mma_bf16(d, adesc, bdesc, id_lo, (kb > T.kb0 || kk > 0) ? 1u : 0u);
          if (two) {
            // rows 128 .. 255 of the A stage (128 rows x 128 bytes further) into the other half
            const uint32_t a_hi = a_addr + kGemmBM * BK * 2;
            const uint64_t adesc_hi = BK == 64 ? smem_desc_sw128(a_hi + kk * 32) : smem_desc_sw64(a_hi + kk * 32);
            tc_mma_bf16(tmem_base + BN, adesc_hi, bdesc, id_hi, (kb > T.kb0 || kk > 0) ? 1u : 0u);
          }
        }
        issued = true;
        tc_commit(emptyA(sa));
        tc_commit(emptyB(sb));
        if (++sa == SA) {
          sa = 0;
          pa ^= 1u;
        }
        if (++sb == SB) {
          sb = 0;
          pb ^= 1u;
        }
      }
      if (ok) tc_commit(tfull_bar(acc));
    }
    if (!ok) {
      *abort_flag = 1;
      record_status(args.status, ST_WAIT_TIMEOUT);
      if (issued) {
        int dummy = 0;
        tc_commit(drain_bar);
        mbar_wait(drain_bar, 0, &dummy);
      }
    }
  } else if (warp >= 2 && warp < 2 + C::EPI_WARPS) {
    // ------------------------------------------------------------ epilogue
    // warp w reads TMEM lanes 32 (w % 4) ..; with PAIR warps 2-5 take the
    // tile's first 128 rows (TMEM columns 0 ..), warps 6-9 the next 128
    // (columns 256 ..)
    const int q = warp & 3;
    const int half = PAIR ? (warp - 2) >> 2 : 0;
    const int row = half * kGemmBM + q * 32 + lane;
    for (int it = 0;; ++it) {
      int t = -1;
      const uint32_t qslot = tq.slot();
      if (!__all_sync(0xffffffffu, tq.pop(t, abort_flag, false))) {
        if (lane == 0) {
          *abort_flag = 1;
          record_status(args.status, ST_WAIT_TIMEOUT);
        }
        break;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(tq.empty(qslot));
      if (t < 0) break;
      Tile T;
      decode_tile<BMT>(t, sch, G, total0, args, T);
      const int acc = PAIR ? 0 : (it & 1);
      const uint32_t acc_phase = PAIR ? (it & 1) : ((it >> 1) & 1);
      const bool ok = __all_sync(0xffffffffu, mbar_wait(tfull_bar(acc), acc_phase, abort_flag));
      if (!ok) {
        if (lane == 0) {
          *abort_flag = 1;
          record_status(args.status, ST_WAIT_TIMEOUT);
        }
        break;
      }
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + (PAIR ? half : acc) * BN;
      // the upper half of a half tile holds no rows (and no result)
      if (half == 0 || T.rows > BM) {
        // an M = 64 half (at most 64 rows): row 16 q + lane in lanes 0-15
        const int half_rows = half == 0 ? min(T.rows, BM) : T.rows - BM;
        const bool m64 = EPI != EPI_F32 && half_rows <= kTailRows;
        const int erow = m64 ? half * kGemmBM + q * 16 + lane : row;
        // arrives on tempty itself
        epilogue_tile<EPI, PAIR && EPI == EPI_BF16, COMB>(T, args, taddr, erow, tempty_bar(acc),
                                                          stage_all + (warp - 2) * (kStageWarpBytes / 16), lane,
                                                          m64 ? 16 : 32, COMB ? nullptr : (T.p1 ? &tmO1 : &tmO0));
      } else {
        tc_fence_before();
        mbar_arrive(tempty_bar(acc));
      }
    }
    // the warp's TMA stores are complete before its staging buffer goes away
    if (lane == 0) bulk_wait_group0();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

template <int EPI, bool PAIR, bool COMB = false>
cudaError_t set_attr() {
  return cudaFuncSetAttribute(grouped_gemm_kernel<EPI, PAIR, COMB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem_bytes<EPI, PAIR>()));
}

template <int EPI, bool PAIR, bool COMB = false>
void launch(const CUtensorMap* maps, const GemmArgs& args, int grid, cudaStream_t stream) {
  grouped_gemm_kernel<EPI, PAIR, COMB>
      <<<dim3(grid), dim3(Gemm<EPI, PAIR>::kThreads), smem_bytes<EPI, PAIR>(), stream>>>(maps[0], maps[1], maps[2],
                                                                                        maps[3], args);
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                              CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                              CUtensorMapFloatOOBfill);

EncodeFn get_encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

}  // namespace

static_assert(sizeof(Sched) + 0 <= 8192, "schedule table");

cudaError_t gemm_set_attributes() {
  cudaError_t e = set_attr<EPI_SWIGLU, false>();
  if (e == cudaSuccess) e = set_attr<EPI_SWIGLU, true>();
  if (e == cudaSuccess) e = set_attr<EPI_BF16, false>();
  if (e == cudaSuccess) e = set_attr<EPI_BF16, true>();
  if (e == cudaSuccess) e = set_attr<EPI_BF16, false, true>();
  if (e == cudaSuccess) e = set_attr<EPI_BF16, true, true>();
  if (e == cudaSuccess) e = set_attr<EPI_F32, false>();
  return e;
}

cudaError_t gemm_launch(int epi, bool pair, const CUtensorMap* maps, const GemmArgs& args, int grid,
                        cudaStream_t stream) {
  if (grid <= 0) return cudaSuccess;
  if (epi == EPI_SWIGLU) {
    if (pair) launch<EPI_SWIGLU, true>(maps, args, grid, stream);
    else launch<EPI_SWIGLU, false>(maps, args, grid, stream);
  } else if (epi == EPI_BF16) {
    if (args.comb_cnt) {
      if (pair) launch<EPI_BF16, true, true>(maps, args, grid, stream);
      else launch<EPI_BF16, false, true>(maps, args, grid, stream);
    } else if (pair) {
      launch<EPI_BF16, true>(maps, args, grid, stream);
    } else {
      launch<EPI_BF16, false>(maps, args, grid, stream);
    }
  } else {
    if (pair) return cudaErrorInvalidValue;
    launch<EPI_F32, false>(maps, args, grid, stream);
  }
  return cudaGetLastError();
}

bool encode_tmap_bf16(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols,
                      uint32_t box_rows, std::string* err) {
  EncodeFn fn = get_encode_fn();
  if (!fn) {
    if (err) *err = "cuTensorMapEncodeTiled is not available from the driver";
    return false;
  }
  if ((reinterpret_cast<uintptr_t>(ptr) & 15u) != 0 || (cols * 2) % 16 != 0 || rows == 0) {
    if (err) *err = "tensor for TMA must be 16-byte aligned with 16-byte row stride and >= 1 row";
    return false;
  }
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        BK == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (err) *err = "cuTensorMapEncodeTiled failed with CUresult " + std::to_string(static_cast<int>(r));
    return false;
  }
  return true;
}

}  // namespace asap
