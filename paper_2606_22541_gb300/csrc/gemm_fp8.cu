// Grouped GEMM with e4m3 operands and fp32 block scales on the sm_103a
// tensor core (tcgen05.mma kind::f8f6f4), fed by TMA.
//
// The FP8 configuration of the MoE layer stores expert weights as e4m3 with
// one fp32 scale per 128 x 128 block and quantises activations per token per
// 128 channels.  The scales are arbitrary fp32 values, so they cannot ride
// in the tensor core's power-of-two block-scale path; instead every 128-wide
// K block is multiplied into one of two TMEM partial buffers (ping-pong) and
// the epilogue warps add it, times (row scale x block scale), into fp32
// register accumulators while the tensor core already works on the next
// block.  The per-row and per-block scales of the next two K blocks are
// loaded ahead, so their L2 latency stays off the promotion path.
//
// Roles (one CTA per SM, persistent, 352 threads):
//   warp 0    : weight producer, boxes [256 rows, 128 B], 4-stage ring
//   last warp : activation producer, boxes [128 rows, 128 B], 4-stage ring
//   warp 1    : TMEM allocator (512 columns) and MMA issuer: per K block
//               4 x tcgen05.mma.cta_group::1.kind::f8f6f4 M=128 N=256 K=32
//   epilogue  : 8 warps; warp w owns TMEM lanes 32*(w%4).. and, with
//               cq = (w-2)/4, one half of the 256 columns of a tile
// Tile schedule, masking and bounded waits as in the bf16 kernel.
#include "common.cuh"
#include "gemm_sched.cuh"
#include "internal.h"

#include <cuda_fp8.h>

#include <mutex>

namespace asap {

namespace {

constexpr int BM = kGemmBM, BN = kGemmBN, BK = kFp8BK;
constexpr int SA = 4, SB = 4;
constexpr int A_BYTES = BM * BK;  // 16 KB
constexpr int B_BYTES = BN * BK;  // 32 KB
#ifndef ASAP_FP8_EPI_WARPS
#define ASAP_FP8_EPI_WARPS 8
#endif
constexpr int kEpiWarps = ASAP_FP8_EPI_WARPS;   // 8 or 16: 2 or 4 per TMEM lane quarter
constexpr int kColGroups = kEpiWarps / 4;       // column groups per row
constexpr int kCols = BN / kColGroups;          // accumulator columns per thread
constexpr int kThreads = 32 * (3 + kEpiWarps);
constexpr int kAProdWarp = 2 + kEpiWarps;
constexpr uint32_t kTmemCols = 2 * BN;          // two partial buffers
// kind::f8f6f4: fp32 accumulator (bits 4-5 = 1), A and B e4m3 (format 0),
// both K-major, N >> 3 in bits 17-22, M >> 4 in bits 24-28.
constexpr uint32_t kIdescF8 = (1u << 4) | (static_cast<uint32_t>(BN >> 3) << 17) | (static_cast<uint32_t>(BM >> 4) << 24);

constexpr int kBarBytes = 384;
// outputs are stored through 2 KB of shared memory per epilogue warp (32 rows x 4 chunks of 16 bytes)
constexpr int kStageWarpBytes = 32 * 4 * 16;
// rings first (1024-byte aligned, declared and checked), then barriers, store
// staging, schedule, amax exchange
constexpr size_t kSmemBytes = SA * A_BYTES + SB * B_BYTES + kBarBytes + kEpiWarps * kStageWarpBytes + sizeof(Sched) +
                              2 * 4 * BM * sizeof(float);
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
static_assert(8 * (2 * SA + 2 * SB + 7) + kTileQBytes + 12 <= kBarBytes, "barrier area");
// consumers of each queued tile id: A producer, MMA issuer, the epilogue warps
constexpr int kTileQConsumers = 2 + kEpiWarps;

__device__ __forceinline__ void tc_mma_f8(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(kIdescF8), "r"(accumulate)
      : "memory");
}

#ifndef ASAP_FP8_PROMOTE
#define ASAP_FP8_PROMOTE 16
#endif
// acc[j] += s * partial[j] for 32 consecutive TMEM columns
__device__ __forceinline__ void promote32(float* acc, uint32_t taddr, float s) {
  if constexpr (ASAP_FP8_PROMOTE == 32) {
    uint32_t v[32];
    tmem_ld32(taddr, v);
    tmem_ld_wait();
#pragma unroll
    for (int j = 0; j < 32; ++j) acc[j] = fmaf(s, __uint_as_float(v[j]), acc[j]);
  } else {
#pragma unroll
    for (int c = 0; c < 32; c += 16) {
      uint32_t v[16];
      tmem_ld16(taddr + c, v);
      tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < 16; ++j) acc[c + j] = fmaf(s, __uint_as_float(v[j]), acc[c + j]);
    }
  }
}

// One round of a warp's coalesced stores: lane l holds 4 chunks of 16 bytes
// (w, 16 words) of its row l.  Every lane writes them to the warp's 2 KB
// staging buffer (chunk j of row r at slot j ^ ((r / 2) % 4), so neither side
// of the exchange has bank conflicts), then lanes 4u .. 4u+3 store the 4
// chunks of rows u, u + 8, ...: each store instruction writes eight rows x 64
// contiguous bytes instead of 32 rows x 16 bytes.  Rows from ``valid_rows`` on
// are not stored.  out: the warp's first row at the round's first byte.
__device__ __forceinline__ void store_round4(const uint32_t* w, uint4* stage, int lane, uint8_t* out,
                                             long long ldo_bytes, int valid_rows) {
#pragma unroll
  for (int j = 0; j < 4; ++j)
    stage[lane * 4 + (j ^ ((lane >> 1) & 3))] = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
  __syncwarp();
  const int ru = lane >> 2, cu = lane & 3;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int r = ru + 8 * k;
    const uint4 v = stage[r * 4 + (cu ^ ((r >> 1) & 3))];
    if (r < valid_rows) *reinterpret_cast<uint4*>(out + r * ldo_bytes + cu * 16) = v;
  }
  __syncwarp();
}

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    grouped_gemm_fp8_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                            const Fp8Args fa) {
  const GemmArgs& args = fa.g;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  if (base & 1023u) {  // uniform for the CTA: nothing is initialised yet
    if (threadIdx.x == 0) record_status(args.status, ST_SMEM_ALIGN);
    return;
  }
  uint8_t* gbase = smem_raw;
  const uint32_t sA = base;
  const uint32_t sB = base + SA * A_BYTES;
  uint8_t* bar_area = gbase + SA * A_BYTES + SB * B_BYTES;
  const uint32_t bar0 = smem_u32(bar_area);
  auto fullA = [&](int s) { return bar0 + 8u * s; };
  auto emptyA = [&](int s) { return bar0 + 8u * (SA + s); };
  auto fullB = [&](int s) { return bar0 + 8u * (2 * SA + s); };
  auto emptyB = [&](int s) { return bar0 + 8u * (2 * SA + SB + s); };
  auto pfull = [&](int b) { return bar0 + 8u * (2 * SA + 2 * SB + b); };
  auto pempty = [&](int b) { return bar0 + 8u * (2 * SA + 2 * SB + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * SA + 2 * SB + 4);
  // amax exchange between the two epilogue halves of a row (per tile parity)
  auto xchg = [&](int b) { return bar0 + 8u * (2 * SA + 2 * SB + 5 + b); };
  const uint32_t tq_base = bar0 + 8u * (2 * SA + 2 * SB + 7);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_area + 8 * (2 * SA + 2 * SB + 7) + kTileQBytes);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* layer_slot = reinterpret_cast<int*>(tmem_slot + 2);  // layer id, shared with the epilogue
  uint4* stage_all = reinterpret_cast<uint4*>(bar_area + kBarBytes);  // 16-byte aligned
  Sched* sch = reinterpret_cast<Sched*>(bar_area + kBarBytes + kEpiWarps * kStageWarpBytes);
  float* amax_x = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(sch) + sizeof(Sched));  // [2][4][BM]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int G = args.offsets ? args.groups : 1;
  // weight descriptors of this launch's layer (read by the B producer)
  const CUtensorMap* tmB0 = nullptr;
  const CUtensorMap* tmB1 = nullptr;

  if (warp == 0) {
    if (lane == 0) {
      const int l = load_layer(args.lref.layer, args.lref.n_layers, args.status, blockIdx.x == 0);
      *layer_slot = l;
      tmB0 = &args.lref.table[l].map[args.bmap0];
      tmB1 = &args.lref.table[l].map[args.bmap1];
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
      for (int b = 0; b < 2; ++b) {
        mbar_init(pfull(b), 1);
        mbar_init(pempty(b), kEpiWarps * 32);
      }
      mbar_init(drain_bar, 1);
      mbar_init(xchg(0), kEpiWarps * 32);
      mbar_init(xchg(1), kEpiWarps * 32);
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
    build_schedule(args, sch, G, lane);
  } else if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total0 = sch->tile_start[G];
  const int total = total0 + (sch->m1 > 0 ? ((sch->m1 + BM - 1) / BM) * args.n_tiles1 : 0);
  TileQueue tq{tq_base};

  if ((warp == 0 || warp == kAProdWarp) && lane == 0) {
    // ------------------------------------------------------------ producers
    const bool isB = warp == 0;
    const uint32_t bytes = isB ? B_BYTES : A_BYTES;
    const uint32_t ring = isB ? sB : sA;
    const int nst = isB ? SB : SA;
    const uint64_t pol = l2_policy(isB ? args.hint_b : args.hint_a);
    int stage = 0;
    uint32_t phase = 0;
    uint32_t pending = 0, issued_phase = 0;
    bool ok = true;
    int t = blockIdx.x;
    while (ok) {
      int cur;
      if (isB) {  // warp 0 claims the tiles
        cur = t < total ? t : -1;
        if (!tq.push(cur, abort_flag)) {
          ok = false;
          break;
        }
        if (cur >= 0) t = next_tile(args, cur);
      } else if (!tq.pop(cur, abort_flag, true)) {
        ok = false;
        break;
      }
      if (cur < 0) break;
      Tile T;
      decode_tile(cur, sch, G, total0, args, T);
      const CUtensorMap* m = isB ? (T.p1 ? tmB1 : tmB0) : (T.p1 ? &tmA1 : &tmA0);
      const int row = isB ? T.b_row : T.a_row;
      // tile-contiguous weights: box (b_row / BN, kb) is rows ((b_row / BN) k_iters + kb) BN
      const bool tiled = isB && args.b_tiled;
      const long long tile_row0 = static_cast<long long>(row / BN) * (T.p1 ? args.k_iters1 : args.k_iters0);
      for (int kb = T.kb0; kb < T.kb1; ++kb) {
        const uint32_t full = isB ? fullB(stage) : fullA(stage);
        if (!mbar_wait(isB ? emptyB(stage) : emptyA(stage), phase ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(full, bytes);
        if (tiled)
          tma_load_2d(ring + stage * bytes, m, full, 0, static_cast<int>((tile_row0 + kb) * BN), pol);
        else
          tma_load_2d(ring + stage * bytes, m, full, kb * BK, row, pol);
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
      int dummy = 0;
      for (int s = 0; s < nst; ++s)
        if (pending & (1u << s)) mbar_wait(isB ? fullB(s) : fullA(s), (issued_phase >> s) & 1u, &dummy);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    int sa = 0, sb = 0;
    uint32_t pa = 0, pb = 0;
    uint32_t kc = 0;  // K blocks issued by this CTA (partial-buffer ping-pong)
    bool ok = true, issued = false;
    while (ok) {
      int t;
      if (!tq.pop(t, abort_flag, true)) {
        ok = false;
        break;
      }
      if (t < 0) break;
      Tile T;
      decode_tile(t, sch, G, total0, args, T);
      for (int kb = T.kb0; kb < T.kb1; ++kb, ++kc) {
        const int buf = kc & 1;
        if (!mbar_wait(pempty(buf), ((kc >> 1) & 1) ^ 1u, abort_flag) || !mbar_wait(fullA(sa), pa, abort_flag) ||
            !mbar_wait(fullB(sb), pb, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_addr = sA + sa * A_BYTES;
        const uint32_t b_addr = sB + sb * B_BYTES;
        const uint32_t d = tmem_base + buf * BN;
#pragma unroll
        for (int kk = 0; kk < BK / 32; ++kk)
          tc_mma_f8(d, smem_desc_sw128(a_addr + kk * 32), smem_desc_sw128(b_addr + kk * 32), kk > 0 ? 1u : 0u);
        issued = true;
        tc_commit(emptyA(sa));
        tc_commit(emptyB(sb));
        tc_commit(pfull(buf));
        if (++sa == SA) {
          sa = 0;
          pa ^= 1u;
        }
        if (++sb == SB) {
          sb = 0;
          pb ^= 1u;
        }
      }
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
  } else if (warp >= 2 && warp < 2 + kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    // warp w reads TMEM lanes 32*(w%4).. (rows) and column quarter cq:
    // SwiGLU tiles: gate columns [32cq, 32cq+32) and the matching up columns
    // 128 + [32cq, 32cq+32), i.e. h channels [32cq, 32cq+32) of the tile;
    // plain tiles: columns [64cq, 64cq+64).
    const int q = warp & 3;
    const int cq = (warp - 2) >> 2;  // column group
    const int r = q * 32 + lane;
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    uint32_t kc = 0;
    bool ok = true;
    for (int it = 0; ok; ++it) {
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
      decode_tile(t, sch, G, total0, args, T);
      const int mrows = T.p1 ? sch->m1 : args.m0;
      const long long row = static_cast<long long>(T.a_row) + r;
      const long long srow = row < mrows ? row : mrows - 1;  // in-bounds scale row for masked rows
      const int asld = T.p1 ? fa.a_sld1 : fa.a_sld0;
      const float* arow = (T.p1 ? fa.a_scale1 : fa.a_scale0) + srow * asld;
      const int nblk = T.p1 ? fa.b_nblk1 : fa.b_nblk0;
      // B scales of this layer (looked up per tile: no registers held across tiles)
      const float* bs = args.lref.table[*layer_slot].scale[T.p1 ? args.bmap1 : args.bmap0] +
                        static_cast<long long>(T.group) * nblk * asld;
      // scale rows of this warp's columns: SwiGLU tiles hold gate block nt
      // (scale row 2nt) and up block nt (2nt+1); plain tiles blocks 2nt, 2nt+1
      const int lo_blk = EPI == EPI_SWIGLU ? 0 : (cq * kCols) / 128;
      const float* bs_lo = bs + static_cast<long long>(2 * T.n_tile + lo_blk) * asld;
      const float* bs_hi = bs + static_cast<long long>(2 * T.n_tile + 1) * asld;
      // scales of the next two K blocks are loaded ahead (L2 latency)
      auto ld_scales = [&](int kb, float& a, float& bl, float& bh) {
        if (kb < T.kb1) {
          a = __ldg(arow + kb);
          bl = __ldg(bs_lo + kb);
          bh = EPI == EPI_SWIGLU ? __ldg(bs_hi + kb) : 0.f;
        }
      };
      float a0 = 0.f, l0 = 0.f, h0 = 0.f, a1 = 0.f, l1 = 0.f, h1 = 0.f;
      ld_scales(T.kb0, a0, l0, h0);
      ld_scales(T.kb0 + 1, a1, l1, h1);

      float acc[kCols];
#pragma unroll
      for (int j = 0; j < kCols; ++j) acc[j] = 0.f;
      for (int kb = T.kb0; kb < T.kb1; ++kb, ++kc) {
        const int buf = kc & 1;
        const float s_lo = a0 * l0;
        const float s_hi = a0 * h0;
        a0 = a1;
        l0 = l1;
        h0 = h1;
        ld_scales(kb + 2, a1, l1, h1);
        if (!__all_sync(0xffffffffu, mbar_wait(pfull(buf), (kc >> 1) & 1, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t pb = lane_addr + buf * BN;
        if constexpr (EPI == EPI_SWIGLU) {
          // h channels [cq*kCols/2, +kCols/2): gate columns, then the matching up columns
#pragma unroll
          for (int c = 0; c < kCols / 2; c += 32) promote32(acc + c, pb + cq * (kCols / 2) + c, s_lo);
#pragma unroll
          for (int c = 0; c < kCols / 2; c += 32)
            promote32(acc + kCols / 2 + c, pb + 128 + cq * (kCols / 2) + c, s_hi);
        } else {
#pragma unroll
          for (int c = 0; c < kCols; c += 32) promote32(acc + c, pb + cq * kCols + c, s_lo);
        }
        tc_fence_before();
        mbar_arrive(pempty(buf));
      }
      if (!ok) break;
      const bool valid = r < T.rows;
      uint4* stage = stage_all + (warp - 2) * (kStageWarpBytes / 16);
      const int valid_rows = T.rows - q * 32;  // rows of this warp (rows q*32 .. q*32+31) that are stored
      const long long wrow0 = static_cast<long long>(T.a_row) + q * 32;
      if constexpr (EPI == EPI_SWIGLU) {
        // h = silu(gate) * up for 32 channels, then e4m3 with one scale per
        // row per 128 channels (this tile's 128 h columns): the four column
        // quarters of a row exchange their partial amax through shared memory
        constexpr int kH = kCols / 2;  // h channels per thread
        float amax = 0.f;
#pragma unroll
        for (int j = 0; j < kH; ++j) {
          const float gv = acc[j];
          const float hv = __fdividef(gv, 1.0f + __expf(-gv)) * acc[kH + j];
          acc[j] = hv;
          amax = fmaxf(amax, fabsf(hv));
        }
        float* xs = amax_x + (it & 1) * 4 * BM;
        xs[cq * BM + r] = amax;
        mbar_arrive(xchg(it & 1));
        if (!__all_sync(0xffffffffu, mbar_wait(xchg(it & 1), (it >> 1) & 1, abort_flag))) {
          ok = false;
          break;
        }
#pragma unroll
        for (int u = 0; u < kColGroups; ++u) amax = fmaxf(amax, xs[u * BM + r]);
        const float scale = amax > 0.f ? amax / 448.0f : 1.0f;
        const float inv = 1.0f / scale;  // one division; the quotients below are products
        // kH = 64 e4m3 values: 4 chunks of 16 bytes, one staged round
        static_assert(kH == 64, "one store round of e4m3 h per thread");
        uint32_t w[16];
#pragma unroll
        for (int j = 0; j < kH; j += 4) {
          const __nv_fp8x2_storage_t lo = __nv_cvt_float2_to_fp8x2(make_float2(acc[j] * inv, acc[j + 1] * inv),
                                                                    __NV_SATFINITE, __NV_E4M3);
          const __nv_fp8x2_storage_t hi = __nv_cvt_float2_to_fp8x2(make_float2(acc[j + 2] * inv, acc[j + 3] * inv),
                                                                    __NV_SATFINITE, __NV_E4M3);
          w[j / 4] = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
        }
        uint8_t* out = static_cast<uint8_t*>(T.p1 ? args.out1 : args.out0);
        const long long ldo = T.p1 ? args.ldo1 : args.ldo0;
        store_round4(w, stage, lane, out + wrow0 * ldo + static_cast<long long>(T.n_tile) * (BN / 2) + cq * kH, ldo,
                     valid_rows);
        if (valid && cq == 0) {
          float* os = T.p1 ? fa.out_scale1 : fa.out_scale0;
          const int osld = T.p1 ? fa.o_sld1 : fa.o_sld0;
          os[row * osld + T.n_tile] = scale;
        }
      } else {
        // kCols = 128 bf16 values: 16 chunks, four staged rounds of 64 bytes
        uint8_t* out = static_cast<uint8_t*>(T.p1 ? args.out1 : args.out0);
        const long long ldo_b = 2 * (T.p1 ? args.ldo1 : args.ldo0);
        uint8_t* out_w = out + wrow0 * ldo_b + 2 * (static_cast<long long>(T.n_tile) * BN + cq * kCols);
#pragma unroll
        for (int rd = 0; rd < kCols / 32; ++rd) {
          uint32_t w[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) w[i] = pack_bf16x2(acc[32 * rd + 2 * i], acc[32 * rd + 2 * i + 1]);
          store_round4(w, stage, lane, out_w + 64 * rd, ldo_b, valid_rows);
        }
      }
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      record_status(args.status, ST_WAIT_TIMEOUT);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
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

cudaError_t fp8_gemm_set_attributes() {
  cudaError_t e = cudaFuncSetAttribute(grouped_gemm_fp8_kernel<EPI_SWIGLU>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kSmemBytes));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(grouped_gemm_fp8_kernel<EPI_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kSmemBytes));
  return e;
}

cudaError_t fp8_gemm_launch(int epi, const CUtensorMap* maps, const Fp8Args& args, int grid, cudaStream_t stream) {
  if (grid <= 0) return cudaSuccess;
  if (epi == EPI_SWIGLU)
    grouped_gemm_fp8_kernel<EPI_SWIGLU><<<grid, kThreads, kSmemBytes, stream>>>(maps[0], maps[1], args);
  else
    grouped_gemm_fp8_kernel<EPI_BF16><<<grid, kThreads, kSmemBytes, stream>>>(maps[0], maps[1], args);
  return cudaGetLastError();
}

bool encode_tmap_u8(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                    std::string* err) {
  EncodeFn fn = encode_fn();
  if (!fn) {
    if (err) *err = "cuTensorMapEncodeTiled is not available from the driver";
    return false;
  }
  if ((reinterpret_cast<uintptr_t>(ptr) & 15u) != 0 || cols % 16 != 0 || rows == 0) {
    if (err) *err = "tensor for TMA must be 16-byte aligned with 16-byte row stride and >= 1 row";
    return false;
  }
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (err) *err = "cuTensorMapEncodeTiled failed with CUresult " + std::to_string(static_cast<int>(r));
    return false;
  }
  return true;
}

}  // namespace asap
