// Tile scheduler shared by the grouped GEMM kernels: the tile list of a
// launch is derived on the device from the per-group row offsets (expert
// segments), so the host never reads the per-expert counts back.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace asap {

// Per-group tile starts and row segments of problem 0 (group g: rows
// [row_base[g], row_base[g+1]), tiles [tile_start[g], tile_start[g+1])).
struct Sched {
  int tile_start[kMaxExperts + 1];
  int row_base[kMaxExperts + 1];
  int m1;  // rows of problem 1 in this launch (args.m1, or *args.m1_dev clamped to [0, args.m1])
};

struct Tile {
  int a_row, b_row, rows, n_tile, kb0, kb1, split, group;
  bool p1;
};

// ------------------------------------------------------------ tile queue
// Which tiles a CTA computes is decided while the launch runs: the B producer
// takes tile blockIdx.x first, then claims the next unclaimed tile from a
// global counter (args.tile_counter, zero when the launch starts; without one
// the order is static, blockIdx.x + i * gridDim.x).  A CTA that starts late
// because its SM was busy with another kernel then simply takes fewer tiles,
// instead of running its share after everyone else.  Claimed ids reach the
// other roles of the CTA through a ring of kTileQ shared-memory slots guarded
// by mbarriers; id -1 ends every role's loop.
constexpr int kTileQ = 4;
// Shared-memory bytes of the queue: kTileQ full and kTileQ empty mbarriers,
// then kTileQ int slots.
constexpr int kTileQBytes = 20 * kTileQ;

struct TileQueue {
  uint32_t full0;  // shared address of the queue (8-byte aligned)
  uint32_t n = 0;  // ids this thread has pushed or popped

  __device__ __forceinline__ uint32_t slot() const { return n % kTileQ; }
  __device__ __forceinline__ uint32_t phase() const { return (n / kTileQ) & 1u; }
  __device__ __forceinline__ uint32_t full(uint32_t s) const { return full0 + 8u * s; }
  __device__ __forceinline__ uint32_t empty(uint32_t s) const { return full0 + 8u * (kTileQ + s); }
  __device__ __forceinline__ uint32_t id_addr(uint32_t s) const { return full0 + 16u * kTileQ + 4u * s; }

  __device__ __forceinline__ void init(int consumers) const {
    for (uint32_t s = 0; s < kTileQ; ++s) {
      mbar_init(full(s), 1);
      mbar_init(empty(s), consumers);
    }
  }
  // producer: publish the next tile id (or -1)
  __device__ __forceinline__ bool push(int t, volatile int* abort_flag) {
    const uint32_t s = slot();
    if (!mbar_wait(empty(s), phase() ^ 1u, abort_flag)) return false;
    asm volatile("st.shared.b32 [%0], %1;" ::"r"(id_addr(s)), "r"(t) : "memory");
    mbar_arrive(full(s));
    ++n;
    return true;
  }
  // consumer: read the next tile id; ``release`` arrives on the slot's empty
  // barrier (one arrival per consuming thread or warp, as initialised)
  __device__ __forceinline__ bool pop(int& t, volatile int* abort_flag, bool release) {
    const uint32_t s = slot();
    if (!mbar_wait(full(s), phase(), abort_flag)) return false;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(t) : "r"(id_addr(s)) : "memory");
    if (release) mbar_arrive(empty(s));
    ++n;
    return true;
  }
};

// The tile after t for this CTA.
__device__ __forceinline__ int next_tile(const GemmArgs& a, int t) {
  return a.tile_counter ? static_cast<int>(gridDim.x) + atomicAdd(a.tile_counter, 1) : t + static_cast<int>(gridDim.x);
}

// Tile t of the launch: problem 0 groups in order (inside a group: K slice,
// then n-tile, then m-tile innermost), then problem 1 (n-tile, m-tile).
// Tiles are BMT rows high.
template <int BMT = kGemmBM>
__device__ __forceinline__ void decode_tile(int t, const Sched* s, int G, int total0,
                                            const GemmArgs& a, Tile& T) {
  if (t < total0) {
    int lo = 0, hi = G;  // largest g with tile_start[g] <= t
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (s->tile_start[mid] <= t) lo = mid; else hi = mid;
    }
    const int g = lo;
    int local = t - s->tile_start[g];
    const int r0 = s->row_base[g];
    const int mrows = s->row_base[g + 1] - r0;
    const int mt = (mrows + BMT - 1) / BMT;
    const int per_split = mt * a.n_tiles0;
    const int split = local / per_split;   // K slice (split-K of problem 0)
    local -= split * per_split;
    const int nt = local / mt;
    const int mi = local - nt * mt;
    T.a_row = r0 + mi * BMT;
    T.rows = min(BMT, mrows - mi * BMT);
    T.b_row = g * a.b_stride0 + nt * kGemmBN;
    T.n_tile = nt;
    T.split = split;
    T.group = g;
    T.kb0 = static_cast<int>(static_cast<long long>(a.k_iters0) * split / a.k_splits);
    T.kb1 = static_cast<int>(static_cast<long long>(a.k_iters0) * (split + 1) / a.k_splits);
    T.p1 = false;
  } else {
    const int u = t - total0;
    const int mt = (s->m1 + BMT - 1) / BMT;
    const int nt = u / mt;
    const int mi = u - nt * mt;
    T.a_row = mi * BMT;
    T.rows = min(BMT, s->m1 - mi * BMT);
    T.b_row = nt * kGemmBN;
    T.n_tile = nt;
    T.split = 0;
    T.group = 0;
    T.kb0 = 0;
    T.kb1 = a.k_iters1;
    T.p1 = true;
  }
}

// Warp-level construction of the schedule table (called by one full warp):
// per-group counts of BMT-row m-tiles and their exclusive prefix; each lane owns up to 8
// consecutive groups.  Offsets that are negative, not monotone or run past
// the rows are reported in the status word and leave problem 0 empty.
template <int BMT = kGemmBM>
__device__ __forceinline__ void build_schedule(const GemmArgs& args, Sched* sch, int G, int lane) {
  if (lane == 0) sch->m1 = args.m1_dev ? min(max(__ldg(args.m1_dev), 0), args.m1) : args.m1;
  int local = 0;
  int cnt[8];
  int lo[8];
  bool bad = false;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int g = lane * 8 + i;
    cnt[i] = 0;
    lo[i] = 0;
    if (g < G) {
      int m = args.m0;
      if (args.offsets) {
        lo[i] = __ldg(args.offsets + g);
        const int hi = __ldg(args.offsets + g + 1);
        m = hi - lo[i];
        bad |= lo[i] < 0 || m < 0 || hi > args.m0;
      }
      cnt[i] = (max(m, 0) + BMT - 1) / BMT;
      local += cnt[i] * args.n_tiles0 * args.k_splits;
    }
  }
  if (__any_sync(0xffffffffu, bad)) {
    if (lane == 0) record_status(args.status, ST_BAD_OFFSETS);
    for (int g = lane; g <= G; g += 32) {
      sch->tile_start[g] = 0;
      sch->row_base[g] = 0;
    }
    return;
  }
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  int run = incl - local;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int g = lane * 8 + i;
    if (g < G) {
      sch->tile_start[g] = run;
      sch->row_base[g] = lo[i];
      run += cnt[i] * args.n_tiles0 * args.k_splits;
    }
  }
  if (lane == 31) {
    sch->tile_start[G] = incl;
    sch->row_base[G] = args.offsets ? __ldg(args.offsets + G) : args.m0;
  }
}

}  // namespace asap
