// Tile scheduler shared by the grouped GEMM kernels: the tile list of a
// launch is derived on the device from the per-group row offsets (expert
// segments), so the host never reads the per-expert counts back.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace asap {

struct Sched {
  int tile_start[kMaxExperts + 1];
  int mtiles[kMaxExperts];
  int row_base[kMaxExperts];
  int mrows[kMaxExperts];
};

struct Tile {
  int a_row, b_row, rows, n_tile, kb0, kb1, split, group;
  bool p1;
};

// Tile t of the launch: problem 0 groups in order (inside a group: K slice,
// then n-tile, then m-tile innermost), then problem 1 (n-tile, m-tile).
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
    const int mt = s->mtiles[g];
    const int per_split = mt * a.n_tiles0;
    const int split = local / per_split;   // K slice (split-K of problem 0)
    local -= split * per_split;
    const int nt = local / mt;
    const int mi = local - nt * mt;
    T.a_row = s->row_base[g] + mi * kGemmBM;
    T.rows = min(kGemmBM, s->mrows[g] - mi * kGemmBM);
    T.b_row = g * a.b_stride0 + nt * kGemmBN;
    T.n_tile = nt;
    T.split = split;
    T.group = g;
    T.kb0 = static_cast<int>(static_cast<long long>(a.k_iters0) * split / a.k_splits);
    T.kb1 = static_cast<int>(static_cast<long long>(a.k_iters0) * (split + 1) / a.k_splits);
    T.p1 = false;
  } else {
    const int u = t - total0;
    const int mt = (a.m1 + kGemmBM - 1) / kGemmBM;
    const int nt = u / mt;
    const int mi = u - nt * mt;
    T.a_row = mi * kGemmBM;
    T.rows = min(kGemmBM, a.m1 - mi * kGemmBM);
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
// per-group m-tile counts and their exclusive prefix; each lane owns up to 8
// consecutive groups.  Offsets that are not monotone or run past the rows
// make the group empty and are reported in the status word.
__device__ __forceinline__ void build_schedule(const GemmArgs& args, Sched* sch, int G, int lane) {
    // Per-group m-tile counts and their exclusive prefix (warp scan; each
    // lane owns up to 8 consecutive groups).  Bad offsets -> empty group.
    int local = 0;
    int cnt[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int g = lane * 8 + i;
      cnt[i] = 0;
      if (g < G) {
        int lo = 0, m = args.m0;
        if (args.offsets) {
          lo = __ldg(args.offsets + g);
          const int hi = __ldg(args.offsets + g + 1);
          m = hi - lo;
          if (lo < 0 || m < 0 || hi > args.m0) {
            record_status(args.status, ST_BAD_OFFSETS);
            lo = 0;
            m = 0;
          }
        }
        sch->row_base[g] = lo;
        sch->mrows[g] = m;
        cnt[i] = (m + kGemmBM - 1) / kGemmBM;
        sch->mtiles[g] = cnt[i];
        local += cnt[i] * args.n_tiles0 * args.k_splits;
      }
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
        run += cnt[i] * args.n_tiles0 * args.k_splits;
      }
    }
    if (lane == 31) sch->tile_start[G] = incl;
}

}  // namespace asap
