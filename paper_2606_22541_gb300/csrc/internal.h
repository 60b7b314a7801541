// Host-side declarations shared by the translation units of libasap_moe.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

namespace asap {

// ------------------------------------------------------------ grouped GEMM
// One launch computes up to two problems with the same epilogue:
//  problem 0: ``groups`` row segments of A (segment g = rows
//             [offsets[g], offsets[g+1]) ), each multiplied by its own B block
//             (rows g*b_stride0 ... of the B tensor); or, with offsets ==
//             nullptr, one plain GEMM of m0 rows.
//  problem 1: one plain GEMM of m1 rows (the shared expert), optional.
// C = A B^T with A [rows, K] and B [N, K] both K-major bf16.
enum { EPI_SWIGLU = 0, EPI_BF16 = 1, EPI_F32 = 2 };

// ------------------------------------------------------------ layer table
// The layer-oblivious kernels of Section 3.4.2: every weight a kernel reads is
// found through a device array with one entry per layer, indexed by a layer id
// the kernel loads from device memory when it runs.  The entry holds the TMA
// descriptors of that layer's packed weights (the pre-computed addresses) and
// plain pointers for what is not read by TMA.
enum { MAP_ROUTER = 0, MAP_GATE_UP = 1, MAP_DOWN = 2, MAP_SH_GATE_UP = 3, MAP_SH_DOWN = 4, kLayerMaps = 5 };

struct alignas(128) LayerEntry {
  CUtensorMap map[kLayerMaps];     // indexed by MAP_*; unused maps are zero
  const float* scale[kLayerMaps];  // FP8 block scales of the same matrices, else nullptr
  const void* router_w;            // [E, H] bf16
  const float* router_bias;        // [E] fp32 or nullptr
};

// Which entry a launch uses: table[*layer].  An id outside [0, n_layers) is
// recorded as ST_BAD_LAYER and replaced by 0, so no access leaves the table.
struct LayerRef {
  const LayerEntry* table;  // device [n_layers]
  const int32_t* layer;     // device int32, read by the kernel
  int n_layers;
};

struct GemmArgs {
  const int32_t* offsets;  // [groups + 1] or nullptr
  int groups;              // 1 when offsets == nullptr
  int m0;                  // rows of A0 (segment ends are checked against it)
  int b_stride0;           // B0 rows between consecutive groups
  int n_tiles0;            // 256-wide N tiles per group
  int k_iters0;            // K0 / 64
  void* out0;
  long long ldo0;          // elements between output rows
  int m1;                  // rows of problem 1 (0 = none; the upper bound when m1_dev is set)
  const int32_t* m1_dev;   // nullable: rows of problem 1 read when the launch runs, clamped to [0, m1]
  int n_tiles1;
  int k_iters1;
  void* out1;
  long long ldo1;
  uint32_t* status;
  int hint_a, hint_b;      // L2 priority of A / B loads: 0 normal, 1 first, 2 last
  int k_splits;            // problem 0 split into this many K slices (>= 1)
  long long split_rows0;   // output rows between the planes of consecutive K slices
  LayerRef lref;           // B of problem p is lref.table[layer].map[bmap_p]
  int bmap0, bmap1;
  int* tile_counter;       // zero at launch: tiles are claimed dynamically; nullptr: static order
  int b_tiled;             // B in tile-contiguous order (launch_retile): box row ((b_row/256) k_iters + kb) 256
  // combine fused into the down GEMM (EPI_BF16 only; comb_cnt == nullptr: off)
  int* comb_cnt;             // [comb_n, n_tiles0] arrivals per token slice, zero at launch
  const int32_t* comb_src;   // [m0] token of each routed row (perm_src)
  const int32_t* comb_dst;   // [comb_n, comb_k] routed row of each token slot (perm_dst)
  const float* comb_w;       // [comb_n, comb_k] routing weights
  void* comb_out;            // [comb_n, ldo0] bf16 layer output
  int comb_n, comb_k;        // tokens (problem 1's rows when it exists) and slots per token
};

constexpr int kTileCounters = 2;  // per call: gate/up GEMM, down GEMM
constexpr int kGemmBM = 128;
constexpr int kGemmBN = 256;
// K per stage: 64 bf16, one 128-byte swizzled row per box row (the weight
// packing of launch_retile and the tile-contiguous addressing assume it)
constexpr int kGemmBK = 64;

cudaError_t gemm_set_attributes();
// maps: A0, A1 (A1 may repeat A0 when m1 == 0), encoded for boxes of 128 rows,
// or 256 rows with pair; then O0, O1, the bf16 outputs out0 / out1 encoded for
// boxes of 32 rows (O1 may repeat O0 when m1 == 0; EPI_F32 ignores both).  The
// B maps come from the layer table.  pair: tiles of two 128-row m-tiles
// sharing the weight boxes (EPI_SWIGLU and EPI_BF16).
cudaError_t gemm_launch(int epi, bool pair, const CUtensorMap* maps, const GemmArgs& args, int grid,
                        cudaStream_t stream);
// Encode a 2-D row-major bf16 tensor [rows, cols] for 128-byte-swizzled
// boxes of [box_rows, 64].  Returns false and fills *err on failure.
bool encode_tmap_bf16(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols,
                      uint32_t box_rows, std::string* err);

// ------------------------------------------------------------ FP8 grouped GEMM
// e4m3 A and B with fp32 block scales: A scales per row per 128-wide K block
// ([rows][K/128]), B scales per 128 x 128 block ([groups][N/128][K/128]).
// Per 128-wide K block the tensor core accumulates into one of two TMEM
// partial buffers; the epilogue warps add each partial, times the row and
// block scales, into fp32 registers.
//  EPI_SWIGLU: out = e4m3 h [rows][N/2] (B rows interleaved 128 gate / 128 up
//              per 256-row tile, B scale rows interleaved gate / up) and
//              out_scale = per row per 128 channels of h ([rows][N/256]).
//  EPI_BF16:   out = bf16 [rows][N].
struct Fp8Args {
  GemmArgs g;
  const float* a_scale0;  // [m0][a_sld0]
  const float* a_scale1;  // [m1][a_sld1]
  int a_sld0, a_sld1;     // K/128
  // B scales: table[layer].scale[bmap_p], [groups][b_nblk0][a_sld0] for
  // problem 0 and [b_nblk1][a_sld1] for problem 1
  int b_nblk0, b_nblk1;   // N/128
  float* out_scale0;      // EPI_SWIGLU only: [m0][o_sld0]
  float* out_scale1;
  int o_sld0, o_sld1;
};
constexpr int kFp8BK = 128;  // K elements (bytes) per stage and per scale block

cudaError_t fp8_gemm_set_attributes();
cudaError_t fp8_gemm_launch(int epi, const CUtensorMap* maps, const Fp8Args& args, int grid, cudaStream_t stream);
// 2-D row-major byte tensor [rows, cols] for 128-byte-swizzled boxes of [box_rows, 128].
bool encode_tmap_u8(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                    std::string* err);

// Rows of bf16 -> e4m3 with one fp32 scale per row per 128 channels
// (s = amax / 448, q = round-to-nearest-even of v / s, saturated).
cudaError_t launch_quantize_rows(const void* x, int rows, int cols, void* q, float* s, cudaStream_t st);

// ------------------------------------------------------------ routing
struct GateParams {
  int n_experts, top_k, gating, n_groups, topk_groups;
  float route_scale;
  LayerRef lref;  // selection bias: table[layer].router_bias ([E] or nullptr)
  uint32_t* status;
  int32_t* ticket;  // the scan's ticket, zeroed by the gate launch (nullable)
};
// Router on the CUDA cores (E < 256): weights table[layer].router_w.
cudaError_t launch_router_small(const void* x, const LayerRef& lref, int n, int H, int E, float* logits,
                                uint32_t* status, cudaStream_t s);
// logits: ``splits`` planes of [n, E] partial sums, added in plane order.
// hist is written chunk-major: hist[chunk * E + e].
cudaError_t launch_gate(const float* logits, int splits, int n, const GateParams& p, int32_t* idx, float* w,
                        int32_t* hist, cudaStream_t s);
cudaError_t launch_reduce_splits(const float* parts, int splits, long long plane, float* out, cudaStream_t s);
// Gating of one micro-batch among several served together: its chunks are
// rows [chunk0, chunk0 + ceil(n/32)) of the chunk-major histogram with
// n_chunks_total rows.
cudaError_t launch_gate_seg(const float* logits, int splits, int n, const GateParams& p, int32_t* idx, float* w,
                            int32_t* hist, int chunk0, int n_chunks_total, cudaStream_t s);
// hist as launch_gate writes it; zeroes the scan's ticket.
cudaError_t launch_hist(const int32_t* idx, int n, int k, int E, int32_t* hist, uint32_t* status, int32_t* ticket,
                        cudaStream_t s);
// counts, offsets, and chunk_base[c][e] = entries of expert e in chunks
// before c (relative: the absolute base is offsets[e] + chunk_base[c][e]);
// hist and chunk_base are chunk-major [n_chunks][E].
// ticket: one int, zero at launch (the gate / hist launch zeroes it), left
// zero.  tile_counters (nullable): kTileCounters ints zeroed for the grouped
// GEMMs that follow on the stream.
cudaError_t launch_scan(const int32_t* hist, int n_chunks, int E, int32_t* counts, int32_t* offsets,
                        int32_t* chunk_base, int32_t* ticket, cudaStream_t s, int32_t* tile_counters = nullptr);

// Routing of one micro-batch in one launch (E = 256 on the tensor core,
// grouped sigmoid gating with 1, 2, 4 or 8 groups): router logits over
// ``splits`` K slices (a cluster of that many CTAs per 128-token tile, slices
// added in order), gating, idx / w, the chunk-major histogram of its chunks
// (rows chunk0 + c of n_chunks_total) and, when ticket is non-null, the
// scan into chunk_base, counts and offsets by the last CTA (ticket zero at
// launch, left zero) which also zeroes tile_counters (nullable).
constexpr int kRouteExperts = 256;
struct RouteFusedArgs {
  LayerRef lref;  // router weights: table[layer].map[MAP_ROUTER]; selection bias
  uint32_t* status;
  int n, k_iters, splits;
  // seq_slices > 1 (with splits == 1): one CTA per tile computes the partial
  // logits of that many K slices one after the other and adds them in slice
  // order, the bits of a cluster of seq_slices CTAs without the cluster
  int seq_slices;
  int top_k, n_groups, topk_groups;
  float route_scale;
  int32_t* idx;
  float* w;
  int32_t* hist;
  int chunk0, n_chunks_total;
  int32_t* ticket;
  int32_t* counts;
  int32_t* offsets;
  int32_t* chunk_base;
  int32_t* tile_counters;
};
cudaError_t route_fused_set_attributes();
// tmX: x [n, H] for [128, 64] boxes (encode_tmap_bf16).
cudaError_t launch_route_fused(const CUtensorMap& tmX, const RouteFusedArgs& a, cudaStream_t s);

// ------------------------------------------------------------ permute
// Place of one micro-batch among several served by one call: its chunks start
// at column chunk0 of chunk_base (n_chunks_total columns), its tokens at
// global index tok0, positions run over rows_total rows; x_sh (bf16 only,
// nullable) receives its rows for the shared expert (pointer already offset
// to the micro-batch's first token).
struct DispatchSeg {
  const int32_t* expert_offsets;  // offsets[e] (the scan's output)
  int chunk0;
  int n_chunks_total;
  int tok0;
  long long rows_total;
  void* x_sh;
};
cudaError_t launch_dispatch(const void* x, int n, int H, int k, int E, const int32_t* idx,
                            const int32_t* chunk_base, const int32_t* offsets, void* x_perm, int32_t* perm_src,
                            int32_t* perm_dst, uint32_t* status, cudaStream_t s);
// FP8 dispatch: every token row is quantised once (e4m3, fp32 scale per 128
// channels) and written to its k positions of xq / xs, and to row t of
// xq_sh / xs_sh when those are non-null (shared expert input).
cudaError_t launch_dispatch_fp8(const void* x, int n, int H, int k, int E, const int32_t* idx,
                                const int32_t* chunk_base, const int32_t* offsets, void* xq, float* xs,
                                void* xq_sh, float* xs_sh, int32_t* perm_src, int32_t* perm_dst, uint32_t* status,
                                cudaStream_t s);
// rows_total: rows of y_perm the positions may address (0 = n * k).
cudaError_t launch_combine(const void* y_perm, const void* y_shared, const float* w,
                           const int32_t* perm_dst, int n, int H, int k, void* out,
                           uint32_t* status, cudaStream_t s, long long rows_total = 0);
cudaError_t launch_dispatch_seg(const void* x, int n, int H, int k, int E, const int32_t* idx,
                                const int32_t* chunk_base, void* x_perm, int32_t* perm_src, int32_t* perm_dst,
                                uint32_t* status, const DispatchSeg& seg, cudaStream_t s);
cudaError_t launch_dispatch_fp8_seg(const void* x, int n, int H, int k, int E, const int32_t* idx,
                                    const int32_t* chunk_base, void* xq, float* xs, void* xq_sh, float* xs_sh,
                                    int32_t* perm_src, int32_t* perm_dst, uint32_t* status, const DispatchSeg& seg,
                                    cudaStream_t s);
// Expert weights in tile-contiguous order for the grouped GEMMs' weight
// boxes: box (e, nt, kb) = rows nt*256 .. nt*256+255 of expert e's packed
// matrix ([E][R] rows of row_bytes; gate_up: packed row nt*256 + r is gate
// row nt*128 + r for r < 128, else up row nt*128 + r - 128, a = gate, b = up),
// bytes [kb*128, kb*128+128) of each row, stored as 256 consecutive 128-byte
// rows.  R % 256 == 0 and row_bytes % 128 == 0.
cudaError_t launch_retile(const void* a, const void* b, int E, int R, long long row_bytes, bool gate_up, void* dst,
                          cudaStream_t s);

// ------------------------------------------------------------ mailbox
// The single-GPU form of ASAP's asynchronous dispatch and combine (Sections
// 3.2.1 and 3.2.2): each attention DP group posts a routed micro-batch into
// its slot and sets the slot's ready flag (an epoch); a service round claims
// every slot whose flag is set when the round starts, "migrates" the claimed
// payloads into one expert-major buffer, runs one grouped GEMM pass over all
// of them, writes each micro-batch's output and sets the slot's completion
// flag.  Waits inside the kernels are on flags written before the waiting
// kernel was enqueued (the host orders them with events); each is bounded.
constexpr int kMboxMaxSlots = 64;
constexpr int kMboxLog = 4096;  // rounds whose claimed-slot count is recorded

struct MboxSlot {            // one per slot, device memory
  unsigned long long posted;  // epoch of the slot's last published post (release by the publish kernel)
  unsigned long long served;  // epoch of its last served post (release by a round's finish kernel)
  const void* x;              // the post's hidden states [n, H]
  void* out;                  // its layer output [n, H]
  int n;
  int layer;                  // the MoE layer the post belongs to (its id when it was published)
};

struct MboxRound {           // the set the current service round claimed (its claim kernel writes it)
  int count;                 // claimed slots
  int n_total;               // their tokens: rows of the shared expert's input
  int chunks_total;          // their histogram rows (rowmap entries)
  int rounds;                // service rounds run so far, this one included
  int layer;                 // the layer every claimed post belongs to (the GEMMs read its weights)
  int index_of[kMboxMaxSlots];  // claimed slot -> its index i below (unclaimed slots: stale)
  int slot[kMboxMaxSlots];   // claimed slots, increasing
  int n[kMboxMaxSlots];
  int tok0[kMboxMaxSlots];   // first token in the round's combined token order
  unsigned long long epoch[kMboxMaxSlots];
  const void* x[kMboxMaxSlots];
  void* out[kMboxMaxSlots];
};

// Where each slot's per-post data sits (fixed when the mailbox is made):
// slot s owns tokens [s * slot_tokens, (s + 1) * slot_tokens) of the idx, w
// and perm_dst arrays (k entries per token) and histogram rows
// [s * slot_chunks, (s + 1) * slot_chunks).
struct MboxGeom {
  int n_slots, slot_tokens, slot_chunks;
  int k, E, H;
};

// Producer: publish a post (after its routing on the same stream) of the
// layer whose id is *layer.  Records ST_MBOX_OVERRUN when the slot's previous
// post has not been served.
cudaError_t launch_mbox_publish(MboxSlot* slots, int slot, const void* x, int n, void* out, const int32_t* layer,
                                unsigned long long epoch, uint32_t* status, cudaStream_t s);
// Service round, step 1: wait (at most wait_ns) until slot own_slot has
// published epoch own_epoch (own_slot < 0: no wait; a wait that runs out
// records ST_MBOX_WAIT), then claim every slot with posted > served whose post
// belongs to the same layer as that post (after a wait that ran out: as the
// lowest pending slot's post) into *r, write the histogram row map, zero the
// scan's ticket.
cudaError_t launch_mbox_claim(MboxSlot* slots, MboxGeom g, int own_slot, unsigned long long own_epoch,
                              unsigned long long wait_ns, MboxRound* r, int32_t* rowmap, int32_t* ticket,
                              uint32_t* status, cudaStream_t s);
// The scan over the histogram rows rowmap[0 .. *n_chunks) (chunk_base written
// at the same rows), otherwise as launch_scan.
cudaError_t launch_scan_mapped(const int32_t* hist, const int32_t* rowmap, const int32_t* n_chunks, int max_chunks,
                               int E, int32_t* counts, int32_t* offsets, int32_t* chunk_base, int32_t* ticket,
                               int32_t* tile_counters, cudaStream_t s);
// Dispatch of every claimed post into the combined expert segments (rows in
// (claimed slot, token, slot of k) order); perm_src holds combined token
// indices, perm_dst the slot's own region; x_sh / xq_sh, xs_sh receive the
// combined rows of the shared expert.
// rowmap: the round's histogram rows (the claim kernel's map).
cudaError_t launch_dispatch_mbox(const MboxRound* r, MboxGeom g, const int32_t* rowmap, const int32_t* idx,
                                 const int32_t* chunk_base, const int32_t* offsets, void* x_perm, int32_t* perm_src,
                                 int32_t* perm_dst, void* x_sh, uint32_t* status, cudaStream_t s);
cudaError_t launch_dispatch_fp8_mbox(const MboxRound* r, MboxGeom g, const int32_t* rowmap, const int32_t* idx,
                                     const int32_t* chunk_base, const int32_t* offsets, void* xq, float* xs,
                                     void* xq_sh, float* xs_sh, int32_t* perm_src, int32_t* perm_dst,
                                     uint32_t* status, cudaStream_t s);
// Combine of every claimed post into its own output.
cudaError_t launch_combine_mbox(const MboxRound* r, MboxGeom g, const void* y_perm, const void* y_shared,
                                const float* w, const int32_t* perm_dst, uint32_t* status, cudaStream_t s);
// Service round, last step: release each claimed slot's completion epoch (and
// its copy in host-mapped memory, nullable) and log the claimed count.
cudaError_t launch_mbox_finish(MboxSlot* slots, const MboxRound* r, int32_t* log, unsigned long long* served_host,
                               cudaStream_t s);

inline int ceil_div(long long a, long long b) { return static_cast<int>((a + b - 1) / b); }

}  // namespace asap
