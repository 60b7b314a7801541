/*
 * asap_moe.h -- C ABI of the expert-side MoE layer of ASAP's data-parallel
 * prefill path, for one NVIDIA GB300 (sm_103a).
 *
 * The layer (ASAP Sections 3.2 and 3.4.2; shapes from Table 1 and Section 5.1):
 *
 *   route     : logits L = x Wr^T; top-k gating -> idx[n,k], w[n,k];
 *               per-expert token counts and their exclusive prefix offsets
 *               (the "token metadata" the MoE side receives, Section 3.2.1)
 *   dispatch  : hidden states grouped per expert, x_perm[offsets[e] + r] = x[t]
 *               (the "token payload", Section 3.2.1)
 *   expert_ffn: grouped GEMM, hidden states on the left and one layer's expert
 *               weights on the right (Section 3.4.2):
 *               h = silu(X_e Wg_e^T) * (X_e Wu_e^T);  y = h Wd_e^T,
 *               plus the always-active shared expert on every token (Section 5.1)
 *   combine   : out[t] = sum_j w[t,j] y_perm[perm_dst[t,j]] + y_shared[t]
 *               (expert results returned through the expert IDs, Section 3.2.2)
 *
 * Conventions for every call below:
 *  - Tensors are row-major device pointers owned by the caller, except the
 *    packed weight copies a handle makes in asap_moe_create.  Inputs and
 *    outputs of a call must not overlap.
 *  - Calls other than create / destroy / status only ENQUEUE work on the given
 *    stream: no host synchronisation, no allocation, no read-back of counts.
 *    Micro-batches from different attention DP groups can therefore be
 *    submitted on different streams with no host barrier between them
 *    (Section 3.4.2, bubble-free dispatching).
 *  - Each call in flight needs its own workspace (asap_moe_workspace_size);
 *    two calls that run at the same time must not share one.
 *  - n == 0 is a successful no-op.  n > max_tokens, NULL pointers for
 *    required tensors or a workspace smaller than required return
 *    ASAP_ERR_INVALID / ASAP_ERR_WORKSPACE without enqueuing anything.
 *  - Launch failures return ASAP_ERR_CUDA.  asap_moe_last_error() returns a
 *    thread-local message describing the last failure of this thread.
 *  - A handle is immutable after create; concurrent calls on different
 *    streams with different workspaces are safe.
 *  - A handle belongs to the device that was current at create.  Enqueuing
 *    calls launch on the caller's current device, so they must be made with
 *    that device current and a stream (or NULL, its default stream) of it;
 *    create, destroy, status and the mailbox's create, destroy and rounds
 *    select the handle's device themselves.
 *  - Kernels that detect a bad index or a wait that exceeds its time limit
 *    record it in a device status word of the handle instead of trapping;
 *    asap_moe_status reads and clears it.
 *
 * Layouts (bf16 unless stated; H hidden, E experts, k top-k, I intermediate):
 *   x        [n, H]          hidden states of one micro-batch
 *   idx      [n, k] int32    expert of (token, slot); slot order = descending
 *                            selection score, ties by lower expert index
 *   w        [n, k] fp32     routing weight of (token, slot)
 *   counts   [E]    int32    tokens per expert
 *   offsets  [E+1]  int32    exclusive prefix sum of counts, offsets[E] = n*k
 *   perm_src [n*k]  int32    position -> token
 *   perm_dst [n*k]  int32    (token t, slot j) at t*k + j -> position; inside
 *                            a segment positions follow increasing (t, j)
 *   x_perm   [n*k, H]        expert-grouped hidden states
 *   y_perm   [n*k, H]        expert outputs, same order as x_perm
 *   y_shared [n, H]          shared-expert output (unused when n_shared == 0)
 *   out      [n, H]          layer output
 */
#ifndef ASAP_MOE_H
#define ASAP_MOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ASAP_MOE_MAX_EXPERTS 256
#define ASAP_MOE_MAX_TOPK 8

typedef enum {
  ASAP_OK = 0,
  ASAP_ERR_INVALID = -1,      /* bad argument or configuration */
  ASAP_ERR_UNSUPPORTED = -2,  /* valid request the library does not implement */
  ASAP_ERR_WORKSPACE = -3,    /* workspace missing or too small */
  ASAP_ERR_CUDA = -4,         /* a CUDA runtime call or launch failed */
  ASAP_ERR_DEVICE_STATUS = -5 /* a kernel recorded an error (asap_moe_status) */
} asap_status;

/* Gating rules (the paper names the model, not the rule; these are the
 * published definitions of the model families):
 *  SOFTMAX          p = softmax(L); top-k of p; w = p (no renormalisation)
 *  SOFTMAX_RENORM   as SOFTMAX, then w = p / sum of the selected p
 *  SIGMOID_GROUPED  s = sigmoid(L); selection score s + bias; n_groups equal
 *                   contiguous groups scored by the sum of their two best
 *                   selection scores; keep topk_groups groups; top-k of their
 *                   experts; w = s / sum of selected s * route_scale.
 * Ties go to the lower expert (group) index.                                */
typedef enum {
  ASAP_GATE_SOFTMAX = 0,
  ASAP_GATE_SOFTMAX_RENORM = 1,
  ASAP_GATE_SIGMOID_GROUPED = 2
} asap_gating;

typedef enum {
  ASAP_BF16 = 0,              /* bf16 storage, fp32 accumulation */
  ASAP_FP8_E4M3_BLOCK128 = 1  /* e4m3 expert weights with one fp32 scale per
                                 128 x 128 block; activations (x before the
                                 gate/up GEMM, h before the down GEMM) e4m3 per
                                 token per 128 channels with fp32 scales
                                 s = amax / 448; fp32 accumulation; bf16 out.
                                 The router stays bf16. */
} asap_dtype;

/* Shape and gating of one MoE layer.  Table 1 of the paper: E_total = 256,
 * K = 8, H = 7168, 16-bit data; Section 5.1: one shared expert.
 * Requirements: hidden % 256 == 0; inter % 128 == 0; shared_inter % 128 == 0
 * when n_shared == 1; 1 <= n_experts <= 256; 1 <= top_k <= min(8, n_experts);
 * for SIGMOID_GROUPED n_experts % n_groups == 0, group size >= 2 and
 * top_k <= topk_groups * group size; max_tokens * top_k < 2^31.            */
typedef struct {
  int32_t hidden;        /* H */
  int32_t n_experts;     /* E, routed experts */
  int32_t top_k;         /* k */
  int32_t inter;         /* I, routed-expert intermediate size */
  int32_t n_shared;      /* 0 or 1 shared expert */
  int32_t shared_inter;  /* I_s */
  int32_t gating;        /* asap_gating */
  int32_t n_groups;      /* SIGMOID_GROUPED only */
  int32_t topk_groups;   /* SIGMOID_GROUPED only */
  float route_scale;     /* SIGMOID_GROUPED only */
  int32_t dtype;         /* asap_dtype */
  int32_t max_tokens;    /* largest micro-batch a call may pass */
} asap_moe_config;

/* Device pointers to one layer's weights (row-major).  They are copied (and
 * re-packed) by asap_moe_create; the caller may free them afterwards.
 *   router_w  [E, H] bf16
 *   router_bias [E] fp32 or NULL: selection-only correction bias
 *   w_gate, w_up [E][I, H];  w_down [E][H, I]  (bf16, or e4m3 for FP8)
 *   sh_gate, sh_up [I_s, H]; sh_down [H, I_s]   (NULL when n_shared == 0)
 *   FP8 only, fp32 scales of 128 x 128 blocks (NULL for bf16):
 *   s_gate, s_up [E][I/128][H/128]; s_down [E][H/128][I/128];
 *   sh_s_gate, sh_s_up [I_s/128][H/128]; sh_s_down [H/128][I_s/128]      */
typedef struct {
  const void* router_w;
  const float* router_bias;
  const void* w_gate;
  const void* w_up;
  const void* w_down;
  const float* s_gate;
  const float* s_up;
  const float* s_down;
  const void* sh_gate;
  const void* sh_up;
  const void* sh_down;
  const float* sh_s_gate;
  const float* sh_s_up;
  const float* sh_s_down;
} asap_moe_weights;

typedef struct asap_moe_s* asap_moe_t;

/* Validate cfg, allocate the handle's device memory on the current device,
 * copy and pack the weights (gate/up rows interleaved in blocks of 128 so one
 * 256-wide GEMM tile holds matching gate and up columns) and build the weight
 * TMA descriptors.  Synchronous: it first synchronises the device, so weights
 * still being written on any stream are complete before they are read.  On
 * failure *out is NULL. */
int asap_moe_create(const asap_moe_config* cfg, const asap_moe_weights* weights,
                    asap_moe_t* out);

/* One handle over n_layers MoE layers of the same shape: the layer-oblivious
 * MoE Super Kernel of Section 3.4.2 (Section 4.3 describes it as a layer-ID
 * input plus a pre-computed list of weight addresses).
 *  - weights points to n_layers structs; layer l is copied and packed as
 *    asap_moe_create does, and occupies that much HBM (all layers stay
 *    resident).
 *  - A device table receives, per layer, the TMA descriptors of its packed
 *    weights and its router, bias and scale pointers.  Every kernel of this
 *    library that reads weights finds them in that table at a layer id it
 *    loads from device memory when it starts.
 *  - Calls without a layer_id argument use layer 0.  asap_moe_create(c, w, o)
 *    is asap_moe_create_layers(c, w, 1, o).
 *  - 1 <= n_layers <= 4096, else ASAP_ERR_INVALID.  Synchronous, like
 *    asap_moe_create.                                                      */
int asap_moe_create_layers(const asap_moe_config* cfg, const asap_moe_weights* weights,
                           int32_t n_layers, asap_moe_t* out);

/* Number of layers of the handle (1 for asap_moe_create). */
int asap_moe_n_layers(asap_moe_t h, int32_t* n_layers);

/* Tile shape of the BF16 grouped expert GEMMs (gate/up and down) of the
 * calls that follow on this handle (the FP8 GEMMs have one shape):
 *  - ASAP_TILING_AUTO (the default): per launch, paired tiles when the
 *    routed rows average at least 128 per expert and the launch has at least
 *    three waves of paired tiles (estimated from n, top_k and the expert
 *    count; one tile per SM per wave), else single tiles.
 *  - ASAP_TILING_SINGLE: 128-row m-tiles.
 *  - ASAP_TILING_PAIRED: two 128-row m-tiles of one expert per tile, sharing
 *    every weight box; a segment's last <= 128 rows form a half tile.
 * Every mode computes each output element with the same products in the same
 * order, so the results are bit-identical; only the speed differs.  Another
 * mode returns ASAP_ERR_INVALID.  Host state only (nothing is enqueued); do
 * not call it while another thread enqueues on the same handle. */
enum {
  ASAP_TILING_AUTO = 0,
  ASAP_TILING_SINGLE = 1,
  ASAP_TILING_PAIRED = 2
};
int asap_moe_set_tiling(asap_moe_t h, int32_t mode);

/* Where asap_moe_layer and asap_moe_layer_dyn combine (bf16 layers): in a
 * separate kernel after the down GEMM (ASAP_COMBINE_SEPARATE, the default), or
 * inside the down GEMM's epilogue (ASAP_COMBINE_FUSED): each
 * warp that has stored its rows of an output tile counts one arrival per row
 * for the row's token slice (token, 256 output columns), and the arrival that
 * completes a slice (the token's k routed rows and its shared-expert row)
 * sums that slice in slot order with the separate kernel's arithmetic, so
 * the output bits are the same in both modes.  Measured slower at the
 * DeepSeek-V3 shape (most slices complete in the launch's last tiles, whose
 * warps then hold back the tensor core), hence not the default.  The other
 * calls keep their separate combine.  FP8 handles return ASAP_ERR_UNSUPPORTED
 * for ASAP_COMBINE_FUSED; another mode returns ASAP_ERR_INVALID.  Host state
 * only; do not call it while another thread enqueues on the same handle. */
enum {
  ASAP_COMBINE_SEPARATE = 0,
  ASAP_COMBINE_FUSED = 1
};
int asap_moe_set_combine(asap_moe_t h, int32_t mode);

/* Free everything create allocated.  Synchronises the device first.  NULL is
 * accepted.  Refused with ASAP_ERR_INVALID (nothing freed) while a mailbox
 * created on h is alive: destroy the mailboxes first. */
int asap_moe_destroy(asap_moe_t h);

/* Pure host computation: bytes of workspace one call with n tokens needs.  The
 * same size serves every enqueuing call below.  Needs no GPU. */
int asap_moe_workspace_size(const asap_moe_config* cfg, int32_t n_tokens, size_t* bytes);

/* Pure host computation: ASAP_OK when cfg satisfies the requirements above,
 * otherwise ASAP_ERR_INVALID / ASAP_ERR_UNSUPPORTED and a message.  Needs no
 * GPU. */
int asap_moe_check_config(const asap_moe_config* cfg);

/* Router logits only: logits[n, E] (fp32) = x Wr^T, fp32 accumulation of
 * bf16 products.  Needs a workspace: the tensor-core router splits K into
 * slices and adds them in slice order, exactly as asap_moe_route does, so
 * asap_moe_route_logits on these logits reproduces asap_moe_route. */
int asap_moe_router_logits(asap_moe_t h, const void* x, int32_t n, float* logits,
                           void* ws, size_t ws_bytes, void* stream);

/* Routing (Table 1: top-K of E_total experts; Section 3.2.1: per-expert token
 * counts): logits, gating, idx/w, counts, offsets.  counts and offsets are
 * deterministic.  For E = 256 with grouped sigmoid gating (1, 2, 4 or 8
 * groups) this is one kernel launch (router GEMM over a thread-block cluster,
 * gating and scan) after a 260-byte memset of the workspace's counters; the
 * logits are not written.  Other configurations launch the router, gate and
 * scan kernels in turn. */
int asap_moe_route(asap_moe_t h, const void* x, int32_t n, int32_t* idx, float* w,
                   int32_t* counts, int32_t* offsets, void* ws, size_t ws_bytes,
                   void* stream);

/* Routing from given fp32 logits [n, E] (lets exact ties be tested). */
int asap_moe_route_logits(asap_moe_t h, const float* logits, int32_t n, int32_t* idx,
                          float* w, int32_t* counts, int32_t* offsets, void* ws,
                          size_t ws_bytes, void* stream);

/* Dispatch (Section 3.2.1 token payload): from idx, build perm_src/perm_dst
 * and copy every token row into its k expert segments of x_perm.  idx values
 * outside [0, E) are recorded in the status word and the entry is skipped.
 * FP8 configuration: x_perm is e4m3 [n*k, H] and x_perm_scales fp32
 * [n*k, H/128] (one scale per row per 128 channels, s = amax / 448); each
 * token row is quantised once and written k times.  bf16: x_perm_scales is
 * ignored (pass NULL). */
int asap_moe_dispatch(asap_moe_t h, const void* x, int32_t n, const int32_t* idx,
                      void* x_perm, float* x_perm_scales, int32_t* perm_src,
                      int32_t* perm_dst, void* ws, size_t ws_bytes, void* stream);

/* Expert FFN (Section 3.4.2 GMM): y_perm rows of expert e's segment
 * [offsets[e], offsets[e+1]) = SwiGLU_e(x_perm rows); y_shared = shared
 * SwiGLU of x (ignored when n_shared == 0).  The grouped GEMMs find their
 * tiles on the device from offsets (offsets[E] must equal n*k).  FP8
 * configuration: x_perm / x_perm_scales as produced by asap_moe_dispatch; x
 * stays bf16 (quantised here for the shared expert); h is quantised to e4m3
 * per row per 128 channels between the two GEMMs; y_perm, y_shared bf16. */
int asap_moe_expert_ffn(asap_moe_t h, const void* x_perm, const float* x_perm_scales,
                        const int32_t* offsets, const void* x, int32_t n, void* y_perm,
                        void* y_shared, void* ws, size_t ws_bytes, void* stream);

/* The two halves of asap_moe_expert_ffn, for callers that keep the
 * intermediate activations or time the GEMMs separately (same kernels, same
 * bits):
 *   gate_up: h_perm [n*k, I] = silu(X_e Wg_e^T) * (X_e Wu_e^T) per segment,
 *            h_shared [n, I_s] likewise for the shared expert on x;
 *   down   : y_perm = h_perm Wd_e^T per segment, y_shared = h_shared Ws_d^T.
 * The workspace is optional.  With one (asap_moe_workspace_size for n) the
 * CTAs claim tiles dynamically from a counter in it, as asap_moe_expert_ffn
 * does; with ws == NULL they take tiles in a fixed order, which is slower
 * when other kernels share the GPU.  Same bits either way.  bf16
 * configuration only (the FP8 configuration returns ASAP_ERR_UNSUPPORTED; its
 * h is e4m3 with scales, use asap_moe_expert_ffn); *_scales are ignored
 * (pass NULL). */
int asap_moe_expert_gate_up(asap_moe_t h, const void* x_perm, const float* x_perm_scales,
                            const int32_t* offsets, const void* x, int32_t n, void* h_perm,
                            void* h_shared, void* ws, size_t ws_bytes, void* stream);
int asap_moe_expert_down(asap_moe_t h, const void* h_perm, const float* h_perm_scales,
                         const int32_t* offsets, const void* h_shared, int32_t n, void* y_perm,
                         void* y_shared, void* ws, size_t ws_bytes, void* stream);

/* Combine (Section 3.2.2): out[t] = sum_{j<k} w[t,j] y_perm[perm_dst[t*k+j]]
 * (+ y_shared[t]), fp32 in slot order then the shared row, rounded to bf16.
 * y_shared may be NULL. */
int asap_moe_combine(asap_moe_t h, const void* y_perm, const void* y_shared,
                     const float* w, const int32_t* perm_dst, int32_t n, void* out,
                     void* stream);

/* The whole layer for one micro-batch: route -> dispatch -> expert_ffn ->
 * combine, enqueued on one stream with no host synchronisation.  Bit-identical
 * to the four calls composed. */
int asap_moe_layer(asap_moe_t h, const void* x, int32_t n, void* out, void* ws,
                   size_t ws_bytes, void* stream);

/* asap_moe_layer for the layer whose id is the int32 at layer_id (a device
 * pointer).  The kernels load the id when they run, so what is enqueued does
 * not depend on the layer: a sequence of these calls can be enqueued, or
 * captured once in a CUDA graph and replayed, before the layer of each
 * micro-batch is known (bubble-free kernel dispatching, Section 3.4.2).
 *  - *layer_id must not change from the start of the call's first kernel to
 *    the end of its last: write it on the same stream before the call, or
 *    order the writer with an event.
 *  - An id outside [0, n_layers) sets status bit 16 (asap_moe_status) and
 *    the kernels use layer 0; nothing outside the table is read.
 *  - NULL or unaligned layer_id returns ASAP_ERR_INVALID.
 *  - out for layer l is bit-identical to asap_moe_layer on a handle created
 *    from layer l's weights alone. */
int asap_moe_layer_dyn(asap_moe_t h, const int32_t* layer_id, const void* x, int32_t n,
                       void* out, void* ws, size_t ws_bytes, void* stream);

/* Timing hook: the next asap_moe_layer or asap_moe_layer_dyn call made by
 * this thread records events[0] (a cudaEvent_t; NULL entries are skipped) on
 * its stream before its first kernel and events[i] after its i-th step:
 * 1 route, 2 dispatch, 3 gate/up GEMM, 4 down GEMM, 5 combine, so each of
 * the layer's own kernels can be timed where it runs.  count in [0, 6]
 * (0 clears the request); the request is consumed by that next call even if
 * it fails or has n = 0, which then records nothing.  The events must stay
 * valid until that call returns (recording a destroyed event fails the call
 * with ASAP_ERR_CUDA).  Host state of the calling thread only; enqueues
 * nothing itself. */
int asap_moe_time_layer(int32_t count, void* const* events);

/* asap_moe_route without any device allocation (no counterpart in the
 * paper; this entry point exists for callers that cannot allocate).
 *
 * Some callers cannot call cudaMalloc when they route: their device memory is
 * owned entirely by another allocator (for example a serving framework's pool
 * that reserved the GPU at start-up), or allocation on that path is forbidden
 * or would synchronise the device.  This call takes the same inputs and
 * outputs as asap_moe_route but keeps its scratch (router logits, per-chunk
 * histograms, chunk bases and a counter) in one static device array of the
 * library: 4096 tokens x 256 experts x up to 4 router K-slice planes,
 * 16 MiB + 256 KiB + 256 B, held by every GPU that loads libasap_moe until
 * the process exits.  It calls no cudaMalloc, cudaFree or other allocating
 * routine.
 *  - n > 4096 (or n > max_tokens) returns ASAP_ERR_INVALID with a message.
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture.
 *  - Every call shares the one array, so calls whose work overlaps on the
 *    GPU (for example on two streams without ordering between them) race and
 *    may return wrong routing; order them on one stream or with events.
 *  - The array keeps the last call's contents; every element a call reads is
 *    written earlier by the same call (the counter by a 4-byte memset on the
 *    stream, which allocates nothing).
 *  - It returns the same bits as asap_moe_route for every configuration:
 *    for E = 256 with grouped sigmoid gating it runs the same single launch;
 *    otherwise the same router kernels with the same K slices, the same gate
 *    and the same scan.                                                    */
int asap_moe_route_noalloc(asap_moe_t h, const void* x, int32_t n, int32_t* idx, float* w,
                           int32_t* counts, int32_t* offsets, void* stream);

/* Several micro-batches that are ready at the same time, served in one pass:
 * each is routed exactly as asap_moe_layer would route it alone, then the
 * rows of all of them share the expert segments, so each expert's weights
 * stream from HBM once for the whole set (one grouped GEMM per weight
 * matrix) instead of once per micro-batch.  The paper serves DP groups one at
 * a time and names the lower token density per MoE invocation as the cost of
 * that (Section 3.3); this call trades the independence of the groups for
 * that density when several are ready together.  out for micro-batch i is
 * bit-identical to asap_moe_layer on xs[i] alone.
 *   count      1..64; xs, ns, outs: host arrays of count device pointers /
 *              sizes (ns[i] may be 0)
 *   sum(ns) <= max_tokens; the workspace is asap_moe_workspace_size for
 *   sum(ns) tokens. */
int asap_moe_layer_batched(asap_moe_t h, int32_t count, const void* const* xs, const int32_t* ns,
                           void* const* outs, void* ws, size_t ws_bytes, void* stream);

/* asap_moe_layer_batched for micro-batches that all belong to the layer whose
 * id is at layer_id (device int32), with the rules of asap_moe_layer_dyn. */
int asap_moe_layer_batched_dyn(asap_moe_t h, const int32_t* layer_id, int32_t count,
                               const void* const* xs, const int32_t* ns, void* const* outs,
                               void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Mailbox: the device decides which micro-batches one grouped GEMM pass
 * serves.  The single-GPU form of the asynchronous primitives of Sections
 * 3.2.1 and 3.2.2 (Table 2: per DP group, regions for the token data and the
 * per-expert counts plus ready bits that the MoE side checks before copying a
 * group's data into its own memory; results return with completion bits),
 * with the MoE side serving DP groups out of order (Section 3.3).
 *
 *  - A DP group's stream POSTS a micro-batch into its slot: the post routes
 *    it (the bits of asap_moe_route; for E = 256 with grouped gating one CTA
 *    per 128-token tile instead of a cluster, so posts made together route
 *    side by side) into the slot's region and then sets the slot's ready
 *    flag, an epoch, with a release store.
 *  - The MoE stream SERVES: a service round claims, on the device, every
 *    post whose flag is set and that has not been served when the round
 *    starts; dispatches all claimed posts into one expert-major buffer (the
 *    migration); runs one gate/up and one down grouped GEMM over all of them,
 *    so each expert's weights stream from HBM once per round, not once per
 *    micro-batch; combines each post into its own out; then sets each claimed
 *    slot's completion flag (an epoch in device memory and in host-mapped
 *    memory).
 *  - out of every post is bit-identical to asap_moe_layer on the same x,
 *    whichever other posts share its round.
 *
 * Ordering (no kernel waits for a kernel that may be queued behind it):
 *  - asap_moe_mailbox_serve(slot, epoch) makes the MoE stream wait, with a
 *    CUDA event, for the last post made to that slot; call it after the post
 *    that returned epoch.  The round then claims that post and every other
 *    ready one.  The round's claim kernel also checks the slot's flag and,
 *    if epoch has not been published (a post that was announced but never
 *    made), waits at most wait_ns, records status bit 128 and serves the
 *    posts that are ready.
 *  - A post to a slot waits (on its own stream, with an event) for the round
 *    that served the slot's previous post; posting again before a serve call
 *    was made for the previous post returns ASAP_ERR_INVALID (the sender's
 *    backpressure of Section 3.2.1).
 *  - x and out of a post must stay valid until the post is served.
 *  - Rounds run one after another: each serve call makes its stream wait for
 *    the mailbox's previous round (they share one server workspace), so
 *    serve calls may come from any stream; one MoE stream is the usual case,
 *    where that wait costs nothing.
 *
 * Layers: each post belongs to one MoE layer of the handle (a device int32
 * layer id read when the post is published; see asap_moe_layer_dyn).  A round
 * claims only posts of the layer of the post it was started for, and its
 * grouped GEMMs read that layer's weights, so one mailbox serves every layer
 * of a multi-layer handle, in whatever order the layers' posts arrive
 * (Section 3.4.2); posts of other layers wait for a round of their own.
 *
 * A mailbox owns its memory: a server workspace for n_slots * slot_tokens
 * tokens (asap_moe_workspace_size of that many tokens) and a few KB of state.
 * Calls are thread-safe with respect to each other (one lock per mailbox).
 * ------------------------------------------------------------------------ */
typedef struct asap_moe_mailbox_s* asap_moe_mailbox_t;

/* Create a mailbox of n_slots slots (1..64) of up to slot_tokens tokens
 * (<= max_tokens) each on h's device.  layer_id: the layer of posts made
 * without one, NULL (layer 0) or a 4-byte aligned device int32.  wait_ns > 0:
 * the limit of a round's wait for a post that has not been published.
 * Allocates; synchronous.  h must outlive the mailbox: asap_moe_destroy(h)
 * is refused while the mailbox is alive. */
int asap_moe_mailbox_create(asap_moe_t h, int32_t n_slots, int32_t slot_tokens,
                            const int32_t* layer_id, int64_t wait_ns, asap_moe_mailbox_t* out);

/* Free the mailbox (synchronises the device first).  NULL is accepted. */
int asap_moe_mailbox_destroy(asap_moe_mailbox_t m);

/* Post n tokens of x (0 <= n <= slot_tokens) of the layer at layer_id
 * (NULL: the mailbox's default layer; a device int32 read when the post's
 * kernels run, rules of asap_moe_layer_dyn) into slot on stream: waits on the
 * stream for the slot's previous round, routes with that layer's router,
 * publishes.  *epoch (nullable) receives the post's epoch (1, 2, ... per
 * slot), the value to serve it with.  Enqueues only. */
int asap_moe_mailbox_post(asap_moe_mailbox_t m, int32_t slot, const void* x, int32_t n,
                          void* out, const int32_t* layer_id, void* stream, uint64_t* epoch);

/* One service round on stream for post epoch of slot, as described above.
 * Enqueues only. */
int asap_moe_mailbox_serve(asap_moe_mailbox_t m, int32_t slot, uint64_t epoch, void* stream);

/* One service round on stream for several posts the caller knows were made:
 * count (1..n_slots) distinct slots with, per slot, the epoch
 * asap_moe_mailbox_post returned (a post already made; otherwise
 * ASAP_ERR_INVALID).  The stream waits for all of them, so the round serves
 * them all (with any other ready post of the first one's layer), and each
 * listed slot's completion is ordered after this round: a sender that posts
 * again once its previous post is served (a closed loop) is released by the
 * round that served it.  No counterpart in the paper, whose MoE side serves
 * one DP group at a time.  Enqueues only. */
int asap_moe_mailbox_serve_many(asap_moe_mailbox_t m, int32_t count, const int32_t* slots,
                                const uint64_t* epochs, void* stream);

/* Make stream wait until the round of the serve call for slot's last post
 * has finished (its out is then complete).  ASAP_ERR_INVALID when no serve
 * call has been made for that post. */
int asap_moe_mailbox_wait(asap_moe_mailbox_t m, int32_t slot, void* stream);

/* The slot's completion epoch as the device last released it to host-mapped
 * memory (0 = none yet).  Non-blocking: for a host thread that polls. */
int asap_moe_mailbox_served(asap_moe_mailbox_t m, int32_t slot, uint64_t* epoch);

/* Record ev_before / ev_after (cudaEvent_t) on the stream right before the
 * first and right after the last grouped GEMM of the next serve call (for
 * timing the GEMMs of a round).  NULL events clear the request.  The next
 * asap_moe_mailbox_serve or _serve_many call takes the request whatever its
 * outcome (a call that fails before its GEMMs records nothing); the events
 * must stay valid until that call returns. */
int asap_moe_mailbox_time_gemms(asap_moe_mailbox_t m, void* ev_before, void* ev_after);

/* Synchronise the device; *rounds = service rounds run so far; claimed
 * (nullable) receives the number of posts each of the first min(cap,
 * rounds, 4096) rounds claimed. */
int asap_moe_mailbox_rounds(asap_moe_mailbox_t m, int32_t* rounds, int32_t* claimed, int32_t cap);

/* Synchronise the device, return ASAP_OK or ASAP_ERR_DEVICE_STATUS, write the
 * raw status word (0 = clean) to *word if non-NULL, then clear it.  Bits:
 * 1 expert index outside [0, E); 2 permutation position out of range;
 * 4 a wait passed its time limit; 8 offsets not monotone or past the rows;
 * 16 layer id outside [0, n_layers); 32 a grouped GEMM found its dynamic
 * shared memory misaligned and did nothing; 64 a mailbox slot was published
 * again before its previous post was served; 128 a mailbox round's wait for
 * the post it was started for ran out. */
int asap_moe_status(asap_moe_t h, uint32_t* word);

/* Thread-local text of this thread's last failure ("" if none). */
const char* asap_moe_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* ASAP_MOE_H */
