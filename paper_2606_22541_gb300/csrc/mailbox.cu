// Control kernels of the single-GPU mailbox: the form the asynchronous
// dispatch / combine primitives of ASAP (Sections 3.2.1 and 3.2.2, Table 2)
// take when the attention DP groups and the MoE side share one GPU.
//
//  - A DP group posts a routed micro-batch into its slot: its token metadata
//    (idx, weights, per-chunk expert histogram) sits in the slot's region, and
//    the publish kernel sets the slot's ready flag, an epoch, with a release
//    store (the "bitmap" of region 3 of Table 2).
//  - A service round's claim kernel polls every slot's flag once and claims
//    every post that is ready and not yet served and belongs to the same MoE
//    layer as the post the round was started for (async-dispatch-recv): the
//    MoE side serves whatever has arrived for that layer, in slot order,
//    without waiting for the others; the grouped GEMMs read the layer's
//    weights at the id the claim wrote (the layer-oblivious kernels of
//    Section 3.4.2), so layers are served in whatever order their posts come.
//  - After the round's grouped GEMMs and combine, the finish kernel sets each
//    claimed slot's completion flag (async-combine-send; also written to
//    host-mapped memory, which the attention side can poll).
//
// No kernel here waits for a kernel that may still be queued behind it: the
// host orders every publish before the round that must include it with a CUDA
// event, so the claim kernel's wait for its own post ends at once; the wait is
// bounded (it records ST_MBOX_WAIT and goes on) for posts that never come.
#include "common.cuh"
#include "internal.h"

namespace asap {

namespace {

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_gpu_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ void st_release_sys_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.sys.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// One thread: the slot's descriptor, then its ready epoch (release).
__global__ void mbox_publish_kernel(MboxSlot* slots, int slot, const void* x, int n, void* out,
                                    const int32_t* layer, unsigned long long epoch, uint32_t* status) {
  if (threadIdx.x != 0) return;
  MboxSlot* m = slots + slot;
  // the previous post of this slot must have been served (the host makes the
  // publishing stream wait for that round first)
  if (ld_acquire_u64(&m->served) != ld_acquire_u64(&m->posted)) record_status(status, ST_MBOX_OVERRUN);
  m->x = x;
  m->out = out;
  m->n = n;
  m->layer = *reinterpret_cast<const volatile int32_t*>(layer);
  __threadfence();
  st_release_gpu_u64(&m->posted, epoch);
}

// One CTA, one thread per slot.
__global__ void __launch_bounds__(kMboxMaxSlots) mbox_claim_kernel(MboxSlot* slots, const MboxGeom g, int own_slot,
                                                                   unsigned long long own_epoch,
                                                                   unsigned long long wait_ns, MboxRound* r,
                                                                   int32_t* rowmap, int32_t* ticket,
                                                                   uint32_t* status) {
  __shared__ int s_cnt[2], s_tok[2], s_chk[2];
  __shared__ int s_layer, s_first;
  const int s = threadIdx.x, lane = s & 31, warp = s >> 5;
  if (s == 0) {
    bool own = false;
    if (own_slot >= 0) {
      const uint64_t t0 = globaltimer_ns();
      while (!(own = ld_acquire_u64(&slots[own_slot].posted) >= own_epoch)) {
        if (globaltimer_ns() - t0 > wait_ns) {
          record_status(status, ST_MBOX_WAIT);
          break;
        }
        __nanosleep(2000);
      }
    }
    // the round serves the layer of the post it was started for
    s_layer = own ? slots[own_slot].layer : 0;
    s_first = own ? -1 : kMboxMaxSlots;
  }
  __syncthreads();
  bool pend = false;
  unsigned long long posted = 0;
  if (s < g.n_slots) {
    posted = ld_acquire_u64(&slots[s].posted);
    pend = posted > slots[s].served;  // served: written only by this stream's finish kernels
  }
  if (s_first >= 0) {
    // no post to follow (its wait ran out): the layer of the lowest pending slot
    if (pend) atomicMin(&s_first, s);
    __syncthreads();
    if (s == 0 && s_first < g.n_slots) s_layer = slots[s_first].layer;
    __syncthreads();
  }
  const int layer = s_layer;
  int n = 0;
  if (pend) {
    pend = slots[s].layer == layer;  // posts of other layers wait for a round of their own
    if (pend) n = min(max(slots[s].n, 0), g.slot_tokens);
  }
  const int ch = pend ? (n + kChunkTokens - 1) / kChunkTokens : 0;
  // exclusive prefix, in slot order, of (claimed, tokens, histogram rows)
  int ic = pend ? 1 : 0, it = n, ih = ch;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int a = __shfl_up_sync(0xffffffffu, ic, o), b = __shfl_up_sync(0xffffffffu, it, o),
              c = __shfl_up_sync(0xffffffffu, ih, o);
    if (lane >= o) {
      ic += a;
      it += b;
      ih += c;
    }
  }
  if (lane == 31) {
    s_cnt[warp] = ic;
    s_tok[warp] = it;
    s_chk[warp] = ih;
  }
  __syncthreads();
  if (warp == 1) {
    ic += s_cnt[0];
    it += s_tok[0];
    ih += s_chk[0];
  }
  if (pend) {
    const int i = ic - 1;
    r->index_of[s] = i;
    r->slot[i] = s;
    r->n[i] = n;
    r->tok0[i] = it - n;
    r->epoch[i] = posted;
    r->x[i] = slots[s].x;
    r->out[i] = slots[s].out;
    for (int c = 0; c < ch; ++c) rowmap[ih - ch + c] = s * g.slot_chunks + c;
  }
  if (s == kMboxMaxSlots - 1) {
    r->count = ic;
    r->n_total = it;
    r->chunks_total = ih;
    r->layer = layer;
    r->rounds += 1;
    *ticket = 0;  // the scan that follows counts its CTAs on it
  }
}

// One thread per claimed slot.
__global__ void __launch_bounds__(kMboxMaxSlots) mbox_finish_kernel(MboxSlot* slots, const MboxRound* r,
                                                                    int32_t* log,
                                                                    unsigned long long* served_host) {
  const int i = threadIdx.x;
  if (i < r->count) {
    const int s = r->slot[i];
    const unsigned long long e = r->epoch[i];
    __threadfence_system();
    st_release_gpu_u64(&slots[s].served, e);
    if (served_host) st_release_sys_u64(served_host + s, e);
  }
  if (i == 0 && log) {
    const int k = r->rounds - 1;
    if (k >= 0 && k < kMboxLog) log[k] = r->count;
  }
}

}  // namespace

cudaError_t launch_mbox_publish(MboxSlot* slots, int slot, const void* x, int n, void* out, const int32_t* layer,
                                unsigned long long epoch, uint32_t* status, cudaStream_t s) {
  mbox_publish_kernel<<<1, 32, 0, s>>>(slots, slot, x, n, out, layer, epoch, status);
  return cudaGetLastError();
}

cudaError_t launch_mbox_claim(MboxSlot* slots, MboxGeom g, int own_slot, unsigned long long own_epoch,
                              unsigned long long wait_ns, MboxRound* r, int32_t* rowmap, int32_t* ticket,
                              uint32_t* status, cudaStream_t s) {
  mbox_claim_kernel<<<1, kMboxMaxSlots, 0, s>>>(slots, g, own_slot, own_epoch, wait_ns, r, rowmap, ticket, status);
  return cudaGetLastError();
}

cudaError_t launch_mbox_finish(MboxSlot* slots, const MboxRound* r, int32_t* log, unsigned long long* served_host,
                               cudaStream_t s) {
  mbox_finish_kernel<<<1, kMboxMaxSlots, 0, s>>>(slots, r, log, served_host);
  return cudaGetLastError();
}

}  // namespace asap
