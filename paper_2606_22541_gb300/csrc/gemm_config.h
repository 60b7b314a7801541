// Tuning parameters of the grouped GEMMs (ring depths per launch kind and
// the L2 priority of their loads), measured on GB300; build-time defines
// override them.
#pragma once

// Ring depths (stages of A [128 x 64] and B [256 x 64] bf16 boxes).  A k-step
// needs both boxes, so the pipeline depth that counts is that of the
// shallowest ring whose operand comes from HBM.  Measured at 4096 DeepSeek-V3
// tokens with the weights in tile-contiguous order (one 32 KB read per box):
// gate/up (GU) 4 + 4 (2.45 ms; 3 + 5: 2.58, 5 + 3: 2.69, 2 + 6: 3.23); down
// (DN) 4 + 4 (1.34 ms; 3 + 5: 1.36, 2 + 6: 1.64, 3 + 4: 1.37).  router (RT):
// activations from HBM, the 256 x H router weights from L2, 6 + 3 (70.5 ->
// 64.5 us at 16384 tokens).
#ifndef ASAP_RING_GU_A
#define ASAP_RING_GU_A 4
#endif
#ifndef ASAP_RING_GU_B
#define ASAP_RING_GU_B 4
#endif
#ifndef ASAP_RING_DN_A
#define ASAP_RING_DN_A 4
#endif
#ifndef ASAP_RING_DN_B
#define ASAP_RING_DN_B 4
#endif
// paired m-tiles (two 128-row m-tiles per tile sharing the weight boxes): A
// stages of 2 x 128 rows (32 KB) and B boxes of 32 KB, 3 + 3 stages.
#ifndef ASAP_RING_PAIR_A
#define ASAP_RING_PAIR_A 3
#endif
#ifndef ASAP_RING_PAIR_B
#define ASAP_RING_PAIR_B 3
#endif
// A launch runs paired m-tiles when it has at least this many waves of them
// (estimated, one tile per SM per wave).  Measured on a GB300 against single
// m-tiles: paired tiles (with half tiles for segment tails) win the gate/up
// GEMM at every measured size (DeepSeek-V3 4096 tokens 2.40 vs 2.45 ms,
// Mixtral 1024 tokens 0.44 vs 0.46 ms) and the down GEMM from about three
// waves (Mixtral 4096 tokens, 3.8 waves: 0.61 vs 0.71 ms), but lose the
// Mixtral down GEMM at 2.9 waves and below (3072 tokens 0.56 vs 0.53 ms).
#ifndef ASAP_PAIR_MIN_WAVES
#define ASAP_PAIR_MIN_WAVES 3
#endif
#ifndef ASAP_RING_RT_A
#define ASAP_RING_RT_A 6
#endif
#ifndef ASAP_RING_RT_B
#define ASAP_RING_RT_B 3
#endif

// L2 priority of the grouped GEMMs' loads (0 normal, 1 evict-first, 2
// evict-last): activations (A) are re-read by every n-tile of their expert
// and stay evict-last; the bf16 weights (B) are read by the m-tiles of one
// expert at about the same time, which find them in L2 only at normal
// priority (measured on GB300 at 4096 DeepSeek-V3 tokens: gate/up 2.90 ->
// 2.59 ms, down 1.78 -> 1.54 ms against evict-first weights).  The FP8 GEMMs
// measured 2 % faster with evict-first weights.
#ifndef ASAP_HINT_BF16_A
#define ASAP_HINT_BF16_A 2
#endif
#ifndef ASAP_HINT_BF16_B
#define ASAP_HINT_BF16_B 0
#endif
// the down GEMM's activations (h), re-read by every n-tile of their expert:
// evict-last as for gate/up (measured: 1.33 ms; normal 1.35, evict-first 1.42)
#ifndef ASAP_HINT_BF16_DN_A
#define ASAP_HINT_BF16_DN_A ASAP_HINT_BF16_A
#endif
#ifndef ASAP_HINT_FP8_A
#define ASAP_HINT_FP8_A 2
#endif
#ifndef ASAP_HINT_FP8_B
#define ASAP_HINT_FP8_B 1
#endif
