// wq_stack.h -- the single-launch decode stack (wq_stack.cu): its launch plan
// and arguments, shared by the host API (wq_api.cu) and the kernel.  Not part
// of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda.h>
#include <cuda_runtime.h>

namespace wq {

// Per-launch constants computed on the host (stack_plan); identical for all CTAs.
struct StackPlan {
  int G;                 // CTAs (one per SM)
  int RTg, KBg;          // gate/up row tiles, gate/up 128-feature blocks
  int RTd, U;            // down row tiles (= y tiles), down 64-feature half blocks
  int cells;             // U * RTd (down work cells, half-block major)
  int WPT;               // math warps per gate/up row tile
  int Tmax, nj_max, own_max;
  int kps, cps;          // gate/up k-blocks per stage, down cells per stage
  int SB, NS;            // stage bytes, stages in the ring
  int Qp;                // tile-partial stride
  int h_barrier;         // a CTA's down slice needs other CTAs' h: barrier before the down phase
  int nchk;              // chunks of the tile-partial sum
  int Tbox;              // row tiles per gate/up TMA box (all of a CTA's when every CTA has Tmax, else 1)
  int gmy;               // groups per gate/up meta box row: kps * 128 / group rounded up to even (128-byte rows)
  int RPS;               // down row tiles per stage (one TMA box)
  uint32_t smem;
  uint32_t off_full, off_empty, off_misc, off_x, off_xsc, off_xs, off_slot, off_h, off_hp, off_hsc, off_hxs, off_lb,
      off_la, off_rt, off_yo, off_red, off_ring;
  int xstride;           // halves per token row of the activation panel
};

struct StackLayerDev {
  const uint16_t *lora_a;     // bf16 [2r][d]
  const uint16_t *lora_b[2];  // bf16 [inter][r]
  float lora_scale;
};

// Layers a launch carries (longer stacks take several launches): the tensor
// maps of a layer take 768 bytes of the launch's 32 KB parameter space.
constexpr int kStackMaxLayers = 32;

// TMA tensor maps of a layer's packed weights (3-D views of the packed format):
//   gate/up codes [RT][KB * BPK / 128][128 B], boxes of Tbox row tiles x kps blocks;
//   gate/up meta  [RT][KB * 128 / group][64 B], boxes of Tbox row tiles x gmy groups;
//   down codes    [RT][KB * 8][128 B], boxes of RPS row tiles x one 64-feature half block;
//   down meta     [RT][NG][64 B], boxes of RPS row tiles x the groups of a half block.
struct StackMaps {
  CUtensorMap m[kStackMaxLayers][6];  // gate codes, up codes, gate meta, up meta, down codes, down meta
};

struct StackArgs {
  int M, d, inter, r, g_gu, g_dn, bits_gu, n_layers, prenorm;
  const uint16_t *x_in;      // bf16 [M][d]
  uint16_t *y_out;           // bf16 [M][d]
  uint16_t *states;          // bf16 [n][M][d] or null
  uint16_t *h_states;        // bf16 [n][M][inter] or null
  uint16_t *xw;              // working residual stream, bf16 [M][d]
  float *tp;                 // [RTd][M][Qp] per-tile RMSNorm / LoRA-A partial sums
  uint16_t *hg;              // h in global memory, bf16 [M][inter] (h_barrier plans)
  float *part;               // [U][M][d] down partial sums
  unsigned long long *ctr;   // grid-barrier arrival counter (a multiple of G between launches)
  StackLayerDev L[kStackMaxLayers];
};

// The launch plan of an (M, d, inter, r, bits, groups) stack on num_sms SMs;
// false when the stack kernel does not take this shape.
bool stack_plan(int M, int d, int inter, int r, int bits_gu, int g_gu, int g_dn, int num_sms, StackPlan *out);
// Workspace bytes of its buffers (after the arrival counter).
size_t stack_buffer_bytes(int M, int d, int inter, int r);
// The tensor maps of one layer (cached by pointer and shape).
cudaError_t stack_layer_maps(const void *gate_codes, const void *up_codes, const void *gate_meta, const void *up_meta,
                             const void *down_codes, const void *down_meta, int d, int inter, int bits_gu, int group,
                             const StackPlan &p, CUtensorMap out[6]);
cudaError_t launch_stack(const StackArgs &a, const StackPlan &p, const StackMaps &maps, cudaStream_t s);
// Reads and clears the stack kernel's device status word.
cudaError_t read_stack_status(int *status);
// The bounded-wait self-check (wq_wait_check).
cudaError_t launch_wait_check(cudaStream_t s);

}  // namespace wq
