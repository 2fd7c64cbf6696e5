// wq_internal.h -- types shared by the host-side API (wq_api.cu) and the
// kernel translation units.  Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace wq {

constexpr int kMaxTokens = 64;      // tokens per call the dequant-GEMV kernels can take
constexpr int kGemvPreferTokens = 16;  // above this many tokens the calls take the dequant-GEMM path
constexpr int kMaxGemmTokens = 16384;  // tokens per call on the dequant-GEMM path (above kMaxTokens)
constexpr int kMaxRank = 64;        // LoRA rank limit
constexpr float kRmsEps = 1e-6f;    // RMSNorm epsilon of WQ_PRENORM

// How one dequant-GEMV launch splits its work.
//   Row tiles (16 output rows) are grouped into row blocks of RB tiles; the
//   input features (128-wide blocks) into P panels of KP blocks.  One CTA
//   computes one (row block, panel) unit with RB/TPW*WK warps: warp (rg, wk)
//   owns row tiles rg*TPW .. rg*TPW+TPW-1 of the block and the wk-th share
//   of the panel's blocks.  With P > 1 the panel partial sums of a row tile
//   are added by whichever CTA finishes that row tile last (arrival counter,
//   fixed summation order).
struct GemvPlan {
  int RT, KB;          // row tiles, 128-feature blocks of the whole matrix
  int RB, KP, WK;      // row tiles per unit, blocks per panel, warps along k
  int P, NRB;          // panels, row blocks
  int M, MPAD, NT;     // tokens, tokens padded to the token-chunk size, 8-token tiles per chunk
  int TPW;             // row tiles per warp (1 or 2)
  int threads;         // RB / TPW * WK * 32
  int units;           // grid size = NRB * P
  int r;               // LoRA rank the shared-memory layout was sized for
  uint32_t smem;       // dynamic shared memory bytes
  // byte offsets inside dynamic shared memory
  uint32_t off_codes, off_meta, off_lorab, off_an, off_xp, off_xs, off_sc, off_slots, off_red, off_rt, off_yv,
      off_bar, off_last;
  int xstride;         // halves per token row of the converted activation panel
};

// Per-16-feature "tile partials" connect consecutive launches: for every tile
// of 16 input features and every token, 1 + 2r fp32 values
//   [0]      sum of x^2 over the tile's features            (RMSNorm)
//   [1 + j]  sum over the tile's features of A[j, c] * x[c]   (LoRA-A, Eq. 1)
// padded with zeros to WQ_TP_STRIDE(r) (a multiple of 4) and laid out
// [tile][token][stride].  The gate/up launch adds them over all tiles.
#define WQ_TP_STRIDE(r) ((1 + 2 * (r) + 3) & ~3)
struct GemvArgs {
  const void *act;           // bf16 [M, K]
  int M, K, N, group;
  const uint32_t *codes[2];  // packed codes of the (one or two) matrices
  const uint16_t *meta[2];   // packed binary16 scales / zeros
  // gate/up: tile partials of the input (null when neither prenorm nor LoRA)
  const float *tp;           // [ntp][M][WQ_TP_STRIDE(r)]
  int ntp;                   // tiles = K / 16
  int prenorm;               // scale the products by 1/sqrt(mean(x^2) + eps)
  const void *lora_b[2];     // bf16 [N, r]
  int r;                     // gate/up: LoRA rank; down: rank of lora_a_next
  float lora_scale;
  // down: residual, output and (optionally) the next layer's tile partials
  const void *residual;      // bf16 [M, N] or null
  void *out;                 // bf16 or fp32 [M, N]
  int out_f32;
  const void *lora_a_next;   // bf16 [2r, N] (down with tp_out)
  float *tp_out;             // [ceil(N/16)][M][WQ_TP_STRIDE(r)] or null
  // gate/up in the decode chain: the output h also as the down launch's
  // ready-made binary16 panel (null otherwise; needs RB a multiple of 4):
  //   hq_out  [M][hq_stride] binary16, per 16-feature k-step in the order of
  //           the m16n8k16 B fragments, scaled by 2^e per (64 features,
  //           token) and by 16^-1 on features 8..15 of every k-step (the
  //           4-bit code class), e putting the largest |h| in [2^14, 2^15)
  //   hsc_out [ceil(N/64)][M]  2^(24 - e)
  //   hxs_out [ceil(N/32)][M]  sum of h over 32 features (zero-point term)
  uint16_t *hq_out;
  float *hsc_out, *hxs_out;
  int hq_stride;
  // down: that panel instead of converting act (null: convert act)
  const uint16_t *pre_x;
  const float *pre_sc, *pre_xs;
  int pre_stride;
  float *partials;           // [RT][P][NPROJ][16][M] fp32 (P > 1)
  unsigned *counters;        // [RT] arrival counters, zero between calls
  // Routed experts (launch_gemv_slots only): slot s = blockIdx.y runs the
  // matrix of expert slot_expert[s] (rows e*N .. e*N+N-1 of the stacked
  // codes, meta and LoRA-B) on input row s / slot_div of act, writing output
  // row s; tp, partials and counters hold one region per slot.
  const int *slot_expert;    // [slots], written by the routing kernel
  int n_experts, slot_div;
  int slot_expert_ready;     // the routing kernel completed before this launch can start (not the previous launch)
  // buffer sizes in bytes (checked by the debug build, WQ_DEBUG_CHECKS)
  size_t nb_codes[2], nb_meta[2], nb_lora_b[2], nb_act, nb_tp, nb_res, nb_out, nb_an, nb_tp_out, nb_part, nb_cnt;
  size_t nb_hq, nb_hsc, nb_hxs, nb_pre_x, nb_pre_sc, nb_pre_xs;
};

enum GemvKind { kGateUpW2 = 0, kGateUpW4 = 1, kDownW4 = 2, kGateUpW3 = 3 };
// The gate/up kind of a code width (2, 3 or 4 bits).
inline GemvKind gateup_kind(int bits) { return bits == 2 ? kGateUpW2 : bits == 3 ? kGateUpW3 : kGateUpW4; }

// Batched (prefill-size) dequant-GEMM on the tcgen05 tensor cores (wq_gemm.cu).
struct GemmArgs {
  const uint16_t *act;       // binary16 activations [M][lda] (zero padded to whole 128-feature blocks)
  int lda;
  int M, N, K, group;
  const uint32_t *codes[2];  // packed codes (gate, up) or (down)
  const uint16_t *meta[2];
  const uint16_t *ta;        // gate/up with LoRA: binary16 [M][2r] = lora_scale * x A^T (gate rows, up rows)
  int r;
  const void *lora_b[2];     // bf16 [N][r]
  const float *rs;           // per token: the factor of the fp32 sums (2^-e of the binary16 activations'
                             // scale, times the RMSNorm scale for gate/up), or null for 1
  const void *residual;      // down: bf16 [M][N] or null
  void *out;                 // bf16 (or fp32 for down with out_f32) [M][N]
  int out_f32;
  int mt;                    // token halves of 128 per CTA (1 or 2; set by launch_gemm)
  // stream-K scratch (null: one CTA per tile): gemm_scratch_floats() fp32 and
  // gemm_counters() arrival counters, zero between launches
  float *sk_part;
  unsigned *sk_cnt;
};
cudaError_t launch_gemm(GemvKind kind, const GemmArgs &args, cudaStream_t stream);
// Per token m of x [M, K]: an exact power of two 2^e puts max|x[m]| in
// [2^4, 2^5); x16 [M][lda16] = binary16(2^e x), ta [M][r2] = binary16(2^e
// lora_scale x A^T) (r2 > 0), rs[m] = 2^-e / sqrt(mean(x^2) + eps) (prenorm)
// or 2^-e: the factor the gate/up GEMM's epilogue applies to its sums.
cudaError_t launch_gemm_prep(const void *x, int M, int K, int lda16, const void *lora_a, int r2, float lora_scale,
                             int prenorm, uint16_t *x16, float *rs, uint16_t *ta, cudaStream_t stream);
// x16 [M][lda16] = binary16(2^e x) (zero padded), e per token putting its
// max|x| in [2^4, 2^5); sx[m] = 2^-e (the down GEMM's epilogue factor).
cudaError_t launch_to_f16(const void *x, int M, int K, int lda16, uint16_t *x16, float *sx, cudaStream_t stream);
// Stream-K scratch a GEMM launch of this shape can need: fp32 partial sums
// and per-tile arrival counters (num_sms: the device's SM count).
size_t gemm_scratch_floats(int M, int N, int K, int nproj, int num_sms);
size_t gemm_counters(int M, int N);
int gemm_stages(GemvKind kind, int group);  // depth of the activation-tile ring
// Reads and clears the GEMM kernels' device status word.
cudaError_t read_gemm_status(int *status);

// Plans a launch (memoized); returns false if no configuration fits.
// r: LoRA rank read by the launch (gate/up: its adapter; down: the next
// layer's LoRA-A whose tile partials it writes, 0 for none).
bool plan_gemv(GemvKind kind, int N, int K, int M, int group, int r, int num_sms, GemvPlan *plan);

// Registers per thread of the kernel instantiation a plan selects (device query, cached).
int kernel_regs(GemvKind kind, int group, int NT, int TPW);

// Launches the dequant-GEMV kernel of `kind` (programmatic dependent launch
// when `pdl`).  Returns the CUDA error of the launch.
cudaError_t launch_gemv(GemvKind kind, const GemvPlan &plan, const GemvArgs &args, cudaStream_t stream, bool pdl);

// The same kernels over `slots` routed-expert slots (grid.y; one token each,
// plan made for M = 1 and one expert's N rows).  Needs args.slot_expert.
cudaError_t launch_gemv_slots(GemvKind kind, const GemvPlan &plan, const GemvArgs &args, int slots,
                              cudaStream_t stream, bool pdl);

// Launches the tile-partials kernel of an input x [M, d] (d a multiple of
// 16): tp[tile][m][0] = sum x^2, tp[tile][m][1 + j] = A[j] . x over the
// tile (r2 = 2r rows of A), zeros up to the stride.
cudaError_t launch_tile_prep(const void *x, int M, int d, const void *lora_a, int r2, float *tp, cudaStream_t stream,
                             bool pdl);

// Launches the quantizer / packer (two kernels).
cudaError_t launch_pack(const float *w, int n, int k, int group, int bits, uint32_t *codes, uint16_t *meta,
                        int *nonfinite, cudaStream_t stream);

// Reads and clears the device status word of the current device.
cudaError_t read_device_status(int *status);

// Debug builds (WQ_DEBUG_CHECKS): first failed bounds / alignment check
// {site, line, value, count}; zeros when none failed.  Clears the record.
cudaError_t read_debug_record(long long rec[4]);

}  // namespace wq
