/*
 * wq.h -- C ABI of the W4/W2-GateUp decode MLP library (libwq.so, sm_103a).
 *
 * The library computes the decode-regime gated-MLP block of the W4/W2-GateUp
 * scheme: gate and up projections quantized to 2 bits, the down projection
 * to 4 bits (Sec. 3.3), with the Recover-LoRA adapters left unmerged on gate
 * and up (Eq. 1, Y = W X + alpha B A X; Sec. 4.2 allows deploying them either
 * merged or as an extra low-rank path, and this library takes the second
 * option).  The quantizer is the Stage-1 group-wise post-training
 * quantization of Sec. 4.1.
 *
 * Conventions shared by every call:
 *   - All tensor arguments are DEVICE pointers owned by the caller.  The
 *     library never allocates device memory and never synchronizes; every
 *     call is asynchronous on `stream` (a cudaStream_t, NULL = legacy default
 *     stream).  Argument errors are detected on the host before any launch.
 *   - Device pointers must be 16-byte aligned (WQ_ERR_ALIGN otherwise).
 *   - Weights are row-major [out, in] (W in R^{d x k}, Y = W X, Eq. 1).
 *     Activations are token-major [m, features].  bf16 tensors are passed as
 *     `void*` holding IEEE bfloat16 values.
 *   - Quantized weights use the packed format described at wq_qweight.
 *   - Supported: group in {32, 64, 128}; in-features a multiple of the group
 *     (WQ_ERR_SHAPE otherwise); 1 <= m <= 16384 tokens (m == 0 is a no-op);
 *     LoRA rank r a multiple of 8, r <= 64 (r == 0: no adapter).
 *   - Two paths behind the same calls: up to 16 tokens (8 for layers of
 *     hidden size d >= 4096) the dequant-GEMV kernels (exact products of the
 *     codes and binary16 activations on the mma.sync tensor-core path, fp32
 *     sums); above that, and for a layer
 *     shape the GEMV kernels have no launch configuration for at the given
 *     token count, the batched dequant-GEMM on the tcgen05 tensor cores
 *     (activations and each dequantized weight s (q - z) rounded once to
 *     binary16, fp32 accumulation; with fp32 output of wq_down_w4 the weights
 *     enter as two exact binary16 parts).  The workspace size covers the path
 *     a call takes.
 *   - On error the call returns a negative wq_status and wq_last_error()
 *     describes it (per host thread).  Kernel-side waits are bounded; a wait
 *     that runs out records WQ_ERR_TIMEOUT, read back by wq_device_status().
 */
#ifndef WQ_H
#define WQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    WQ_OK = 0,
    WQ_ERR_ARG = -1,          /* null pointer, negative size, bad flag */
    WQ_ERR_SHAPE = -2,        /* shapes inconsistent or outside the supported set */
    WQ_ERR_ALIGN = -3,        /* a device pointer is not 16-byte aligned */
    WQ_ERR_UNSUPPORTED = -4,  /* valid request this library does not implement */
    WQ_ERR_CUDA = -5,         /* a CUDA runtime call or launch failed */
    WQ_ERR_TIMEOUT = -6,      /* a bounded device-side wait ran out */
    WQ_ERR_WORKSPACE = -7     /* workspace missing or smaller than required */
} wq_status;

/* Flags of wq_gateup_* and wq_mlp_forward. */
#define WQ_PRENORM 1u       /* unit-weight RMSNorm (eps 1e-6) of the MLP input first */
#define WQ_LAUNCH_CHAIN 2u  /* wq_mlp_forward*: run the per-layer launch chain even where the
                               single-launch stack kernel would be chosen (for tests and comparisons) */
#define WQ_LAUNCH_STACK 4u  /* wq_mlp_forward*: run the single-launch stack kernel wherever it can
                               take the stack (1..8 tokens, every layer with the same bits, groups
                               and rank), also where the launch chain is the measured-faster route */

/* Output element types of wq_down_w4. */
#define WQ_BF16 0
#define WQ_F32 1

/*
 * A group-quantized weight matrix W[n, k] (n output rows, k input features)
 * in the packed format (device memory, caller-owned):
 *
 *   Rows are padded to a multiple of 16 and k to a multiple of 128 with
 *   codes 0 and scales/zeros 0.  RT = ceil(n/16) row tiles, KB = ceil(k/128)
 *   feature blocks, NG = KB*128/group groups per row.
 *
 *   codes: uint32 words; block (rt, kb) of 16 rows x 128 features starts at
 *   word (rt*KB + kb) * WPB, WPB = 128 (bits 2), 192 (bits 3) or 256 (bits 4).
 *   The code of local row i and local feature c sits at
 *       lane = (i%8)*4 + (c%8)/2,  half = c%2
 *       bits 2: word = lane*4 + c/32,
 *               bit  = 16*half + 8*(i/8) + 2*(2*((c%32)/16) + (c%16)/8)
 *       bits 4: word = (c/64)*128 + lane*4 + (c%64)/16,
 *               bit  = 16*half + 8*(i/8) + 4*((c%16)/8)
 *       bits 3 (App. B's INT3 gate/up), two bit planes: code % 4 in words
 *               0..127 exactly where a 2-bit code sits, and code / 4 at
 *               word = 128 + lane*2 + (c/32)/2,
 *               bit  = 16*half + 8*((c/32)%2) + 2*(2*((c%32)/16) + (c%16)/8) + i/8
 *   so that one 16-byte load per lane (plus 8 bytes of the second plane for
 *   3 bits) yields that lane's m16n8k16 tensor-core A fragments for a whole
 *   128-feature block (64 codes of 2 or 3 bits) or a 64-feature half block
 *   (32 codes of 4 bits).
 *
 *   meta: binary16 scale s and zero z per (row, group): 32 values per
 *   (rt, group j) at (rt*NG + j)*32, for e = 0..7:
 *       [4e] = s[16rt+e], [4e+1] = s[16rt+e+8], [4e+2] = z[16rt+e], [4e+3] = z[16rt+e+8].
 *
 *   Dequantized weight: W[r, c] = s[r, c/group] * (code[r, c] - z[r, c/group]).
 */
typedef struct {
    uint32_t *codes;
    uint16_t *meta;
    int32_t n, k, group, bits;
} wq_qweight;

/* One gated-MLP layer: h = SiLU(gate x + a_g) * (up x + a_u), y = x + down h,
 * with the unmerged LoRA terms a_g = lora_scale * (x A_g^T) B_g^T and a_u likewise
 * (Eq. 1; alpha of Eq. 1 is lora_scale, e.g. alpha/r in the PEFT convention). */
typedef struct {
    wq_qweight gate, up, down;   /* gate/up: n = inter, k = d.  down: n = d, k = inter; in
                                    wq_mlp_forward* the down may also be dense bf16 (the BF16/W2-GateUp
                                    configuration, Sec. 6.1): bits = 16, codes = the bf16 [d, inter]
                                    matrix (inter a multiple of 32), meta and group unused */
    const void *lora_a;          /* bf16 [2r, d]: rows 0..r-1 = A_gate, r..2r-1 = A_up; NULL if r == 0 */
    const void *lora_b_gate;     /* bf16 [inter, r] */
    const void *lora_b_up;       /* bf16 [inter, r] */
    int32_t r;
    float lora_scale;
} wq_mlp_layer;

/* Sizes in bytes of the packed codes and meta buffers of an [n, k] matrix.
 * Returns WQ_ERR_SHAPE for an unsupported (bits, group) or k % group != 0. */
wq_status wq_packed_sizes(int bits, int n, int k, int group, size_t *code_bytes, size_t *meta_bytes);

/*
 * Stage-1 quantization and packing (Sec. 4.1 selective INT2 quantization of
 * gate/up; INT4 for the remaining layers, Sec. 3.3 and Sec. 7 step 4; INT3
 * for App. B's W3-GateUp variant): bits 2, 3 or 4.
 * Asymmetric min-max round-to-nearest per group of `group` consecutive input
 * features of each row, in IEEE fp32:
 *     s = fp16((max - min) / qmax)  (1.0 if that is zero),
 *     z = clamp(rint(-min / s), 0, qmax),  q = clamp(rint(w / s) + z, 0, qmax),
 * qmax = 2^bits - 1, rint ties-to-even, divisions IEEE-exact.
 *   w:         fp32 [n, k] row-major, device.
 *   out:       host struct whose codes/meta point to device buffers of the
 *              sizes wq_packed_sizes() gives; n, k, group, bits are filled in.
 *   nonfinite: optional device int; the kernel ORs 1 into it if any weight is
 *              NaN or infinite (the caller reads it after synchronizing).
 */
wq_status wq_pack(const float *w, int n, int k, int group, int bits, wq_qweight *out,
                  int *nonfinite, void *stream);
wq_status wq_pack_w2(const float *w, int n, int k, int group, wq_qweight *out, int *nonfinite, void *stream);
wq_status wq_pack_w4(const float *w, int n, int k, int group, wq_qweight *out, int *nonfinite, void *stream);

/*
 * Merged adapters (Sec. 4.2: once trained, the adapters may be merged into the
 * quantized weights instead of kept as a separate module; Sec. 7 step 5
 * deploys either form).  By Eq. 1 the merged matrix is deq(W) + alpha B A:
 *     W'[n, k] = fp32( s (q - z) + lora_scale * sum_rho B[n, rho] A[rho, k] ),
 * evaluated in fp64 (rho ascending, one rounding to fp32 at the end), then
 * quantized and packed exactly as wq_pack does, at the source's bits and
 * group.  The merged layer runs with r = 0 on the same calls.
 *   src:        packed source matrix (device buffers), bits 2 or 4.
 *   lora_b:     bf16 [n, r] row-major, device.  For gate: lora_b_gate.
 *   lora_a:     bf16 [r, k] row-major, device.  For gate: the first r rows of
 *               a layer's lora_a; for up: lora_a + r * k.
 *   r:          0..64 (0: W' = deq(W), which RTN maps back onto the source
 *               codes wherever a group holds both end codes).
 *   lora_scale: alpha of Eq. 1, finite.
 *   w_merged:   device fp32 [n, k] scratch, caller-owned, 16-byte aligned;
 *               holds W' afterwards.
 *   out:        as for wq_pack.  Either src itself (in place: in stream order
 *               the merge reads src completely before the quantizer writes)
 *               or buffers disjoint from src's.
 *   nonfinite:  optional device int, as for wq_pack.
 * Two launches on `stream`, no synchronization, no allocation.
 */
wq_status wq_merge_lora(const wq_qweight *src, const void *lora_b, const void *lora_a, int r, float lora_scale,
                        float *w_merged, wq_qweight *out, int *nonfinite, void *stream);

/*
 * Workspace (device scratch, caller-owned) needed by wq_gateup_*, wq_down_w4
 * and wq_mlp_forward for up to m tokens of a layer of hidden size d,
 * intermediate size inter and LoRA rank r, on the current device.  Before its
 * first use a workspace must be zero-filled (wq_workspace_init); every call
 * leaves its internal arrival counters at zero again (after a call whose
 * device status reads WQ_ERR_TIMEOUT, zero it again).  Calls that share a
 * workspace must not overlap in time on the GPU.
 */
size_t wq_workspace_bytes(int m, int d, int inter, int r);
wq_status wq_workspace_init(void *ws, size_t ws_bytes, void *stream);

/*
 * Fused 2-bit gate/up projection with unmerged LoRA and SiLU(gate) * up
 * (Eq. 1 on gate and up; gated MLP of Sec. 3.3; gate, activation and product
 * fused in one kernel as in the fused MLP modelling of Sec. 5):
 *     xin = (flags & WQ_PRENORM) ? x * rs : x,  rs = 1 / sqrt(mean(x^2) + 1e-6) per token
 *           (the normalized input is never stored, so it is not rounded)
 *     g   = xin deq(Wg)^T + lora_scale * (xin A_g^T) B_g^T      (fp32 accumulate)
 *     u   = xin deq(Wu)^T + lora_scale * (xin A_u^T) B_u^T
 *     h   = bf16( g / (1 + exp(-g)) * u )
 *   x: bf16 [m, d].  gate, up: bits 2, n = inter, k = d.  lora_*: see
 *   wq_mlp_layer (r == 0 and NULLs: no adapter).  h: bf16 [m, inter].
 */
wq_status wq_gateup_w2_lora(const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                            const void *lora_a, const void *lora_b_gate, const void *lora_b_up,
                            int r, float lora_scale, unsigned flags, void *h,
                            void *ws, size_t ws_bytes, void *stream);

/*
 * wq_gateup_w2_lora without a workspace argument, for callers that cannot
 * allocate device memory: code that runs where cudaMalloc is not allowed or
 * not wanted (inside a host callback, between the launches of an engine whose
 * memory is fully planned ahead, under an allocator that owns every device
 * buffer), or a plugin that must not grow its host process's memory.  The
 * paper has no counterpart to this call; it is a deployment convenience.
 *
 * Same arguments and results as wq_gateup_w2_lora minus ws / ws_bytes, for
 * the decode token counts of the dequant-GEMV path (1 <= m <= 16, or 8 for
 * d >= 4096).  The scratch
 * it needs (per-16-feature RMSNorm and LoRA-A partial sums of x, split-K
 * partial sums and arrival counters) lives in a fixed array of
 * WQ_NOALLOC_SCRATCH_BYTES bytes inside the library, which every GPU that
 * loads the library keeps until the process exits.  It returns
 * WQ_ERR_UNSUPPORTED and launches nothing when
 *   - m above the dequant-GEMV path's limit (wq_gateup_w2_lora takes the
 *     dequant-GEMM path there),
 *   - the layer shape has no dequant-GEMV launch configuration at this m
 *     (wq_gateup_w2_lora takes the dequant-GEMM path for it), or
 *   - the layer needs more scratch than the array holds.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress, which may load the library's device code); make
 *     that first call before any stream capture.  The address is kept for
 *     the life of the process: do not use this call on a device after a
 *     device reset (cudaDeviceReset) in the same process.
 *   - Every call clears the array's arrival counters (cudaMemsetAsync on
 *     `stream`) and then reuses the array, which keeps the previous call's
 *     contents otherwise.  All calls share the one array: calls that can
 *     overlap on the GPU (different streams, or different host threads
 *     without ordering) race with each other and must be serialized by the
 *     caller.
 * The call allocates nothing: no cudaMalloc, cudaFree or allocating library
 * routine.
 */
#define WQ_NOALLOC_SCRATCH_BYTES (4u << 20)
wq_status wq_gateup_w2_lora_noalloc(const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                                    const void *lora_a, const void *lora_b_gate, const void *lora_b_up,
                                    int r, float lora_scale, unsigned flags, void *h, void *stream);

/*
 * App. B's W3-GateUp variant: wq_gateup_w2_lora with 3-bit gate/up codes
 * (bits 3, two bit planes; same arguments, same arithmetic).  Runs on the
 * dequant-GEMV kernels at every token count up to 64 (WQ_ERR_UNSUPPORTED
 * above: the dequant-GEMM path takes 2- and 4-bit codes).
 */
wq_status wq_gateup_w3_lora(const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                            const void *lora_a, const void *lora_b_gate, const void *lora_b_up,
                            int r, float lora_scale, unsigned flags, void *h,
                            void *ws, size_t ws_bytes, void *stream);

/* The uniform-W4 comparator: the same block with 4-bit gate/up and no LoRA. */
wq_status wq_gateup_w4(const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                       unsigned flags, void *h, void *ws, size_t ws_bytes, void *stream);

/*
 * 4-bit down projection with optional residual (Sec. 3.3: down stays INT4):
 *     y = residual + h deq(Wd)^T
 *   h: bf16 [m, inter].  down: bits 4, n = d, k = inter.  residual: bf16
 *   [m, d] or NULL.  y: [m, d] of y_dtype (WQ_BF16 rounds to nearest even,
 *   WQ_F32 stores the fp32 accumulator).
 */
wq_status wq_down_w4(const void *h, int m, const wq_qweight *down, const void *residual,
                     void *y, int y_dtype, void *ws, size_t ws_bytes, void *stream);

/*
 * bf16 down projection with optional residual: the down layer of the
 * BF16/W2-GateUp configuration that the accuracy experiments use (Sec. 6.1:
 * gate/up at INT2, every other layer in BF16; Sec. 7):
 *     y = residual + h Wd^T
 *   h:  bf16 [m, inter].  wd: bf16 [d, inter] row-major (device, 16-byte
 *   aligned), inter a multiple of 32.  residual: bf16 [m, d] or NULL.
 *   y:  [m, d] of y_dtype (as for wq_down_w4).
 * Needs no workspace; one launch on `stream`.  Products are exact, sums fp32.
 */
wq_status wq_down_bf16(const void *h, int m, const void *wd, int d, int inter, const void *residual, void *y,
                       int y_dtype, void *stream);

/*
 * A stack of gated-MLP layers for one decode step of m tokens:
 *     x_0 = x,  x_{l+1} = x_l + down_l( SiLU(gate_l(xin_l)) * up_l(xin_l) ),  y = x_L
 * with xin_l = RMSNorm(x_l) (unrounded, as in wq_gateup_w2_lora) when flags has
 * WQ_PRENORM, else x_l.  Each layer's gate/up are 2-bit or 3-bit (App. B; with
 * LoRA) or 4-bit (no LoRA); down is 4-bit (or dense bf16, see wq_mlp_layer).
 * Stacks with 3-bit gate/up take the launch chain at every token count up to
 * 64 (above: WQ_ERR_UNSUPPORTED).  x, y: bf16 [m, d]; the residual stream is stored
 * in bf16 between layers.  Three routes, chosen per call (wq_mlp_forward_info
 * reports which):
 *   - the single-launch stack kernel: every layer in one cooperative launch
 *     (one CTA per SM; up to 32 layers a launch), for 1..8 tokens when every
 *     layer has the same bits, groups and rank, where it is the measured-faster
 *     route (2-bit gate/up at 2..8 tokens, or d >= 4096) or WQ_LAUNCH_STACK asks;
 *   - the launch chain: 2 kernels per layer (plus one for the first layer's
 *     input statistics) with programmatic dependent launch, each down launch
 *     also producing the next layer's RMSNorm and LoRA-A partial sums;
 *   - the dequant-GEMM chain above 16 tokens (8 for d >= 4096).
 * Every route can be captured into a CUDA graph.
 */
wq_status wq_mlp_forward(const void *x, int m, const wq_mlp_layer *layers, int n_layers,
                         unsigned flags, void *y, void *ws, size_t ws_bytes, void *stream);

/*
 * One decode step of grouped-query attention over a bf16 KV cache: the
 * decoder-layer operator around the MLP block whose cost Sec. 5 counts as
 * independent of the weight precision (Sec. 7 step 4 puts its projections at
 * INT4).  Per sequence b (one new token) and query head h (kv head
 * g = h / (n_heads / n_kv)):
 *   rs  = 1 / sqrt(mean(x[b]^2) + 1e-6)           (the layer input's RMSNorm)
 *   q_h = RoPE(headnorm(rs qkv[b, q_h])), k_g = RoPE(headnorm(rs qkv[b, k_g])),
 *   v_g = rs qkv[b, v_g]; k_g, v_g rounded to bf16 and written to the caches at
 *   position lens[b]; headnorm: unit-weight RMSNorm over the head (eps 1e-6);
 *   RoPE: element i with i + head_dim/2, angle lens[b] theta^(-2i/head_dim);
 *   o[b, h] = bf16( softmax_j(q_h . K[b,g,j] / sqrt(head_dim)) V[b,g,j] ), j = 0..lens[b].
 *   qkv:     fp32 [batch, (n_heads + 2 n_kv) head_dim] = x deq(Wqkv)^T before the
 *            RMSNorm scale (e.g. wq_down_w4 with WQ_F32 on the rows of Wq, Wk, Wv).
 *   x:       bf16 [batch, d], the layer input.
 *   lens:    int32 [batch] on the device: positions already cached.  A length
 *            outside [0, max_len) skips that sequence and records WQ_ERR_ARG in
 *            the device status (wq_device_status).
 *   caches:  bf16 [batch, n_kv, max_len, head_dim].  o: bf16 [batch, n_heads head_dim].
 *   Supported: head_dim 64 or 128, n_heads a multiple of n_kv, n_heads / n_kv <= 8.
 *   Workspace: wq_attn_workspace_bytes (split partial results, no zeroing needed).
 */
size_t wq_attn_workspace_bytes(int batch, int n_heads, int n_kv, int head_dim, int max_len);
wq_status wq_attn_decode(const float *qkv, const void *x, const int32_t *lens, int batch, int d, int n_heads,
                         int n_kv, int head_dim, float theta, void *k_cache, void *v_cache, int max_len, void *o,
                         void *ws, size_t ws_bytes, void *stream);

/* A decoder layer: 4-bit attention projections around the MLP block. */
typedef struct {
    wq_qweight qkv;        /* bits 4, [(n_heads + 2 n_kv) head_dim, d]: the rows of Wq, then Wk, then Wv */
    wq_qweight o;          /* bits 4, [d, n_heads head_dim] */
    wq_mlp_layer mlp;
    int32_t n_heads, n_kv, head_dim;
    float rope_theta;
} wq_decoder_layer;

/*
 * One decode step of a decoder layer for `batch` sequences:
 *   qkv = x deq(Wqkv)^T (fp32), o = wq_attn_decode(...), x1 = bf16(x + o deq(Wo)^T),
 *   y = the MLP block on x1 (as wq_gateup_* then wq_down_w4 with residual x1;
 *   flags as for wq_mlp_forward, WQ_PRENORM for the MLP's RMSNorm).
 * Five calls on `stream`; the caches gain position lens[b] (lens is not changed).
 * Workspace: wq_decoder_workspace_bytes, zero-filled before first use (wq_workspace_init).
 */
size_t wq_decoder_workspace_bytes(int batch, const wq_decoder_layer *layer, int max_len);
wq_status wq_decoder_layer_forward(const void *x, int batch, const int32_t *lens, const wq_decoder_layer *layer,
                                   void *k_cache, void *v_cache, int max_len, unsigned flags, void *y, void *ws,
                                   size_t ws_bytes, void *stream);

/*
 * A mixture-of-experts MLP block (the MoE model of Sec. 5: a router picks a
 * few experts per token, so a decode step reads only those experts' weights,
 * which is how expert routing shrinks the realized gain of the 2-bit gate/up).
 * Each expert is a gated MLP of wq_mlp_layer form; the E experts' matrices
 * are stacked row-wise and packed as one matrix each:
 *   experts.gate, experts.up: n = E * inter, k = d (expert e: rows e*inter ..
 *                             e*inter + inter - 1); bits 2 (bits 4, r = 0: the
 *                             uniform-W4 comparator);
 *   experts.down:             bits 4, n = E * d, k = inter;
 *   experts.lora_a:           bf16 [E][2r][d]; lora_b_gate, lora_b_up: bf16 [E * inter][r].
 *   d and inter multiples of 16; 1 <= top_k <= min(E, 16); E <= 256.
 */
typedef struct {
    wq_mlp_layer experts;
    int32_t n_experts, top_k;
} wq_moe_layer;

/*
 * One MoE block for m tokens (1 <= m <= 64; m == 0 is a no-op):
 *   1. routing: per token t, the top_k experts by router logit, the larger
 *      logit first and the lower expert index first among equal logits; their
 *      weights w_j = softmax over the selected logits (fp32);
 *   2. per slot (t, j): h = the gate/up of expert e_j on x[t] (the arithmetic
 *      of wq_gateup_w2_lora, RMSNorm with WQ_PRENORM), y_j = h deq(Wd_e)^T (fp32);
 *   3. y[t] = bf16(x[t] + sum_j w_j y_j), j in order (fp32).
 *   x: bf16 [m, d].  logits: fp32 [m, E], finite.  y: bf16 [m, d].
 *   expert_idx (int32 [m, top_k]), expert_w (fp32 [m, top_k]), h_slots
 *   (bf16 [m top_k, inter]) and y_slots (fp32 [m top_k, d]): optional device
 *   outputs of steps 1-2, slot t*top_k + j (NULL: kept in the workspace).
 * Four launches on `stream` (routing with the tile partials, gate/up and down
 * over the slots, combine); only the selected experts' weights are read.
 * Workspace: wq_moe_workspace_bytes for this layer, token count and flags,
 * zero-filled before first use (wq_workspace_init).
 */
size_t wq_moe_workspace_bytes(int m, const wq_moe_layer *layer, unsigned flags);
wq_status wq_moe_forward(const void *x, int m, const float *logits, const wq_moe_layer *layer, unsigned flags,
                         void *y, int32_t *expert_idx, float *expert_w, void *h_slots, float *y_slots, void *ws,
                         size_t ws_bytes, void *stream);

/*
 * Self-check of the kernels' bounded waits (failure detection without a GPU
 * fault): one launch whose single CTA waits, with the library's own wait
 * routines, on an mbarrier that nothing arrives on and at a grid barrier that
 * nothing advances.  Each wait gives up after its limit (2 s), records
 * WQ_ERR_TIMEOUT and lets the launch end; wq_device_status() then returns
 * WQ_ERR_TIMEOUT and the context stays usable.  About 4 s on `stream`.
 */
wq_status wq_wait_check(void *stream);

/*
 * wq_mlp_forward that also returns every layer's output (the hidden states of
 * the stack) and, optionally, every layer's MLP activation h:
 *   states:   bf16 [n_layers][m][d] (device, 16-byte aligned), states[l] = x_{l+1};
 *   h_states: bf16 [n_layers][m][inter] or NULL, h_states[l] = layer l's
 *             h = SiLU(g) * u as stored for its down projection.
 * y receives x_L as well.  Same launches as wq_mlp_forward with each layer
 * writing into its own slots, plus one device-to-device copy of the last
 * slot into y.
 */
wq_status wq_mlp_forward_states(const void *x, int m, const wq_mlp_layer *layers, int n_layers,
                                unsigned flags, void *y, void *states, void *h_states, void *ws, size_t ws_bytes,
                                void *stream);

/*
 * How wq_mlp_forward runs this stack on the current device (for tests and
 * tuning; validates like wq_mlp_forward and launches nothing).  info[16]:
 *   [0]      route: 0 = per-layer dequant-GEMV launch chain,
 *                   1 = per-layer dequant-GEMM launch chain,
 *                   2 = single-launch stack kernel
 *   [1..6]   route 0: layer 0's gate/up launch: row tiles per CTA, blocks per
 *            panel, warps along k, row tiles per warp, panels, CTAs
 *   [7..12]  route 0: layer 0's down launch (writing layer 1's partial sums
 *            when there is a layer 1): the same fields
 *   [13]     route 0: 1 when the gate/up launch hands the down launch its
 *            ready binary16 panel of h
 *   [1..7]   route 2: CTAs, ring stages, stage bytes, 1 when the down slices
 *            need other CTAs' h (a grid barrier before each down phase), warps
 *            per gate/up row tile, gate/up row tiles per CTA, shared memory bytes
 *   other entries: -1
 */
wq_status wq_mlp_forward_info(int m, const wq_mlp_layer *layers, int n_layers, unsigned flags, int64_t info[16]);

/*
 * Describes how a dequant-GEMV launch of the current device splits its work
 * (for tests and tuning; launches nothing).  kind: 0 = 2-bit gate/up,
 * 1 = 4-bit gate/up, 2 = 4-bit down.  n, k: matrix shape; m tokens; r LoRA
 * rank.  info[0..9] receives: row tiles, 128-feature blocks, row tiles per
 * CTA, blocks per panel, warps along k, panels, CTAs, threads per CTA,
 * dynamic shared memory bytes, tokens per MMA chunk.
 */
wq_status wq_plan_info(int kind, int n, int k, int m, int group, int r, int64_t info[10]);

/* Message of the last error returned on this host thread ("" if none). */
const char *wq_last_error(void);

/* Reads and clears the device-side status words of the current device: WQ_OK,
 * WQ_ERR_TIMEOUT (a bounded wait ran out) or WQ_ERR_ARG (wq_attn_decode met a
 * sequence length outside its cache).  Synchronizes the device. */
wq_status wq_device_status(int *status);

/* Library version string. */
const char *wq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* WQ_H */
