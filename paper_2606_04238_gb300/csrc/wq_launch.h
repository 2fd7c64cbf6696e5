// wq_launch.h -- launchers of the calls outside the decode chain: the adapter
// merge (wq_pack.cu) and the bf16 down projection (wq_dense.cu).  Both take
// arguments the C ABI has already validated and return the launch status.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

namespace wq {

// w[n, k] = fp32(deq(src) + alpha * B A) from a packed source (codes, meta) of
// `bits`; B bf16 [n, r], A bf16 [r, k].
cudaError_t launch_merge_lora(const uint32_t *codes, const uint16_t *meta, int n, int k, int group, int bits,
                              const void *lora_b, const void *lora_a, int r, float alpha, float *w,
                              cudaStream_t stream);

// y[m, d] = residual + h Wd^T with h bf16 [m, inter], Wd bf16 [d, inter].
cudaError_t launch_down_bf16(const void *h, int m, const void *wd, int d, int inter, const void *residual, void *y,
                             bool y_f32, cudaStream_t stream);

// One decode step of grouped-query attention (wq_attn.cu): qkv fp32
// [B][(H + 2 Hkv) HD] projections of x (not yet RMSNorm-scaled), x bf16 [B][d],
// lens [B] device ints, caches bf16 [B][Hkv][max_len][HD] (the new k, v
// written at lens[b]), part fp32 [B][H][S][HD + 2], o bf16 [B][H HD].
cudaError_t launch_attn_decode(const float *qkv, const void *x, const int *lens, int B, int d, int H, int Hkv, int HD,
                               double theta, void *k_cache, void *v_cache, int max_len, float *part, int S, void *o,
                               cudaStream_t s);
// Context splits of a launch (S above).
int attn_splits(int B, int Hkv, int max_len, int num_sms);
// Reads and clears the attention kernels' device status word.
cudaError_t read_attn_status(int *status);

// Mixture-of-experts steps (wq_moe.cu).  Routing and tile partials: per
// token t of x bf16 [m][d], the top_k of the E fp32 logits [m][E] (larger
// first, lower index among equal ones) -> idx [m*top_k] and softmax weights
// w [m*top_k]; with tp non-null, per slot s = t*top_k + j the tile partials
// of x[t] for expert idx[s] (sum x^2 and the r2 rows of lora_a + idx[s]*r2*d)
// at tp + s*(d/16)*stride.  Combine: y[t] = bf16(x[t] + sum_j w ys[t*top_k + j]).
cudaError_t launch_moe_prep(const void *x, int m, int d, const float *logits, int E, int top_k, const void *lora_a,
                            int r2, float *tp, int *idx, float *w, cudaStream_t s);
cudaError_t launch_moe_combine(const void *x, int m, int d, int top_k, const float *w, const float *ys, void *y,
                               cudaStream_t s);
int moe_max_experts();
int moe_max_top_k();

}  // namespace wq
