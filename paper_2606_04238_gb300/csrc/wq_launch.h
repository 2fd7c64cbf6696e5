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

}  // namespace wq
