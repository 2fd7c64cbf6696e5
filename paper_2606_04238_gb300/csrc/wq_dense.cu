// wq_dense.cu -- bf16 down projection with residual (sm_103a):
//     y[t, n] = residual[t, n] + sum_k h[t, k] Wd[n, k],
// the down layer of the BF16/W2-GateUp configuration that the accuracy
// experiments use (Sec. 6.1: gate/up at INT2, every other layer in BF16;
// Sec. 7 names it beside the deployed W4/W2-GateUp form).
//
// Decode-sized token counts make this a weight stream (2 bytes a weight, read
// once), so the kernel is written for HBM: every lane keeps several 16-byte
// loads of Wd in flight, Wd is loaded with the streaming cache hint, and the
// products run on bf16 m16n8k16 MMAs (exact products, fp32 sums) with Wd as
// the 16-row A operand and 8 tokens as the B operand.
//
// The launch is programmatic-dependent: the first step's loads of Wd are issued
// before griddepcontrol.wait (they do not depend on the previous kernel), h and
// the residual only after it, through L2 (ld.global.cg: a read-only-path load
// could be moved above the wait and see h before the previous kernel wrote
// it), and the next launch is let in once this one's inputs are readable, so
// its weight stream overlaps this launch's tail.
//
// A CTA owns one tile of 16 output rows and 16 tokens; its 8 warps split the
// input features into 8 contiguous ranges of 32-feature chunks and their fp32
// partial sums are added in warp order in shared memory (deterministic, no
// workspace).  A lane loads features 8t..8t+7 of a chunk (16 bytes) of rows g
// and g + 8 and of token g, and feeds features 0..3 and 4..7 of them to two
// k-steps in the slots of k 2t, 2t+1, 2t+8, 2t+9: the same permutation of k on
// both operands, so the sums are unchanged.
#include <cuda_bf16.h>

#include "wq_ptx.cuh"
#include "wq_launch.h"

namespace wq {
namespace {

constexpr int kDnWarps = 8;

__device__ __forceinline__ uint32_t u4word(const uint4 &v, int q) {
  return q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w;
}

// NT token tiles of 8; U 32-feature chunks of loads in flight per step (8 for
// up to 8 tokens, 4 for 16: the register budget of 2 CTAs an SM)
template <int NT, int U>
__global__ void __launch_bounds__(kDnWarps * 32, 2)
    down_bf16_kernel(const __nv_bfloat16 *h, int m, const __nv_bfloat16 *__restrict__ w, int d, int K,
                     const __nv_bfloat16 *res, void *__restrict__ y, int y_f32) {
  __shared__ float part[kDnWarps][16][17];  // [warp][row][token]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, g = lane >> 2, t = lane & 3;
  const int r0 = blockIdx.x * 16, m0 = blockIdx.y * 16;
  const int nchunk = K / 32;
  const int c_lo = nchunk * warp / kDnWarps, c_hi = nchunk * (warp + 1) / kDnWarps;
  const bool ra = r0 + g < d, rb = r0 + g + 8 < d;
  const uint4 *wa = reinterpret_cast<const uint4 *>(w + (size_t)(ra ? r0 + g : 0) * K + 8 * t);
  const uint4 *wb = reinterpret_cast<const uint4 *>(w + (size_t)(rb ? r0 + g + 8 : 0) * K + 8 * t);
  const uint4 *hp[NT];
  bool tin[NT];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int tok = m0 + 8 * nt + g;
    tin[nt] = tok < m;
    hp[nt] = reinterpret_cast<const uint4 *>(h + (size_t)(tin[nt] ? tok : 0) * K + 8 * t);
  }
  float acc[NT][4];
#pragma unroll
  for (int i = 0; i < NT * 4; ++i) acc[i / 4][i % 4] = 0.f;
  const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
  for (int c = c_lo; c < c_hi || c == c_lo; c += U) {
    uint4 va[U], vb[U], vh[U][NT];
#pragma unroll
    for (int u = 0; u < U; ++u) {  // every load of the step first (chunk cc = 4 uint4 of a row)
      const int cc = c + u;
      const bool in = cc < c_hi;
      va[u] = in && ra ? __ldcs(wa + 4 * cc) : zero;
      vb[u] = in && rb ? __ldcs(wb + 4 * cc) : zero;
    }
    if (c == c_lo) {  // the weights of the first step are in flight: now wait for the previous kernel
      pdl_wait();
      pdl_launch_dependents();
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int cc = c + u;
      const bool in = cc < c_hi;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) vh[u][nt] = in && tin[nt] ? ldg_cg128(hp[nt] + 4 * cc) : zero;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (c + u >= c_hi) break;  // the same for the whole warp
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        // A: rows g / g + 8, k slots 2t, 2t+1 (features 4hh, 4hh+1 of the lane's 8) and 2t+8, 2t+9 (4hh+2, 4hh+3)
        const uint32_t af[4] = {u4word(va[u], 2 * hh), u4word(vb[u], 2 * hh), u4word(va[u], 2 * hh + 1),
                                u4word(vb[u], 2 * hh + 1)};
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          mma_bf16_16816(acc[nt], af, u4word(vh[u][nt], 2 * hh), u4word(vh[u][nt], 2 * hh + 1));
      }
    }
  }
  // accumulator (row, token) of n-tile nt: rows g / g + 8, tokens 8 nt + 2t, 2t + 1
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    part[warp][g][8 * nt + 2 * t] = acc[nt][0];
    part[warp][g][8 * nt + 2 * t + 1] = acc[nt][1];
    part[warp][g + 8][8 * nt + 2 * t] = acc[nt][2];
    part[warp][g + 8][8 * nt + 2 * t + 1] = acc[nt][3];
  }
  __syncthreads();
  // one (token, row) per thread, rows fastest: the stores of a token are contiguous
  for (int o = tid; o < 8 * NT * 16; o += kDnWarps * 32) {
    const int tl = o >> 4, rl = o & 15;
    const int tok = m0 + tl, row = r0 + rl;
    if (tok >= m || row >= d) continue;
    float v = 0.f;
#pragma unroll
    for (int wi = 0; wi < kDnWarps; ++wi) v += part[wi][rl][tl];
    const size_t at = (size_t)tok * d + row;
    if (res != nullptr) v = __fadd_rn(__bfloat162float(__ldcg(res + at)), v);
    if (y_f32)
      static_cast<float *>(y)[at] = v;
    else
      static_cast<__nv_bfloat16 *>(y)[at] = __float2bfloat16_rn(v);
  }
}

}  // namespace

cudaError_t launch_down_bf16(const void *h, int m, const void *wd, int d, int inter, const void *residual, void *y,
                             bool y_f32, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((d + 15) / 16), (unsigned)((m + 15) / 16));
  cfg.blockDim = dim3(kDnWarps * 32);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const auto *hb = static_cast<const __nv_bfloat16 *>(h);
  const auto *wb = static_cast<const __nv_bfloat16 *>(wd);
  const auto *rb = static_cast<const __nv_bfloat16 *>(residual);
  const int yf = y_f32 ? 1 : 0;
  if (m <= 8) return cudaLaunchKernelEx(&cfg, down_bf16_kernel<1, 8>, hb, m, wb, d, inter, rb, y, yf);
  return cudaLaunchKernelEx(&cfg, down_bf16_kernel<2, 4>, hb, m, wb, d, inter, rb, y, yf);
}

}  // namespace wq
