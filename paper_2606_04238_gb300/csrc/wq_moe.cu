// wq_moe.cu -- the routing and combining steps of a mixture-of-experts MLP
// block (sm_103a).  Sec. 5 analyses an MoE model whose router activates a
// few experts per token, so a decode step reads only those experts' weights.
//
// A step is four launches joined by programmatic dependent launch:
//   1. moe_prep_kernel: per token, the top_k experts by router logit and
//      their softmax weights; per slot (token t, choice j) -> s = t*top_k + j,
//      the tile partials of x[t] the gate/up epilogue needs (sum x^2 for the
//      RMSNorm, A_e x for the adapter of the slot's expert e);
//   2. the gate/up dequant-GEMV over the slots (qgemv_slots_kernel, one token
//      and one expert each) -> h per slot;
//   3. the down dequant-GEMV over the slots -> y_j per slot in fp32;
//   4. moe_combine_kernel: y[t] = bf16(x[t] + sum_j w_j y_j), j in order.
#include <climits>
#include <cstdint>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "wq_internal.h"
#include "wq_ptx.cuh"

namespace wq {

namespace {

constexpr int kMoeMaxExperts = 256;
constexpr int kMoeMaxTopK = 16;
constexpr int kPrepWarps = 8;  // tiles of 16 features a CTA of moe_prep_kernel takes

__device__ __forceinline__ void unpack8(const uint4 v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

// (logit, expert) a ranks before (logit, expert) b: the larger logit first,
// the lower expert index among equal logits.
__device__ __forceinline__ bool ranks_before(float la, int ea, float lb, int eb) {
  return la > lb || (la == lb && ea < eb);
}

// grid (ceil(ntp / 8), slots), 256 threads.  Every CTA routes its own token
// (a few hundred comparisons), so no launch or exchange separates the routing
// from the tile partials.
__global__ void __launch_bounds__(kPrepWarps * 32) moe_prep_kernel(const __nv_bfloat16 *x, int d,
                                                                   const float *logits, int E, int top_k,
                                                                   const __nv_bfloat16 *lora_a, int r2, float *tp,
                                                                   int *idx_out, float *w_out) {
  __shared__ int sel_s[kMoeMaxTopK];
  __shared__ float w_s[kMoeMaxTopK];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int slot = blockIdx.y, t = slot / top_k, j = slot % top_k;
  pdl_launch_dependents();
  pdl_wait();  // x and the logits may come from the previous launch
  if (warp == 0) {
    // lane l holds experts l, l + 32, ..: taken ones are marked by clearing their bit
    constexpr int PER = kMoeMaxExperts / 32;
    float lg[PER];
    uint32_t live = 0u;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int e = lane + 32 * i;
      lg[i] = e < E ? __ldcg(logits + (size_t)t * E + e) : 0.f;
      if (e < E) live |= 1u << i;
    }
    float sel_l[kMoeMaxTopK];
    for (int c = 0; c < top_k; ++c) {
      float bl = 0.f;
      int be = INT_MAX;
#pragma unroll
      for (int i = 0; i < PER; ++i)
        if (((live >> i) & 1u) && (be == INT_MAX || ranks_before(lg[i], lane + 32 * i, bl, be))) {
          bl = lg[i];
          be = lane + 32 * i;
        }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float ol = __shfl_xor_sync(0xffffffffu, bl, o);
        const int oe = __shfl_xor_sync(0xffffffffu, be, o);
        if (oe != INT_MAX && (be == INT_MAX || ranks_before(ol, oe, bl, be))) {
          bl = ol;
          be = oe;
        }
      }
      if (be != INT_MAX && (be & 31) == lane) live &= ~(1u << (be >> 5));
      sel_l[c] = bl;  // top_k <= kMoeMaxTopK (checked by the launcher)
      if (lane == 0) sel_s[c] = be;
    }
    if (lane == 0) {
      // softmax over the selected logits, the largest (the first) subtracted
      float sum = 0.f;
      for (int c = 0; c < top_k; ++c) {
        w_s[c] = expf(sel_l[c] - sel_l[0]);
        sum += w_s[c];
      }
      for (int c = 0; c < top_k; ++c) w_s[c] = __fdiv_rn(w_s[c], sum);
    }
  }
  __syncthreads();
  const int e = sel_s[j];
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    idx_out[slot] = e;
    w_out[slot] = w_s[j];
  }
  if (tp == nullptr) return;
  // tile partials of x[t] for expert e: the arithmetic of tile_prep_kernel
  const int ntp = d / 16, tile = blockIdx.x * kPrepWarps + warp;
  if (tile >= ntp) return;
  const int Q = 1 + r2, Qp = (Q + 3) & ~3;
  float v[16];
  {
    const uint8_t *xr = reinterpret_cast<const uint8_t *>(x) + ((size_t)t * d + (size_t)tile * 16) * 2;
    unpack8(ldg_cg128(xr), *reinterpret_cast<float(*)[8]>(v));
    unpack8(ldg_cg128(xr + 16), *reinterpret_cast<float(*)[8]>(v + 8));
  }
  const uint8_t *ae = reinterpret_cast<const uint8_t *>(lora_a) + (size_t)e * r2 * d * 2;
  float *out = tp + ((size_t)slot * ntp + tile) * Qp;
  for (int q = lane; q < Qp; q += 32) {
    float s = 0.f;
    if (q == 0) {
#pragma unroll
      for (int c = 0; c < 16; ++c) s = fmaf(v[c], v[c], s);
    } else if (q < Q) {
      const uint8_t *ar = ae + ((size_t)(q - 1) * d + (size_t)tile * 16) * 2;
      float w[16];
      unpack8(__ldg(reinterpret_cast<const uint4 *>(ar)), *reinterpret_cast<float(*)[8]>(w));
      unpack8(__ldg(reinterpret_cast<const uint4 *>(ar + 16)), *reinterpret_cast<float(*)[8]>(w + 8));
#pragma unroll
      for (int c = 0; c < 16; ++c) s = fmaf(w[c], v[c], s);
    }
    out[q] = s;
  }
}

// y[t][n] = bf16(x[t][n] + sum_j w[t*k + j] ys[t*k + j][n]), j in order
// (fp32 fma chain); eight features a thread.
__global__ void __launch_bounds__(256) moe_combine_kernel(const __nv_bfloat16 *x, int m, int d, int top_k,
                                                          const float *w, const float *ys, __nv_bfloat16 *y) {
  pdl_launch_dependents();
  pdl_wait();
  const int per_tok = d / 8;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= m * per_tok) return;
  const int t = i / per_tok, n0 = (i % per_tok) * 8;
  float acc[8];
  unpack8(ldg_cg128(reinterpret_cast<const uint8_t *>(x) + ((size_t)t * d + n0) * 2), acc);
  for (int c = 0; c < top_k; ++c) {
    const int s = t * top_k + c;
    const float ws = __ldcg(w + s);
    const float *yr = ys + (size_t)s * d + n0;
    const float4 a = __ldcg(reinterpret_cast<const float4 *>(yr));
    const float4 b = __ldcg(reinterpret_cast<const float4 *>(yr + 4));
    const float yv[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int u = 0; u < 8; ++u) acc[u] = fmaf(ws, yv[u], acc[u]);
  }
  uint32_t o[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * u]));
    const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * u + 1]));
    o[u] = lo | (hi << 16);
  }
  *reinterpret_cast<uint4 *>(reinterpret_cast<uint8_t *>(y) + ((size_t)t * d + n0) * 2) = make_uint4(o[0], o[1], o[2], o[3]);
}

cudaLaunchConfig_t pdl_config(dim3 grid, dim3 block, cudaStream_t s, cudaLaunchAttribute *attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

}  // namespace

int moe_max_experts() { return kMoeMaxExperts; }
int moe_max_top_k() { return kMoeMaxTopK; }

cudaError_t launch_moe_prep(const void *x, int m, int d, const float *logits, int E, int top_k, const void *lora_a,
                            int r2, float *tp, int *idx, float *w, cudaStream_t s) {
  if (E < 1 || E > kMoeMaxExperts || top_k < 1 || top_k > kMoeMaxTopK || top_k > E || d % 16 != 0)
    return cudaErrorInvalidValue;
  const int slots = m * top_k;
  const int gx = tp != nullptr ? (d / 16 + kPrepWarps - 1) / kPrepWarps : 1;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pdl_config(dim3(gx, slots), dim3(kPrepWarps * 32), s, attr);
  return cudaLaunchKernelEx(&cfg, moe_prep_kernel, reinterpret_cast<const __nv_bfloat16 *>(x), d, logits, E, top_k,
                            reinterpret_cast<const __nv_bfloat16 *>(lora_a), r2, tp, idx, w);
}

cudaError_t launch_moe_combine(const void *x, int m, int d, int top_k, const float *w, const float *ys, void *y,
                               cudaStream_t s) {
  if (d % 8 != 0) return cudaErrorInvalidValue;
  const int n = m * (d / 8);
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pdl_config(dim3((n + 255) / 256), dim3(256), s, attr);
  return cudaLaunchKernelEx(&cfg, moe_combine_kernel, reinterpret_cast<const __nv_bfloat16 *>(x), m, d, top_k, w,
                            ys, reinterpret_cast<__nv_bfloat16 *>(y));
}

}  // namespace wq
