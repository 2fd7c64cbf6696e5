// wq_attn.cu -- one decode step of grouped-query attention over a bf16 KV
// cache (sm_103a), the decoder-layer operator around the paper's MLP block
// whose cost Sec. 5 counts as independent of the weight precision.
//
// Per sequence b (one new token at position lens[b]) and kv head g:
//   1. rs = 1/sqrt(mean(x[b]^2) + eps): the layer input's RMSNorm scale,
//      applied to the projections (the normalized input is never rounded);
//   2. q heads h of the group, k and v of g: the fp32 projections x deq(W)^T
//      times rs; q and k normalized per head (unit-weight RMSNorm) and rotated
//      (RoPE, element i with i + hd/2, angle pos theta^(-2i/hd): the
//      frequencies come from the host in fp64, the angle is formed and reduced
//      modulo 2 pi in fp64 -- a few fp64 operations a CTA -- and its cosine
//      and sine taken in fp32 on the reduced argument);
//   3. k and v rounded to bf16 and appended to the cache at lens[b];
//   4. o = softmax(q K^T / sqrt(hd)) V over positions 0..lens[b].
// The context is cut into S splits (grid.y); a CTA of 8 warps takes one
// (b, g) and one split; each warp takes chunks of 8 positions, the lanes the
// head dimension.  A warp copies its next chunk's K and V rows into a shared-
// memory buffer of its own (cp.async, 16 bytes a lane and copy) while it
// computes the current chunk from the other buffer, so two chunks' rows are
// in flight at a time.  The 32
// partial dot products of a chunk (8 positions x 4 query heads) are reduced
// by a butterfly reduce-scatter (31 shuffles), the softmax runs online (max,
// sum, rescaled accumulators) in fp32.  The splits' partial results (max,
// sum, accumulator) are merged in a fixed order by a second kernel.
#include <algorithm>
#include <cmath>
#include <cstdint>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "wq_internal.h"
#include "wq_ptx.cuh"

namespace wq {

// Status word of the attention kernels: WQ_OK (0), or WQ_ERR_ARG (-1) after a
// sequence length outside [0, max_len) was met on the device (that sequence is
// skipped).  Read and cleared by read_attn_status.
__device__ int g_attn_status = 0;

namespace {

constexpr int kAttnWarps = 8;
constexpr int kHG = 4;   // query heads a pass takes (padded with zero heads)
constexpr int kPos = 8;  // positions a chunk takes (kHG * kPos = 32 lanes)

__device__ __forceinline__ float bf_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// HD/32 consecutive bf16 values of a row in shared memory (8 bytes for HD
// 128, 4 for HD 64)
template <int HD>
__device__ __forceinline__ void load_row_s(const __nv_bfloat16 *p, float (&v)[HD / 32]) {
  if (HD == 128) {
    const uint2 w = *reinterpret_cast<const uint2 *>(p);
    v[0] = bf_lo(w.x); v[1] = bf_hi(w.x); v[2] = bf_lo(w.y); v[3] = bf_hi(w.y);
  } else {
    const uint32_t w = *reinterpret_cast<const uint32_t *>(p);
    v[0] = bf_lo(w); v[1] = bf_hi(w);
  }
}

}  // namespace

// RoPE frequencies theta^(-2i/hd), i < hd/2, computed on the host in fp64.
struct RopeFreq {
  double f[64];
};

// grid (B * n_kv, S), block kAttnWarps * 32.  part: [B][H][S][HD + 2] fp32
// (accumulator, max, sum) of every split.
// Copies of one chunk (positions cb .. cb + kPos - 1) of K and V rows into a
// warp's buffer dst ([K, V][kPos][HD], already offset by the lane's column):
// copy i of a lane takes row i * (32 / CPR) + lrow; positions outside
// [p0, p1) and the new position pos are zero-filled.
template <int HD>
__device__ __forceinline__ void attn_issue(__nv_bfloat16 *dst, const __nv_bfloat16 *kbase,
                                           const __nv_bfloat16 *vbase, int lrow, int cb, int p0, int p1, int pos) {
  constexpr int CPR = HD * 2 / 16;
#pragma unroll
  for (int i = 0; i < 2 * kPos * CPR / 32; ++i) {
    const int r = i * (32 / CPR) + lrow;
    const int p = cb + r % kPos;
    const bool in = p < p1 && p != pos;
    const __nv_bfloat16 *src = (r < kPos ? kbase : vbase) + (size_t)(in ? p : p0) * HD;
    cp_async16_zfill(dst + (size_t)r * HD, src, in ? 16u : 0u);
  }
}

// Dynamic shared memory: per warp two chunk buffers of K and V rows,
// [warp][buffer][K, V][kPos][HD] bf16.
template <int HD>
constexpr int attn_smem_bytes() { return kAttnWarps * 2 * 2 * kPos * HD * 2; }

template <int HD>
__global__ void __launch_bounds__(kAttnWarps * 32, 2) attn_split_kernel(
    const float *qkv, const __nv_bfloat16 *x, const int *lens, int d, int H, int Hkv, const RopeFreq fr,
    __nv_bfloat16 *k_cache, __nv_bfloat16 *v_cache, int max_len, float *part, int S) {
  constexpr int E = HD / 32;  // dimensions a lane holds
  extern __shared__ __align__(16) uint8_t attn_dyn[];
  __shared__ float qs[kHG * 2][HD];  // the group's query heads (up to 8), scaled by 1/sqrt(HD)
  __shared__ float kvn[2][HD];       // the new token's k (normalized, rotated, bf16-rounded) and v
  __shared__ float red[kAttnWarps];
  __shared__ float rc[HD / 2], rsn[HD / 2];  // cos, sin of the RoPE angles at this position
  __shared__ float ws_m[kAttnWarps][kHG * 2], ws_l[kAttnWarps][kHG * 2];
  __shared__ float ws_o[kAttnWarps][kHG][HD];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.x / Hkv, g = blockIdx.x % Hkv, split = blockIdx.y;
  const int rep = H / Hkv;
  const int pos = lens[b];          // the new token's position
  if (pos < 0 || pos >= max_len) {  // no room in the cache: record, skip the sequence
    if (threadIdx.x == 0 && blockIdx.y == 0 && g == 0) atomicExch(&g_attn_status, -1);
    return;
  }
  const int L = pos + 1;            // positions attended
  const int C = (L + S - 1) / S;    // positions a split
  const int p0 = split * C, p1 = min(L, p0 + C);
  const int row = (H + 2 * Hkv) * HD;
  const size_t cache_off = ((size_t)b * Hkv + g) * max_len * HD;

  // RoPE angles at the new position: pos f_i in fp64, reduced to [-pi, pi]
  if (tid < HD / 2) {
    const double a = (double)pos * fr.f[tid];
    const double k = rint(a * 0.15915494309189535);  // 1 / (2 pi)
    const double red_a = fma(-k, 6.283185307179586, a);
    const float r = (float)fma(-k, 2.4492935982947064e-16, red_a);  // 2 pi - fl(2 pi)
    float sn, cs;
    sincosf(r, &sn, &cs);
    rc[tid] = cs;
    rsn[tid] = sn;
  }
  // 1. rs of x[b]
  float ss = 0.f;
  for (int i = tid; i < d; i += blockDim.x) {
    const float v = __bfloat162float(x[(size_t)b * d + i]);
    ss = fmaf(v, v, ss);
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  float tot = 0.f;
  for (int w = 0; w < kAttnWarps; ++w) tot += red[w];
  const float rs = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(tot, (float)d), kRmsEps)));

  // 2./3. the group's q heads, k and v: warp w takes head w (q heads, then k, then v)
  const bool has_new = p0 <= pos && pos < p1;
  for (int hh = warp; hh < rep + 2; hh += kAttnWarps) {
    const int col = hh < rep ? (g * rep + hh) * HD : hh == rep ? (H + g) * HD : (H + Hkv + g) * HD;
    float v[E];
#pragma unroll
    for (int e = 0; e < E; ++e) v[e] = qkv[(size_t)b * row + col + lane * E + e] * rs;
    if (hh <= rep) {
      // per-head RMSNorm, then RoPE: element i (< HD/2) with i + HD/2, held by lane and lane ^ 16
      float sq = 0.f;
#pragma unroll
      for (int e = 0; e < E; ++e) sq = fmaf(v[e], v[e], sq);
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
      const float hn = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(sq, (float)HD), kRmsEps)));
#pragma unroll
      for (int e = 0; e < E; ++e) v[e] *= hn;
      float pv[E];
#pragma unroll
      for (int e = 0; e < E; ++e) pv[e] = __shfl_xor_sync(0xffffffffu, v[e], 16);
      const bool lo = lane < 16;
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const int i = (lane & 15) * E + e;  // index in the first half
        const float c = rc[i], s = rsn[i];
        v[e] = lo ? v[e] * c - pv[e] * s : v[e] * c + pv[e] * s;
      }
    }
    if (hh < rep) {
      const float qsc = __frsqrt_rn((float)HD);
#pragma unroll
      for (int e = 0; e < E; ++e) qs[hh][lane * E + e] = v[e] * qsc;
    } else {
      const int kv = hh - rep;  // 0: k, 1: v
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const __nv_bfloat16 bv = __float2bfloat16_rn(v[e]);
        kvn[kv][lane * E + e] = __bfloat162float(bv);
        if (has_new) (kv == 0 ? k_cache : v_cache)[cache_off + (size_t)pos * HD + lane * E + e] = bv;
      }
    }
  }
  __syncthreads();

  // 4. attention over [p0, p1): per pass, 4 query heads
  for (int h0 = 0; h0 < rep; h0 += kHG) {
    float q[kHG][E];
#pragma unroll
    for (int hq = 0; hq < kHG; ++hq)
#pragma unroll
      for (int e = 0; e < E; ++e) q[hq][e] = h0 + hq < rep ? qs[h0 + hq][lane * E + e] : 0.f;
    float m_run = -INFINITY, l_run = 0.f;  // of head h0 + (lane & 3)
    float acc[kHG][E];
#pragma unroll
    for (int hq = 0; hq < kHG; ++hq)
#pragma unroll
      for (int e = 0; e < E; ++e) acc[hq][e] = 0.f;
    // this warp's chunk buffers; positions outside [p0, p1) and the new
    // position (taken from kvn) are zero-filled
    __nv_bfloat16 *wbuf = reinterpret_cast<__nv_bfloat16 *>(attn_dyn) + (size_t)warp * 2 * 2 * kPos * HD;
    constexpr int CPR = HD * 2 / 16;  // 16-byte copies a row
    // copy i of a lane: row r = i * (32 / CPR) + lane / CPR of the [K, V][kPos]
    // rows, 16 bytes at column lane % CPR
    const int lrow = lane / CPR, lcol = (lane % CPR) * 8;
    const __nv_bfloat16 *kbase = k_cache + cache_off + lcol, *vbase = v_cache + cache_off + lcol;
    constexpr int stride = kAttnWarps * kPos;
    int bi = 0;
    if (p0 + warp * kPos < p1)
      attn_issue<HD>(wbuf + lcol, kbase, vbase, lrow, p0 + warp * kPos, p0, p1, pos);
    cp_async_commit();
    for (int c0 = p0 + warp * kPos; c0 < p1; c0 += stride, bi ^= 1) {
      if (c0 + stride < p1)
        attn_issue<HD>(wbuf + (size_t)(bi ^ 1) * 2 * kPos * HD + lcol, kbase, vbase, lrow, c0 + stride, p0, p1, pos);
      cp_async_commit();
      cp_async_wait_group1();  // this chunk's rows have landed
      __syncwarp();
      const __nv_bfloat16 *cur = wbuf + (size_t)bi * 2 * kPos * HD;
      // partial dots of 8 positions x 4 heads: index pp * 4 + hq
      float sv[32];
      float vv[kPos][E];
#pragma unroll
      for (int pp = 0; pp < kPos; ++pp) {
        const int p = c0 + pp;
        float kr[E];
        if (p != pos) {
          load_row_s<HD>(cur + (size_t)pp * HD + lane * E, kr);
          load_row_s<HD>(cur + (size_t)(kPos + pp) * HD + lane * E, vv[pp]);
        } else {
#pragma unroll
          for (int e = 0; e < E; ++e) {
            kr[e] = kvn[0][lane * E + e];
            vv[pp][e] = kvn[1][lane * E + e];
          }
        }
#pragma unroll
        for (int hq = 0; hq < kHG; ++hq) {
          float dsum = 0.f;
#pragma unroll
          for (int e = 0; e < E; ++e) dsum = fmaf(q[hq][e], kr[e], dsum);
          sv[pp * kHG + hq] = dsum;
        }
      }
      // reduce-scatter: afterwards lane l holds the full dot of index l
#pragma unroll
      for (int hb = 16; hb >= 1; hb >>= 1) {
#pragma unroll
        for (int j = 0; j < hb; ++j) {
          const bool up = (lane & hb) != 0;
          const float keep = up ? sv[j + hb] : sv[j];
          const float send = up ? sv[j] : sv[j + hb];
          sv[j] = keep + __shfl_xor_sync(0xffffffffu, send, hb);
        }
      }
      const int my_p = c0 + (lane >> 2);
      const float s = my_p < p1 ? sv[0] : -INFINITY;
      // online softmax per head (the 8 lanes of head lane & 3)
      float mc = s;
      mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, 4));
      mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, 8));
      mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, 16));
      const float m_new = fmaxf(m_run, mc);
      const float alpha = m_new == -INFINITY ? 1.f : __expf(m_run - m_new);
      const float pr = s == -INFINITY ? 0.f : __expf(s - m_new);
      float ps = pr;
      ps += __shfl_xor_sync(0xffffffffu, ps, 4);
      ps += __shfl_xor_sync(0xffffffffu, ps, 8);
      ps += __shfl_xor_sync(0xffffffffu, ps, 16);
      l_run = l_run * alpha + ps;
      m_run = m_new;
      // accumulators: rescale per head, add p v
#pragma unroll
      for (int hq = 0; hq < kHG; ++hq) {
        const float al = __shfl_sync(0xffffffffu, alpha, hq);
#pragma unroll
        for (int e = 0; e < E; ++e) acc[hq][e] *= al;
      }
#pragma unroll
      for (int pp = 0; pp < kPos; ++pp)
#pragma unroll
        for (int hq = 0; hq < kHG; ++hq) {
          const float pw = __shfl_sync(0xffffffffu, pr, pp * kHG + hq);
#pragma unroll
          for (int e = 0; e < E; ++e) acc[hq][e] = fmaf(pw, vv[pp][e], acc[hq][e]);
        }
      __syncwarp();  // every lane is done with this buffer before it is filled again
    }
    cp_async_wait_all();
    // merge the warps (fixed order) and write the split's partials
    if (lane < kHG) {
      ws_m[warp][lane] = m_run;
      ws_l[warp][lane] = l_run;
    }
#pragma unroll
    for (int hq = 0; hq < kHG; ++hq)
#pragma unroll
      for (int e = 0; e < E; ++e) ws_o[warp][hq][lane * E + e] = acc[hq][e];
    __syncthreads();
    for (int i = tid; i < kHG * HD; i += blockDim.x) {
      const int hq = i / HD, e = i % HD;
      if (h0 + hq >= rep) continue;
      float M = -INFINITY;
      for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, ws_m[w][hq]);
      float Ls = 0.f, O = 0.f;
      for (int w = 0; w < kAttnWarps; ++w) {
        const float f = ws_m[w][hq] == -INFINITY ? 0.f : __expf(ws_m[w][hq] - M);
        Ls = fmaf(ws_l[w][hq], f, Ls);
        O = fmaf(ws_o[w][hq][e], f, O);
      }
      const int h = g * rep + h0 + hq;
      float *pt = part + (((size_t)b * H + h) * S + split) * (HD + 2);
      pt[e] = O;
      if (e == 0) {
        pt[HD] = M;
        pt[HD + 1] = Ls;
      }
    }
    __syncthreads();
  }
}

// o[b][h * HD + e] = bf16( sum_s O_s e^(M_s - M) / sum_s L_s e^(M_s - M) ).
// grid B * H, 8 warps: warp w merges the splits w, w + 8, .. in order (its
// own max first), lane l the features l * HD/32 ..; then the warps' results
// are merged in warp order -- a fixed order, so the result is deterministic.
template <int HD>
__global__ void __launch_bounds__(kAttnWarps * 32) attn_combine_kernel(const float *part, const int *lens, int H, int S,
                                                                       int max_len, __nv_bfloat16 *o) {
  constexpr int E = HD / 32;
  __shared__ float wm[kAttnWarps], wl[kAttnWarps], wo[kAttnWarps][HD];
  const int bh = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pos = lens[bh / H];
  if (pos < 0 || pos >= max_len) return;  // skipped by the split kernel
  const float *pt = part + (size_t)bh * S * (HD + 2);
  float M = -INFINITY;
  for (int s = warp; s < S; s += kAttnWarps) M = fmaxf(M, pt[(size_t)s * (HD + 2) + HD]);
  float L = 0.f, O[E];
#pragma unroll
  for (int e = 0; e < E; ++e) O[e] = 0.f;
#pragma unroll 4
  for (int s = warp; s < S; s += kAttnWarps) {
    const float *ps = pt + (size_t)s * (HD + 2);
    const float ms = ps[HD];
    const float f = ms == -INFINITY ? 0.f : __expf(ms - M);
    L = fmaf(ps[HD + 1], f, L);
#pragma unroll
    for (int e = 0; e < E; ++e) O[e] = fmaf(ps[lane * E + e], f, O[e]);
  }
  if (lane == 0) {
    wm[warp] = M;
    wl[warp] = L;
  }
#pragma unroll
  for (int e = 0; e < E; ++e) wo[warp][lane * E + e] = O[e];
  __syncthreads();
  for (int e = threadIdx.x; e < HD; e += blockDim.x) {
    float Mt = -INFINITY;
    for (int w = 0; w < kAttnWarps; ++w) Mt = fmaxf(Mt, wm[w]);
    float Lt = 0.f, Ot = 0.f;
    for (int w = 0; w < kAttnWarps; ++w) {
      const float f = wm[w] == -INFINITY ? 0.f : __expf(wm[w] - Mt);
      Lt = fmaf(wl[w], f, Lt);
      Ot = fmaf(wo[w][e], f, Ot);
    }
    o[(size_t)bh * HD + e] = __float2bfloat16_rn(Ot / Lt);
  }
}

int attn_splits(int B, int Hkv, int max_len, int num_sms) {
  // enough CTAs to cover the SMs twice, at least 64 positions a split
  const int want = std::max(1, (2 * num_sms + B * Hkv - 1) / (B * Hkv));
  return std::max(1, std::min(want, (max_len + 63) / 64));
}

cudaError_t launch_attn_decode(const float *qkv, const void *x, const int *lens, int B, int d, int H, int Hkv, int HD,
                               double theta, void *k_cache, void *v_cache, int max_len, float *part, int S, void *o,
                               cudaStream_t s) {
  const dim3 grid(B * Hkv, S);
  if (HD > 128) return cudaErrorInvalidValue;
  RopeFreq fr{};
  for (int i = 0; i < HD / 2; ++i) fr.f[i] = std::pow(theta, -2.0 * i / HD);
  const auto *xb = reinterpret_cast<const __nv_bfloat16 *>(x);
  auto *kc = reinterpret_cast<__nv_bfloat16 *>(k_cache), *vc = reinterpret_cast<__nv_bfloat16 *>(v_cache);
  auto *ob = reinterpret_cast<__nv_bfloat16 *>(o);
  if (HD == 128) {
    constexpr int sm = attn_smem_bytes<128>();
    cudaError_t e = cudaFuncSetAttribute(attn_split_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
    if (e != cudaSuccess) return e;
    attn_split_kernel<128><<<grid, kAttnWarps * 32, sm, s>>>(qkv, xb, lens, d, H, Hkv, fr, kc, vc, max_len, part, S);
    attn_combine_kernel<128><<<B * H, kAttnWarps * 32, 0, s>>>(part, lens, H, S, max_len, ob);
  } else if (HD == 64) {
    constexpr int sm = attn_smem_bytes<64>();
    cudaError_t e = cudaFuncSetAttribute(attn_split_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
    if (e != cudaSuccess) return e;
    attn_split_kernel<64><<<grid, kAttnWarps * 32, sm, s>>>(qkv, xb, lens, d, H, Hkv, fr, kc, vc, max_len, part, S);
    attn_combine_kernel<64><<<B * H, kAttnWarps * 32, 0, s>>>(part, lens, H, S, max_len, ob);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t read_attn_status(int *status) {
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(status, g_attn_status, sizeof(int));
  if (e != cudaSuccess) return e;
  const int zero = 0;
  return cudaMemcpyToSymbol(g_attn_status, &zero, sizeof(int));
}

}  // namespace wq
