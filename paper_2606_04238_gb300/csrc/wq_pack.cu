// wq_pack.cu -- Stage-1 group-wise quantizer and packer (sm_103a).
//
// Sec. 4.1 quantizes gate/up to INT2 and (Sec. 3.3, Sec. 7 step 4) every
// other linear layer to INT4.  The quantizer is asymmetric min-max
// round-to-nearest per group of `group` consecutive input features of a row,
// computed in IEEE fp32 with explicit round-to-nearest intrinsics so that the
// codes, scales and zeros are reproducible bit for bit:
//   s = fp16((max - min) / qmax) (1.0 if zero), z = clamp(rint(-min/s), 0, qmax),
//   q = clamp(rint(w/s) + z, 0, qmax).
// Two kernels: one warp per (row, group) computes s and z into the packed
// meta layout; then one thread per packed 32-bit word gathers its 16 (2-bit)
// or 8 (4-bit) codes, or for 3-bit codes (App. B) 16 low-plane fields (q % 4)
// or 32 high-plane bits (q / 4).  Offline work: not on the decode path.
// A third kernel merges a trained adapter into a packed matrix before it is
// quantized again (below).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "wq_internal.h"
#include "wq_launch.h"

namespace wq {
namespace {

__global__ void quant_meta_kernel(const float *__restrict__ w, int n, int k, int group, int bits, int RT, int NG,
                                  uint16_t *__restrict__ meta, int *nonfinite) {
  const long long gw = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (long long)RT * 16 * NG) return;  // warp-uniform
  const int row = (int)(gw / NG), j = (int)(gw % NG);
  const int ngk = k / group;
  unsigned short s16 = 0, z16 = 0;
  if (row < n && j < ngk) {
    const float *src = w + (size_t)row * k + (size_t)j * group;
    float mn = INFINITY, mx = -INFINITY;
    bool bad = false;
    for (int i = lane; i < group; i += 32) {
      const float v = src[i];
      bad |= !isfinite(v);
      mn = fminf(mn, v);
      mx = fmaxf(mx, v);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    bad = __any_sync(0xffffffffu, bad);
    const float qmax = (float)((1 << bits) - 1);
    __half sh = __float2half_rn(__fdiv_rn(__fsub_rn(mx, mn), qmax));
    if (__half2float(sh) == 0.f) sh = __float2half_rn(1.f);
    const float sf = __half2float(sh);
    const float zf = __fadd_rn(fminf(fmaxf(rintf(__fdiv_rn(-mn, sf)), 0.f), qmax), 0.f);
    s16 = __half_as_ushort(sh);
    z16 = __half_as_ushort(__float2half_rn(zf));
    if (bad && lane == 0 && nonfinite) atomicOr(nonfinite, 1);
  }
  if (lane == 0) {
    const int rt = row >> 4, i = row & 15;
    const size_t base = ((size_t)rt * NG + j) * 32 + 4 * (i & 7) + (i >> 3);
    meta[base] = s16;
    meta[base + 2] = z16;
  }
}

__global__ void pack_codes_kernel(const float *__restrict__ w, int n, int k, int group, int bits, int RT, int KB,
                                  int NG, const uint16_t *__restrict__ meta, uint32_t *__restrict__ codes) {
  const int WPB = bits == 2 ? 128 : bits == 3 ? 192 : 256;
  const size_t wid = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (wid >= (size_t)RT * KB * WPB) return;
  const size_t blk = wid / WPB;
  const int wl = (int)(wid % WPB);
  const int rt = (int)(blk / KB), kb = (int)(blk % KB);
  const float qmax = (float)((1 << bits) - 1);
  // code of (local row i, block feature c), or 0 outside the matrix
  auto code_at = [&](int i, int c) -> uint32_t {
    const int row = rt * 16 + i, col = kb * 128 + c;
    if (row >= n || col >= k) return 0u;
    const size_t mb = ((size_t)rt * NG + col / group) * 32 + 4 * (i & 7) + (i >> 3);
    const float sf = __half2float(__ushort_as_half(meta[mb]));
    const float zf = __half2float(__ushort_as_half(meta[mb + 2]));
    return (uint32_t)fminf(fmaxf(__fadd_rn(rintf(__fdiv_rn(w[(size_t)row * k + col], sf)), zf), 0.f), qmax);
  };
  if (bits == 3) {
    uint32_t word = 0;
    if (wl < 128) {  // low plane: q % 4 where a 2-bit code would sit
      const int lane = wl >> 2, wi = wl & 3;
      for (int bit = 0; bit < 32; bit += 2) {
        const int half = bit >> 4, rowhalf = (bit >> 3) & 1, cls = (bit & 7) >> 1;
        const int c = wi * 32 + (cls >> 1) * 16 + (cls & 1) * 8 + (lane & 3) * 2 + half;
        word |= (code_at((lane >> 2) + 8 * rowhalf, c) & 3u) << bit;
      }
    } else {  // high plane: word 128 + 2 lane + p holds q / 4 of the features c with (c / 32) / 2 = p
      const int lane = (wl - 128) >> 1, pp = (wl - 128) & 1;
      for (int bit = 0; bit < 32; ++bit) {
        const int half = bit >> 4, cpar = (bit >> 3) & 1, cls = (bit & 7) >> 1, ihi = bit & 1;
        const int c = (2 * pp + cpar) * 32 + (cls >> 1) * 16 + (cls & 1) * 8 + (lane & 3) * 2 + half;
        word |= (code_at((lane >> 2) + 8 * ihi, c) >> 2) << bit;
      }
    }
    codes[wid] = word;
    return;
  }
  const int tile = bits == 2 ? 0 : wl >> 7;  // 64-feature half of a 4-bit block
  const int wl2 = wl & 127;
  const int lane = wl2 >> 2, wi = wl2 & 3;
  uint32_t word = 0;
  for (int bit = 0; bit < 32; bit += bits) {
    const int half = bit >> 4, rowhalf = (bit >> 3) & 1;
    int c;
    if (bits == 2) {
      const int cls = (bit & 7) >> 1;  // 2 * (16-feature step parity) + (upper 8 features)
      c = wi * 32 + (cls >> 1) * 16 + (cls & 1) * 8 + (lane & 3) * 2 + half;
    } else {
      const int hi = (bit & 7) >> 2;
      c = tile * 64 + wi * 16 + hi * 8 + (lane & 3) * 2 + half;
    }
    word |= code_at((lane >> 2) + 8 * rowhalf, c) << bit;
  }
  codes[wid] = word;
}

// Adapter merge (Sec. 4.2 lets the trained adapters be merged into the
// quantized weights; Sec. 7 step 5 deploys them merged or attached).  By
// Eq. 1 the merged matrix is deq(W) + alpha B A:
//   w[row, col] = fp32( s (q - z) + alpha * sum_rho B[row, rho] A[rho, col] ),
// evaluated in fp64 with rho ascending (a product of two bf16 values is exact)
// and rounded to fp32 once.  Every operation is an explicit round-to-nearest
// intrinsic, so no contraction changes the result.  The codes, scales and
// zeros are read from the packed layout of include/wq.h.  A CTA takes 256
// features of a row (rows strided by gridDim.y); the row of B is staged in
// shared memory as fp64.
constexpr int kMergeThreads = 256;

__global__ void __launch_bounds__(kMergeThreads)
    merge_lora_kernel(const uint32_t *__restrict__ codes, const uint16_t *__restrict__ meta, int n, int k,
                      int group, int bits, int KB, int NG, const __nv_bfloat16 *__restrict__ lora_b,
                      const __nv_bfloat16 *__restrict__ lora_a, int r, double alpha, float *__restrict__ w) {
  __shared__ double brow[kMaxRank];
  const int col = blockIdx.x * kMergeThreads + threadIdx.x;
  const int wpb = bits == 2 ? 128 : bits == 3 ? 192 : 256;
  const uint32_t mask = bits == 3 ? 3u : (1u << bits) - 1u;
  for (int row = blockIdx.y; row < n; row += gridDim.y) {
    __syncthreads();  // the previous row's B is read by every thread first
    if (threadIdx.x < r) brow[threadIdx.x] = (double)__bfloat162float(lora_b[(size_t)row * r + threadIdx.x]);
    __syncthreads();
    if (col >= k) continue;
    const int rt = row >> 4, i = row & 15, kb = col >> 7, c = col & 127;
    const int lane = (i & 7) * 4 + ((c & 7) >> 1), half = c & 1;
    int word, bit;
    if (bits != 4) {
      word = lane * 4 + (c >> 5);
      bit = 16 * half + 8 * (i >> 3) + 2 * (2 * ((c & 31) >> 4) + ((c & 15) >> 3));
    } else {
      word = (c >> 6) * 128 + lane * 4 + ((c & 63) >> 4);
      bit = 16 * half + 8 * (i >> 3) + 4 * ((c & 15) >> 3);
    }
    const uint32_t *blk = codes + ((size_t)rt * KB + kb) * wpb;
    uint32_t q = (blk[word] >> bit) & mask;
    if (bits == 3) {  // the high bit from the second plane
      const int cls = 2 * ((c & 31) >> 4) + ((c & 15) >> 3);
      q |= ((blk[128 + lane * 2 + ((c >> 5) >> 1)] >> (16 * half + 8 * ((c >> 5) & 1) + 2 * cls + (i >> 3))) & 1u) << 2;
    }
    const size_t mb = ((size_t)rt * NG + col / group) * 32 + 4 * (i & 7) + (i >> 3);
    const double sf = (double)__half2float(__ushort_as_half(meta[mb]));
    const double zf = (double)__half2float(__ushort_as_half(meta[mb + 2]));
    double ba = 0.0;
    for (int rho = 0; rho < r; ++rho)
      ba = __dadd_rn(ba, __dmul_rn(brow[rho], (double)__bfloat162float(lora_a[(size_t)rho * k + col])));
    const double v = __dadd_rn(__dmul_rn(sf, __dsub_rn((double)q, zf)), __dmul_rn(alpha, ba));
    w[(size_t)row * k + col] = __double2float_rn(v);
  }
}

}  // namespace

cudaError_t launch_merge_lora(const uint32_t *codes, const uint16_t *meta, int n, int k, int group, int bits,
                              const void *lora_b, const void *lora_a, int r, float alpha, float *w,
                              cudaStream_t stream) {
  const int KB = (k + 127) / 128, NG = KB * 128 / group;
  const dim3 grid((unsigned)((k + kMergeThreads - 1) / kMergeThreads), (unsigned)std::min(n, 65535));
  merge_lora_kernel<<<grid, kMergeThreads, 0, stream>>>(codes, meta, n, k, group, bits, KB, NG,
                                                         static_cast<const __nv_bfloat16 *>(lora_b),
                                                         static_cast<const __nv_bfloat16 *>(lora_a), r,
                                                         (double)alpha, w);
  return cudaGetLastError();
}

cudaError_t launch_pack(const float *w, int n, int k, int group, int bits, uint32_t *codes, uint16_t *meta,
                        int *nonfinite, cudaStream_t stream) {
  const int RT = (n + 15) / 16, KB = (k + 127) / 128, NG = KB * 128 / group;
  const long long warps = (long long)RT * 16 * NG;
  const int tpb = 256;
  quant_meta_kernel<<<(unsigned)((warps * 32 + tpb - 1) / tpb), tpb, 0, stream>>>(w, n, k, group, bits, RT, NG, meta,
                                                                                 nonfinite);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const long long words = (long long)RT * KB * (bits == 2 ? 128 : bits == 3 ? 192 : 256);
  pack_codes_kernel<<<(unsigned)((words + tpb - 1) / tpb), tpb, 0, stream>>>(w, n, k, group, bits, RT, KB, NG, meta,
                                                                             codes);
  return cudaGetLastError();
}

}  // namespace wq
