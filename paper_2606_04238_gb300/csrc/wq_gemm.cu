// wq_gemm.cu -- batched (prefill-size) dequant-GEMM on the 5th-generation
// tensor cores (tcgen05, accumulators in tensor memory), sm_103a.
//
// For a token batch of more than a few dozen tokens the gated MLP of the
// W4/W2-GateUp scheme (Sec. 3.3) is a real dense contraction, so the packed
// weights are dequantized to binary16 tiles in shared memory and fed to
// tcgen05.mma with fp32 accumulation in TMEM:
//   * gate/up: D_g = x deq(Wg)^T + (lora_scale x A_g^T) B_g^T, D_u likewise
//     (the unmerged LoRA path of Eq. 1 enters as two more k-steps), then
//     h = SiLU(rs D_g) * (rs D_u) with rs the RMSNorm scale of the token;
//   * down: y = residual + h deq(Wd)^T.
// A CTA computes a tile of 128 tokens x 128 output rows (x 2 projections for
// gate/up) over the whole feature axis, one 128-feature block of the packed
// format per pipeline stage.  Warp roles:
//   warps 0..7  dequantize the stage's codes: code q of row n, group j gives
//               the binary16 value s_nj (q - z_nj), rounded once; they write
//               it in the tcgen05 K-major layout (8-row x 16-byte core
//               matrices), warps 0..3 then run the epilogue from TMEM;
//   warp 8      stages the binary16 activation tile (cp.async, zero fill
//               outside the matrix) and bulk-copies the stage's packed codes
//               and scales/zeros;
//   warp 9      owns the TMEM allocation; its lane 0 issues the MMAs.
// Stages are handed over with mbarriers; every wait is bounded (a timeout
// sets the device status word and the CTA skips the rest of its work).
#include <algorithm>
#include <cmath>

#include "wq_internal.h"
#include "wq_ptx.cuh"

namespace wq {

// Device status word of the GEMM kernels: WQ_OK (0) or WQ_ERR_TIMEOUT (-6).
__device__ int g_gemm_status = 0;

namespace {

constexpr int kBM = 128;                         // tokens per CTA tile (MMA M)
constexpr int kBN = 128;                         // output rows per CTA tile and projection (MMA N)
constexpr int kDeqWarps = 8;                     // dequantizing warps
constexpr int kProducerWarp = kDeqWarps;         // activation / code staging
constexpr int kMmaWarp = kDeqWarps + 1;          // TMEM owner and MMA issuer
constexpr int kGemmThreads = (kDeqWarps + 2) * 32;
constexpr int kTileBytes = kBM * 128 * 2;        // one 128 x 128 binary16 operand tile
constexpr uint32_t kSboTile = 16 * 128;          // bytes between 8-row groups of a 128-feature tile
constexpr uint32_t kGemmSmemLimit = 232448;      // 227 KB opt-in

// EXACT: every weight s (q - z) is written as two binary16 tiles whose sum is
// exact -- s_hi (q - z) and s_lo (q - z), s_hi the scale with its 4 lowest
// mantissa bits cleared and s_lo = s - s_hi -- and the tensor cores add both
// (two MMAs a k-step), so the products are those of the exact weights.  Used
// for fp32 output; otherwise each weight is rounded to binary16 once.
template <int BITS, int NPROJ, int GROUP, bool EXACT>
struct GemmCfg {
  static constexpr int BPK = BITS == 2 ? 512 : 1024;      // code bytes per (16-row tile, block)
  static constexpr int GPB = 128 / GROUP;
  static constexpr int NB = NPROJ * (EXACT ? 2 : 1);      // B tiles a stage
  static constexpr int RAW_TILE = BPK + GPB * 64;          // codes + scales/zeros of a (tile, block)
  static constexpr int RAW = NPROJ * 8 * RAW_TILE;         // a stage's packed weights (8 tiles)
  static constexpr int STAGE = kTileBytes + NB * kTileBytes + RAW;
  // pipeline depth: as many stages as fit, at most 3 (one only for the 4-bit
  // gate/up comparator with groups of 32 or 64)
  static constexpr int S = std::min(3, std::max(1, (int)((kGemmSmemLimit - 1024) / STAGE)));
  static constexpr int OFF_A = 0;
  static constexpr int OFF_B = S * kTileBytes;
  static constexpr int OFF_RAW = OFF_B + S * NB * kTileBytes;
  static constexpr int OFF_BAR = OFF_RAW + S * RAW;        // 4 S + 2 barriers
  static constexpr int SMEM = OFF_BAR + (4 * S + 2) * 8 + 16;
  static constexpr int NCOLS = NPROJ == 2 ? 256 : 128;     // TMEM columns (fp32 accumulators)
  static_assert(SMEM <= (int)kGemmSmemLimit, "GEMM stage does not fit");
};

__device__ __forceinline__ void gemm_timeout() { atomicExch(&g_gemm_status, -6); }

// Byte offset of element (row, k) in a K-major no-swizzle tile whose 8-row
// groups are `sbo` bytes apart (core matrices along K 128 bytes apart).
__device__ __forceinline__ uint32_t kmajor_off(int row, int k, uint32_t sbo) {
  return (uint32_t)(row >> 3) * sbo + (uint32_t)(k >> 3) * 128u + (uint32_t)(row & 7) * 16u + (uint32_t)(k & 7) * 2u;
}

__device__ __forceinline__ uint32_t h2bits(__half2 v) { return *reinterpret_cast<uint32_t *>(&v); }
__device__ __forceinline__ __half2 bits2h(uint32_t v) { return *reinterpret_cast<__half2 *>(&v); }

template <int BITS, int NPROJ, int GROUP, bool EXACT>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_kernel(const GemmArgs a) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  constexpr int S = C::S, GPB = C::GPB, GS = GROUP / 16;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint64_t *raw_full = reinterpret_cast<uint64_t *>(smem + C::OFF_BAR);
  uint64_t *a_full = raw_full + S;
  uint64_t *b_full = a_full + S;
  uint64_t *empty = b_full + S;
  uint64_t *acc_full = empty + S;
  uint32_t *tmem_s = reinterpret_cast<uint32_t *>(acc_full + 2);
  volatile int *abort_s = reinterpret_cast<volatile int *>(tmem_s + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * kBN;
  const int KB = (a.K + 127) / 128;
  const int RT = (a.N + 15) / 16;
  const bool lora = NPROJ == 2 && a.r > 0;
  const int nit = KB + (lora ? 1 : 0);
  const int rp = (a.r + 15) / 16 * 16;  // LoRA rank padded to whole k-steps (zeros)

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&raw_full[s], 1);
      mbar_init(&a_full[s], 1);
      mbar_init(&b_full[s], kDeqWarps);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    *abort_s = 0;
    fence_barrier_init();
  }
  if (warp == kMmaWarp) tmem_alloc(tmem_s, C::NCOLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_s;

  // bounded wait; a timeout (or an earlier one) makes the caller skip its work
  auto wait = [&](uint64_t *bar, uint32_t parity) -> bool {
    if (*abort_s) return false;
    if (mbar_wait(bar, parity)) return true;
    *abort_s = 1;
    if (lane == 0) gemm_timeout();
    return false;
  };

  if (warp == kProducerWarp) {
    // ---- activations (cp.async) and packed weights (bulk copies) ----
    const int nvalid = max(0, min(8, RT - n0 / 16));  // 16-row tiles of this CTA inside the matrix
    // The activation tile of a stage is released to the MMA one iteration
    // later: once its cp.async group has landed, each lane fences its
    // generic-proxy writes against the tensor cores' reads, then lane 0
    // arrives on a_full.
    auto release = [&](int itr) {
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[itr % S]);
    };
    int it = 0;
    for (; it < nit; ++it) {
      const int s = it % S, u = it / S;
      if (it >= S && !wait(&empty[s], (u - 1) & 1)) break;
      uint8_t *As = smem + C::OFF_A + s * kTileBytes;
      if (it < KB) {
        if (lane == 0) {
          mbar_arrive_expect_tx(&raw_full[s], (uint32_t)(NPROJ * nvalid * C::RAW_TILE));
          for (int p = 0; p < NPROJ; ++p)
            for (int j = 0; j < nvalid; ++j) {
              const int rt = n0 / 16 + j;
              uint8_t *dst = smem + C::OFF_RAW + s * C::RAW + (p * 8 + j) * C::RAW_TILE;
              bulk_g2s(dst, reinterpret_cast<const uint8_t *>(a.codes[p]) + ((size_t)rt * KB + it) * C::BPK, C::BPK,
                       &raw_full[s]);
              bulk_g2s(dst + C::BPK,
                       reinterpret_cast<const uint8_t *>(a.meta[p]) + ((size_t)rt * KB * GPB + (size_t)it * GPB) * 64,
                       GPB * 64, &raw_full[s]);
            }
        }
        // 128 tokens x 16 chunks of 8 features
        for (int i = lane; i < kBM * 16; i += 32) {
          const int ml = i >> 4, c = i & 15;
          const int m = m0 + ml, k = it * 128 + c * 8;
          const bool ok = m < a.M && k < a.K;
          const uint16_t *src = ok ? a.act + (size_t)m * a.lda + k : a.act;  // (no bytes read when !ok)
          cp_async16_zfill(As + kmajor_off(ml, c * 8, kSboTile), src, ok ? 16u : 0u);
        }
      } else {
        // LoRA stage: lora_scale * t for gate (first r) and up (next r), K = r
        // padded to rp with zeros
        if (lane == 0) mbar_arrive(&raw_full[s]);
        const int rc = a.r / 8, rpc = rp / 8;
        for (int i = lane; i < NPROJ * kBM * rpc; i += 32) {
          const int p = i / (kBM * rpc), rem = i - p * kBM * rpc;
          const int ml = rem / rpc, c = rem - ml * rpc;
          const int m = m0 + ml;
          const bool ok = m < a.M && c < rc;
          const uint16_t *src = ok ? a.ta + (size_t)m * 2 * a.r + p * a.r + c * 8 : a.ta;
          cp_async16_zfill(As + p * (kBM * rp * 2) + kmajor_off(ml, c * 8, (uint32_t)rpc * 128u), src, ok ? 16u : 0u);
        }
      }
      cp_async_commit();
      if (it >= 1) {
        cp_async_wait_group1();  // the previous stage's group has landed
        release(it - 1);
      }
    }
    cp_async_wait_all();
    if (it >= 1) release(it - 1);
  } else if (warp == kMmaWarp) {
    // ---- MMA issue ----
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_f16(kBM, kBN);
      for (int it = 0; it < nit; ++it) {
        const int s = it % S, u = it / S;
        if (!wait(&a_full[s], u & 1) || !wait(&b_full[s], u & 1)) break;
        tc_fence_after();
        const uint32_t as = smem_addr(smem + C::OFF_A + s * kTileBytes);
        const uint32_t bs = smem_addr(smem + C::OFF_B + s * C::NB * kTileBytes);
        if (it < KB) {
#pragma unroll
          for (int p = 0; p < NPROJ; ++p)
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
              umma_f16(tmem + p * kBN, umma_desc_kmajor(as + ks * 256, 128, kSboTile),
                       umma_desc_kmajor(bs + p * kTileBytes + ks * 256, 128, kSboTile), idesc, (it > 0 || ks > 0) ? 1u : 0u);
              if (EXACT)  // the low parts of the same weights
                umma_f16(tmem + p * kBN, umma_desc_kmajor(as + ks * 256, 128, kSboTile),
                         umma_desc_kmajor(bs + (NPROJ + p) * kTileBytes + ks * 256, 128, kSboTile), idesc, 1u);
            }
        } else {
          const uint32_t sbo = (uint32_t)(rp / 8) * 128u;
          for (int p = 0; p < NPROJ; ++p)
            for (int ks = 0; ks < rp / 16; ++ks)
              umma_f16(tmem + p * kBN, umma_desc_kmajor(as + p * (kBM * rp * 2) + ks * 256, 128, sbo),
                       umma_desc_kmajor(bs + p * kTileBytes + ks * 256, 128, sbo), idesc, 1u);
        }
        umma_commit(&empty[s]);
      }
      umma_commit(acc_full);
    }
    __syncwarp();
  } else {
    // ---- dequantization into the B tiles ----
    const int dt = tid;  // 0 .. 255
    for (int it = 0; it < nit; ++it) {
      const int s = it % S, u = it / S;
      if (!wait(&raw_full[s], u & 1)) break;
      if (it >= S && !wait(&empty[s], (u - 1) & 1)) break;
      uint8_t *Bs = smem + C::OFF_B + s * C::NB * kTileBytes;
      if (it < KB) {
        const uint8_t *raw = smem + C::OFF_RAW + s * C::RAW;
        // item = (projection, 16-row tile, lane of the packed fragment layout)
        for (int item = dt; item < NPROJ * 8 * 32; item += kDeqWarps * 32) {
          const int p = item >> 8, j = (item >> 5) & 7, L = item & 31;
          const int g = L >> 2, t = L & 3;
          uint8_t *Bp = Bs + p * kTileBytes;
          const bool valid = n0 / 16 + j < RT;
          uint32_t wds[BITS == 2 ? 4 : 8];
          const uint8_t *cb = raw + (p * 8 + j) * C::RAW_TILE;
          if (valid) {
            const uint4 w0 = lds128(cb + L * 16);
            wds[0] = w0.x; wds[1] = w0.y; wds[2] = w0.z; wds[3] = w0.w;
            if (BITS == 4) {
              const uint4 w1 = lds128(cb + 512 + L * 16);
              wds[4] = w1.x; wds[5] = w1.y; wds[6] = w1.z; wds[7] = w1.w;
            }
          } else {
#pragma unroll
            for (int q = 0; q < (BITS == 2 ? 4 : 8); ++q) wds[q] = 0u;
          }
#pragma unroll
          for (int gi = 0; gi < GPB; ++gi) {
            // scales and zeros of rows g and g + 8 in group gi (zero for tiles outside the matrix)
            uint2 sz = make_uint2(0u, 0u);
            if (valid) sz = lds64(cb + C::BPK + gi * 64 + g * 8);
            // scales of rows g ("lo" row) and g + 8 ("hi" row); EXACT splits each
            // into a head with the 4 lowest mantissa bits cleared and the tail
            const uint32_t sg = sz.x & 0xffffu, sg8 = sz.x >> 16;
            const __half2 s_lo = __half2half2(__ushort_as_half((unsigned short)(EXACT ? (sg & 0xfff0u) : sg)));
            const __half2 s_hi = __half2half2(__ushort_as_half((unsigned short)(EXACT ? (sg8 & 0xfff0u) : sg8)));
            const __half2 t_lo = __half2half2(__hsub(__ushort_as_half((unsigned short)sg), __ushort_as_half((unsigned short)(sg & 0xfff0u))));
            const __half2 t_hi = __half2half2(__hsub(__ushort_as_half((unsigned short)sg8), __ushort_as_half((unsigned short)(sg8 & 0xfff0u))));
            // 1024 + z: the code read as 1024 + q minus this is q - z exactly
            const __half2 z_lo = __half2half2(__hadd(__ushort_as_half((unsigned short)(sz.y & 0xffffu)), __float2half(1024.f)));
            const __half2 z_hi = __half2half2(__hadd(__ushort_as_half((unsigned short)(sz.y >> 16)), __float2half(1024.f)));
#pragma unroll
            for (int kk = 0; kk < GS; ++kk) {
              const int ks = gi * GS + kk;
              uint32_t q[4];  // (row g, k 2t..2t+1), (row g+8, ...), (row g, k 2t+8..), (row g+8, k 2t+8..)
              if (BITS == 2) {
                const uint32_t x = wds[(ks >> 1) & 3];
                const int s4 = (ks & 1) * 4;
                q[0] = (x >> s4) & 0x00030003u;
                q[1] = (x >> (s4 + 8)) & 0x00030003u;
                q[2] = (x >> (s4 + 2)) & 0x00030003u;
                q[3] = (x >> (s4 + 10)) & 0x00030003u;
              } else {
                const uint32_t x = wds[ks & 7];
                q[0] = x & 0x000F000Fu;
                q[1] = (x >> 8) & 0x000F000Fu;
                q[2] = (x >> 4) & 0x000F000Fu;
                q[3] = (x >> 12) & 0x000F000Fu;
              }
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const __half2 v = bits2h(q[e] | 0x64006400u);  // 1024 + q, exact
                const bool hi_row = (e & 1) != 0;
                const __half2 qz = __hsub2(v, hi_row ? z_hi : z_lo);  // q - z, exact
                const __half2 w = __hmul2(qz, hi_row ? s_hi : s_lo);
                const int row = j * 16 + g + (hi_row ? 8 : 0);
                const int k = ks * 16 + 2 * t + ((e & 2) ? 8 : 0);
                *reinterpret_cast<uint32_t *>(Bp + kmajor_off(row, k, kSboTile)) = h2bits(w);
                if (EXACT)
                  *reinterpret_cast<uint32_t *>(Bp + NPROJ * kTileBytes + kmajor_off(row, k, kSboTile)) =
                      h2bits(__hmul2(qz, hi_row ? t_hi : t_lo));
              }
            }
          }
        }
      } else {
        // LoRA stage: B_p rows n0 .. n0+127 (bf16 [N][r]) -> binary16, K = r
        // padded to rp with zeros
        const int rc = a.r / 8, rpc = rp / 8;
        const uint32_t sbo = (uint32_t)rpc * 128u;
        for (int i = dt; i < NPROJ * kBN * rpc; i += kDeqWarps * 32) {
          const int p = i / (kBN * rpc), rem = i - p * kBN * rpc;
          const int nl = rem / rpc, c = rem - nl * rpc;
          const int n = n0 + nl;
          uint4 v = make_uint4(0u, 0u, 0u, 0u);
          if (n < a.N && c < rc) v = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const uint8_t *>(a.lora_b[p]) + ((size_t)n * a.r + c * 8) * 2));
          const uint32_t w[4] = {v.x, v.y, v.z, v.w};
          uint32_t o[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float lo = __uint_as_float(w[e] << 16), hi = __uint_as_float(w[e] & 0xffff0000u);
            o[e] = h2bits(__floats2half2_rn(lo, hi));
          }
          *reinterpret_cast<uint4 *>(Bs + p * kTileBytes + kmajor_off(nl, c * 8, sbo)) = make_uint4(o[0], o[1], o[2], o[3]);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&b_full[s]);
    }

    // ---- epilogue (warps 0..3: TMEM lanes 32 w .. 32 w + 31 = tokens) ----
    if (warp < 4 && wait(acc_full, 0)) {
      tc_fence_after();
      const int m = m0 + warp * 32 + lane;
      const float rs = (NPROJ == 2 && a.rs != nullptr && m < a.M) ? a.rs[m] : 1.f;
      const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
      for (int c = 0; c < kBN; c += 8) {
        uint32_t g[8], uu[8];
        tmem_ld8(tl + c, g);
        if (NPROJ == 2) tmem_ld8(tl + kBN + c, uu);
        tmem_ld_wait();
        if (m >= a.M) continue;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int n = n0 + c + e;
          if (n >= a.N) continue;
          if (NPROJ == 2) {
            const float gv = rs * __uint_as_float(g[e]), uv = rs * __uint_as_float(uu[e]);
            const float h = gv / (1.f + __expf(-gv)) * uv;
            const __nv_bfloat16 hb = __float2bfloat16_rn(h);
            reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = hb;
            if (a.out_f16) a.out_f16[(size_t)m * a.ldo16 + n] = __half_as_ushort(__float2half_rn(__bfloat162float(hb)));
          } else {
            float y = __uint_as_float(g[e]);
            if (a.residual) y += __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(a.residual)[(size_t)m * a.N + n]);
            if (a.out_f32)
              reinterpret_cast<float *>(a.out)[(size_t)m * a.N + n] = y;
            else
              reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = __float2bfloat16_rn(y);
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, C::NCOLS);
}

// Per token of x [M, K] (bf16): the binary16 copy (the GEMM's A operand), the
// RMSNorm scale rs = 1/sqrt(mean(x^2) + eps) and, with an adapter,
// ta = lora_scale * x A^T as binary16 [M][2r] (gate rows, then up rows).
// One CTA per token; fixed-order reductions.
__global__ void __launch_bounds__(256) gemm_prep_kernel(const __nv_bfloat16 *x, int M, int K, int lda16,
                                                        const __nv_bfloat16 *lora_a, int r2, float lora_scale,
                                                        uint16_t *x16, float *rs, uint16_t *ta) {
  __shared__ float red[8];
  const int m = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (m >= M) return;
  const __nv_bfloat16 *xr = x + (size_t)m * K;
  float ss = 0.f;
  for (int k = tid; k < K; k += blockDim.x) {
    const float v = __bfloat162float(xr[k]);
    ss = fmaf(v, v, ss);
    x16[(size_t)m * lda16 + k] = __half_as_ushort(__float2half_rn(v));
  }
  for (int k = K + tid; k < lda16; k += blockDim.x) x16[(size_t)m * lda16 + k] = 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  if (tid == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += red[w];
    rs[m] = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(t, (float)K), kRmsEps)));
  }
  if (r2 > 0) {
    // warp w handles LoRA-A rows w, w + 8, ...: sum over k in lane stripes, then the warp
    for (int j = warp; j < r2; j += 8) {
      const __nv_bfloat16 *ar = lora_a + (size_t)j * K;
      float acc = 0.f;
      for (int k = lane; k < K; k += 32) acc = fmaf(__bfloat162float(ar[k]), __bfloat162float(xr[k]), acc);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0) ta[(size_t)m * r2 + j] = __half_as_ushort(__float2half_rn(lora_scale * acc));
    }
  }
}

// bf16 [M, K] -> binary16 [M, lda16] (zero padded), the down GEMM's A operand.
__global__ void __launch_bounds__(256) to_f16_kernel(const __nv_bfloat16 *x, int M, int K, int lda16, uint16_t *x16) {
  const size_t n = (size_t)M * lda16;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const size_t m = i / lda16, k = i % lda16;
    x16[i] = k < (size_t)K ? __half_as_ushort(__float2half_rn(__bfloat162float(x[m * K + k]))) : (uint16_t)0;
  }
}

template <int BITS, int NPROJ, int GROUP, bool EXACT>
cudaError_t launch_gemm_t(const GemmArgs &a, cudaStream_t s) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  auto kern = qgemm_kernel<BITS, NPROJ, GROUP, EXACT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const dim3 grid((a.M + kBM - 1) / kBM, (a.N + kBN - 1) / kBN);
  kern<<<grid, kGemmThreads, C::SMEM, s>>>(a);
  return cudaGetLastError();
}

template <int BITS, int NPROJ, bool EXACT>
cudaError_t launch_gemm_g(const GemmArgs &a, cudaStream_t s) {
  switch (a.group) {
    case 32: return launch_gemm_t<BITS, NPROJ, 32, EXACT>(a, s);
    case 64: return launch_gemm_t<BITS, NPROJ, 64, EXACT>(a, s);
    default: return launch_gemm_t<BITS, NPROJ, 128, EXACT>(a, s);
  }
}

}  // namespace

cudaError_t launch_gemm(GemvKind kind, const GemmArgs &a, cudaStream_t s) {
  if (a.M <= 0) return cudaSuccess;
  switch (kind) {
    case kGateUpW2: return launch_gemm_g<2, 2, false>(a, s);
    case kGateUpW4: return launch_gemm_g<4, 2, false>(a, s);
    default: return a.out_f32 ? launch_gemm_g<4, 1, true>(a, s) : launch_gemm_g<4, 1, false>(a, s);
  }
}

cudaError_t launch_gemm_prep(const void *x, int M, int K, int lda16, const void *lora_a, int r2, float lora_scale,
                             uint16_t *x16, float *rs, uint16_t *ta, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  gemm_prep_kernel<<<M, 256, 0, s>>>(reinterpret_cast<const __nv_bfloat16 *>(x), M, K, lda16,
                                     reinterpret_cast<const __nv_bfloat16 *>(lora_a), r2, lora_scale, x16, rs, ta);
  return cudaGetLastError();
}

cudaError_t launch_to_f16(const void *x, int M, int K, int lda16, uint16_t *x16, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  const size_t n = (size_t)M * lda16;
  const int blocks = (int)std::min<size_t>((n + 255) / 256, 4096);
  to_f16_kernel<<<blocks, 256, 0, s>>>(reinterpret_cast<const __nv_bfloat16 *>(x), M, K, lda16, x16);
  return cudaGetLastError();
}

cudaError_t read_gemm_status(int *status) {
  int v = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_gemm_status, sizeof(int));
  if (e != cudaSuccess) return e;
  const int zero = 0;
  e = cudaMemcpyToSymbol(g_gemm_status, &zero, sizeof(int));
  *status = v;
  return e;
}

int gemm_stages(GemvKind kind, int group) {
  switch (kind * 3 + (group == 32 ? 0 : group == 64 ? 1 : 2)) {
    case 0: return GemmCfg<2, 2, 32, false>::S;
    case 1: return GemmCfg<2, 2, 64, false>::S;
    case 2: return GemmCfg<2, 2, 128, false>::S;
    case 3: return GemmCfg<4, 2, 32, false>::S;
    case 4: return GemmCfg<4, 2, 64, false>::S;
    case 5: return GemmCfg<4, 2, 128, false>::S;
    case 6: return GemmCfg<4, 1, 32, false>::S;
    case 7: return GemmCfg<4, 1, 64, false>::S;
    default: return GemmCfg<4, 1, 128, false>::S;
  }
}

}  // namespace wq
