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
// gate/up) over the whole feature axis, 64 features (half a block of the
// packed format) per pipeline stage.  Warp roles:
//   warps 0..15 dequantize the stage's codes: code q of row n, group j gives
//               the binary16 value s_nj (q - z_nj), rounded once; they write
//               it in the tcgen05 K-major layout (8-row x 16-byte core
//               matrices), warps 0..3 then run the epilogue from TMEM;
//   warp 16     loads the binary16 activation tile with the tensor-memory
//               accelerator (TMA; zero fill outside the matrix);
//   warp 17     owns the TMEM allocation; its lane 0 issues the MMAs;
//   warp 18     loads the packed codes and scales/zeros of the CTA's 8 row
//               tiles (TMA, one box each per projection and stage) into their
//               own ring, which runs a stage further ahead than the tiles.
// Stages are handed over with mbarriers; every wait is bounded (a timeout
// sets the device status word and the CTA skips the rest of its work).
#include <algorithm>
#include <cmath>
#include <mutex>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "wq_internal.h"
#include "wq_ptx.cuh"

namespace wq {

// Device status word of the GEMM kernels: WQ_OK (0) or WQ_ERR_TIMEOUT (-6).
__device__ int g_gemm_status = 0;

namespace {

constexpr int kBM = 128;                         // tokens per CTA tile (MMA M)
constexpr int kBN = 128;                         // output rows per CTA tile and projection (MMA N)
constexpr int kDeqWarps = 16;                    // dequantizing warps
constexpr int kProducerWarp = kDeqWarps;         // activation tiles
constexpr int kMmaWarp = kDeqWarps + 1;          // TMEM owner and MMA issuer
constexpr int kRawWarp = kDeqWarps + 2;          // packed-code ring
constexpr int kGemmThreads = (kDeqWarps + 3) * 32;
constexpr int kTileBytes = kBM * 64 * 2;         // one 128 x 64 binary16 operand tile (a stage)
constexpr uint32_t kSboTile = 8 * 128;           // bytes between 8-row groups of a 64-feature B tile
constexpr int kLoraK = 32;                       // LoRA rank columns a stage
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
  static constexpr int RAWP = 8 * RAW_TILE;                // a projection's: [8 tiles][codes], then [8 tiles][meta]
  static constexpr int RAW = NPROJ * RAWP;                 // a block's packed weights (two stages)
  static constexpr int TILES = kTileBytes + NB * kTileBytes;  // a stage's operand tiles
  static constexpr int AVAIL = (int)kGemmSmemLimit - 1024;
  // stages: as many as leave room for two blocks of packed codes, at most 4;
  // code ring: the rest, at most 4 blocks
  static constexpr int S = std::min(4, (AVAIL - 2 * RAW) / TILES);
  static constexpr int R = std::min(4, (AVAIL - S * TILES) / RAW);
  static_assert(S >= 2 && R >= 2, "GEMM pipeline does not fit");
  static constexpr int OFF_A = 0;
  static constexpr int OFF_B = S * kTileBytes;
  static constexpr int OFF_RAW = OFF_B + S * NB * kTileBytes;
  static constexpr int OFF_BAR = OFF_RAW + R * RAW;        // 3 S + 2 R + 1 barriers
  static constexpr int SMEM = OFF_BAR + (3 * S + 2 * R + 2) * 8 + 16;
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

// The tensor maps of a launch: the activations, and per projection the packed
// codes viewed as [RT][KB * BPK / 128][128 bytes] and the scales/zeros as
// [RT][KB * GPB][64 bytes].
struct GemmMaps {
  CUtensorMap act, codes[2], meta[2];
};

// 3-D TMA load (coordinates innermost first), completing on `bar`.
__device__ __forceinline__ void tma_load_3d(void *dst, const CUtensorMap *map, int x, int y, int z, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
          smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}

// 2-D TMA load of a box of the activations into shared memory, completing
// on `bar` with its byte count.  x (the feature coordinate) is a multiple of 8.
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int x, int y, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

template <int BITS, int NPROJ, int GROUP, bool EXACT>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_kernel(const GemmArgs a, const __grid_constant__ GemmMaps tm) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  constexpr int S = C::S, R = C::R, GPB = C::GPB, GS = GROUP / 16;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint64_t *raw_full = reinterpret_cast<uint64_t *>(smem + C::OFF_BAR);
  uint64_t *raw_empty = raw_full + R;
  uint64_t *a_full = raw_empty + R;
  uint64_t *b_full = a_full + S;
  uint64_t *empty = b_full + S;
  uint64_t *acc_full = empty + S;
  uint32_t *tmem_s = reinterpret_cast<uint32_t *>(acc_full + 2);
  volatile int *abort_s = reinterpret_cast<volatile int *>(tmem_s + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * kBN;
  const int KB = (a.K + 127) / 128;
  const int nws = 2 * KB;  // weight stages (64 features each)
  const int nlora = NPROJ == 2 && a.r > 0 ? (a.r + kLoraK - 1) / kLoraK : 0;
  const int nit = nws + nlora;

  if (tid == 0) {
    for (int q = 0; q < R; ++q) {
      mbar_init(&raw_full[q], 1);
      mbar_init(&raw_empty[q], kDeqWarps);
    }
    for (int s = 0; s < S; ++s) {
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

  if (warp == kRawWarp) {
    // ---- packed codes and scales/zeros (TMA) into their ring; row tiles
    // past the matrix read as zeros ----
    if (lane == 0)
      for (int it = 0; it < KB; ++it) {
        const int q = it % R;
        if (it >= R && !wait(&raw_empty[q], (it / R - 1) & 1)) break;
        mbar_arrive_expect_tx(&raw_full[q], (uint32_t)C::RAW);
        for (int p = 0; p < NPROJ; ++p) {
          uint8_t *dst = smem + C::OFF_RAW + q * C::RAW + p * C::RAWP;
          tma_load_3d(dst, &tm.codes[p], 0, it * (C::BPK / 128), n0 / 16, &raw_full[q]);
          tma_load_3d(dst + 8 * C::BPK, &tm.meta[p], 0, it * GPB, n0 / 16, &raw_full[q]);
        }
      }
    __syncwarp();
  } else if (warp == kProducerWarp) {
    // ---- activation tiles (TMA); the LoRA stage's by cp.async ----
    for (int it = 0; it < nit; ++it) {
      const int s = it % S, u = it / S;
      if (it >= S && !wait(&empty[s], (u - 1) & 1)) break;
      uint8_t *As = smem + C::OFF_A + s * kTileBytes;
      if (it < nws) {
        if (lane == 0) {
          // activation tile: 8 boxes of 8 features x 128 tokens, box c landing
          // at c * 2 KB (K-major: core matrices 2 KB apart along K, 8-row
          // groups 128 bytes apart)
          mbar_arrive_expect_tx(&a_full[s], (uint32_t)kTileBytes);
          for (int c = 0; c < 8; ++c) tma_load_2d(As + c * 2048, &tm.act, it * 64 + c * 8, m0, &a_full[s]);
        }
      } else {
        // LoRA stage l: lora_scale * t, rank columns 32 l .. 32 l + 31 of gate
        // (first r columns of ta) and of up (next r), zeros past r
        const int l = it - nws;
        for (int i = lane; i < NPROJ * kBM * 4; i += 32) {
          const int p = i / (kBM * 4), rem = i - p * kBM * 4;
          const int ml = rem >> 2, c = rem & 3;
          const int m = m0 + ml, col = l * kLoraK + c * 8;
          const bool ok = m < a.M && col < a.r;
          const uint16_t *src = ok ? a.ta + (size_t)m * 2 * a.r + p * a.r + col : a.ta;
          cp_async16_zfill(As + p * (kBM * kLoraK * 2) + kmajor_off(ml, c * 8, 4 * 128u), src, ok ? 16u : 0u);
        }
        // once landed, each lane fences its generic-proxy writes against the
        // tensor cores' reads, then lane 0 arrives
        cp_async_wait_all();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&a_full[s]);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---- MMA issue ----
    if (lane == 0) {
      // gate/up: one MMA of N = 256 a k-step (the gate tile and the up tile
      // are adjacent, 256 rows), so the activation tile is read once
      constexpr uint32_t idesc = umma_idesc_f16(kBM, kBN);
      constexpr uint32_t idesc2 = umma_idesc_f16(kBM, 2 * kBN);
      for (int it = 0; it < nit; ++it) {
        const int s = it % S, u = it / S;
        if (!wait(&a_full[s], u & 1) || !wait(&b_full[s], u & 1)) break;
        tc_fence_after();
        const uint32_t as = smem_addr(smem + C::OFF_A + s * kTileBytes);
        const uint32_t bs = smem_addr(smem + C::OFF_B + s * C::NB * kTileBytes);
        if (it < nws && NPROJ == 2 && !EXACT) {
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_f16(tmem, umma_desc_kmajor(as + ks * 4096, 2048, 128), umma_desc_kmajor(bs + ks * 256, 128, kSboTile),
                     idesc2, (it > 0 || ks > 0) ? 1u : 0u);
        } else if (it < nws) {
#pragma unroll
          for (int p = 0; p < NPROJ; ++p)
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
              // A (TMA layout): k-step ks = core matrices 2 ks and 2 ks + 1, 2 KB apart
              umma_f16(tmem + p * kBN, umma_desc_kmajor(as + ks * 4096, 2048, 128),
                       umma_desc_kmajor(bs + p * kTileBytes + ks * 256, 128, kSboTile), idesc, (it > 0 || ks > 0) ? 1u : 0u);
              if (EXACT)  // the low parts of the same weights
                umma_f16(tmem + p * kBN, umma_desc_kmajor(as + ks * 4096, 2048, 128),
                         umma_desc_kmajor(bs + (NPROJ + p) * kTileBytes + ks * 256, 128, kSboTile), idesc, 1u);
            }
        } else {
          constexpr uint32_t sbo = 4 * 128u;  // 32 rank columns a LoRA stage
          for (int p = 0; p < NPROJ; ++p)
            for (int ks = 0; ks < kLoraK / 16; ++ks)
              umma_f16(tmem + p * kBN, umma_desc_kmajor(as + p * (kBM * kLoraK * 2) + ks * 256, 128, sbo),
                       umma_desc_kmajor(bs + p * (kBN * kLoraK * 2) + ks * 256, 128, sbo), idesc, 1u);
        }
        umma_commit(&empty[s]);
      }
      umma_commit(acc_full);
    }
    __syncwarp();
  } else {
    // ---- dequantization into the B tiles ----
    const int dt = tid;  // 0 .. kDeqWarps * 32 - 1
    for (int it = 0; it < nit; ++it) {
      const int s = it % S, u = it / S, kb = it >> 1, hb = it & 1, q = kb % R;
      if (it < nws && !wait(&raw_full[q], (kb / R) & 1)) break;
      if (it >= S && !wait(&empty[s], (u - 1) & 1)) break;
      uint8_t *Bs = smem + C::OFF_B + s * C::NB * kTileBytes;
      if (it < nws) {
        const uint8_t *raw = smem + C::OFF_RAW + q * C::RAW;
        // item = (projection, 16-row tile, lane of the packed fragment layout)
        for (int item = dt; item < NPROJ * 8 * 32; item += kDeqWarps * 32) {
          const int p = item >> 8, j = (item >> 5) & 7, L = item & 31;
          const int g = L >> 2, t = L & 3;
          uint8_t *Bp = Bs + p * kTileBytes;
          // the lane's code words of this half block: 2-bit, words 2 hb, 2 hb + 1
          // of its 16 bytes; 4-bit, the 16 bytes of half hb
          uint32_t wds[BITS == 2 ? 2 : 4];
          const uint8_t *cb = raw + p * C::RAWP + j * C::BPK;               // codes of tile j
          const uint8_t *mb = raw + p * C::RAWP + 8 * C::BPK + j * GPB * 64;  // its scales/zeros
          if (BITS == 2) {
            const uint2 w0 = lds64(cb + L * 16 + hb * 8);
            wds[0] = w0.x; wds[1] = w0.y;
          } else {
            const uint4 w0 = lds128(cb + hb * 512 + L * 16);
            wds[0] = w0.x; wds[1] = w0.y; wds[2] = w0.z; wds[3] = w0.w;
          }
          // this stage: k-steps 4 hb .. 4 hb + 3 of the block
#pragma unroll
          for (int gl = 0; gl < (GS >= 4 ? 1 : 4 / GS); ++gl) {
            const int gi = (4 * hb) / GS + gl;
            // scales and zeros of rows g and g + 8 in group gi (zero for tiles outside the matrix)
            const uint2 sz = lds64(mb + gi * 64 + g * 8);
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
            for (int kk = 0; kk < (GS >= 4 ? 4 : GS); ++kk) {
              const int ks = (GS >= 4 ? 4 * hb : gi * GS) + kk;
              uint32_t q[4];  // (row g, k 2t..2t+1), (row g+8, ...), (row g, k 2t+8..), (row g+8, k 2t+8..)
              const int kl = ks - 4 * hb;  // k-step within the half block
              if (BITS == 2) {
                const uint32_t x = wds[(kl >> 1) & 1];
                const int s4 = (kl & 1) * 4;
                q[0] = (x >> s4) & 0x00030003u;
                q[1] = (x >> (s4 + 8)) & 0x00030003u;
                q[2] = (x >> (s4 + 2)) & 0x00030003u;
                q[3] = (x >> (s4 + 10)) & 0x00030003u;
              } else {
                const uint32_t x = wds[kl & 3];
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
                const int k = kl * 16 + 2 * t + ((e & 2) ? 8 : 0);  // within the stage
                *reinterpret_cast<uint32_t *>(Bp + kmajor_off(row, k, kSboTile)) = h2bits(w);
                if (EXACT)
                  *reinterpret_cast<uint32_t *>(Bp + NPROJ * kTileBytes + kmajor_off(row, k, kSboTile)) =
                      h2bits(__hmul2(qz, hi_row ? t_hi : t_lo));
              }
            }
          }
        }
      } else {
        // LoRA stage l: B_p rows n0 .. n0+127 (bf16 [N][r]), rank columns
        // 32 l .. 32 l + 31 -> binary16, zeros past r
        const int l = it - nws;
        constexpr uint32_t sbo = 4 * 128u;
        for (int i = dt; i < NPROJ * kBN * 4; i += kDeqWarps * 32) {
          const int p = i / (kBN * 4), rem = i - p * kBN * 4;
          const int nl = rem >> 2, c = rem & 3;
          const int n = n0 + nl, col = l * kLoraK + c * 8;
          uint4 v = make_uint4(0u, 0u, 0u, 0u);
          if (n < a.N && col < a.r) v = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const uint8_t *>(a.lora_b[p]) + ((size_t)n * a.r + col) * 2));
          const uint32_t w[4] = {v.x, v.y, v.z, v.w};
          uint32_t o[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float lo = __uint_as_float(w[e] << 16), hi = __uint_as_float(w[e] & 0xffff0000u);
            o[e] = h2bits(__floats2half2_rn(lo, hi));
          }
          *reinterpret_cast<uint4 *>(Bs + p * (kBN * kLoraK * 2) + kmajor_off(nl, c * 8, sbo)) = make_uint4(o[0], o[1], o[2], o[3]);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&b_full[s]);
        if (it < nws && hb == 1) mbar_arrive(&raw_empty[q]);  // both halves of this block's codes are read
      }
    }

    // ---- epilogue (warps 0..3: TMEM lanes 32 w .. 32 w + 31 = tokens) ----
    if (warp < 4 && wait(acc_full, 0)) {
      tc_fence_after();
      const int m = m0 + warp * 32 + lane;
      const float rs = (NPROJ == 2 && a.rs != nullptr && m < a.M) ? a.rs[m] : 1.f;
      const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
      // rows n0 + c .. n0 + c + 7 of this token: 16-byte stores when the
      // row length allows (N a multiple of 8), element stores otherwise
      const bool vec = (a.N & 7) == 0 && (!a.out_f16 || (a.ldo16 & 7) == 0);
      for (int c = 0; c < kBN; c += 8) {
        uint32_t g[8], uu[8];
        tmem_ld8(tl + c, g);
        if (NPROJ == 2) tmem_ld8(tl + kBN + c, uu);
        tmem_ld_wait();
        const int nb = n0 + c;
        if (m >= a.M || nb >= a.N) continue;
        float v[8];
        if (NPROJ == 2) {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float gv = rs * __uint_as_float(g[e]), uv = rs * __uint_as_float(uu[e]);
            v[e] = __bfloat162float(__float2bfloat16_rn(gv / (1.f + __expf(-gv)) * uv));  // h as stored
          }
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) v[e] = __uint_as_float(g[e]);
          if (a.residual) {
            if (vec) {
              const uint4 rv = *reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(a.residual) +
                                                                (size_t)m * a.N + nb);
              const uint32_t rw[4] = {rv.x, rv.y, rv.z, rv.w};
#pragma unroll
              for (int e = 0; e < 8; ++e) v[e] += __uint_as_float(e & 1 ? (rw[e >> 1] & 0xffff0000u) : (rw[e >> 1] << 16));
            } else {
              for (int e = 0; e < 8 && nb + e < a.N; ++e)
                v[e] += __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(a.residual)[(size_t)m * a.N + nb + e]);
            }
          }
        }
        if (vec) {
          if (NPROJ == 1 && a.out_f32) {
            float4 *o = reinterpret_cast<float4 *>(reinterpret_cast<float *>(a.out) + (size_t)m * a.N + nb);
            o[0] = make_float4(v[0], v[1], v[2], v[3]);
            o[1] = make_float4(v[4], v[5], v[6], v[7]);
          } else {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const __nv_bfloat162 b2 = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
              w[e] = *reinterpret_cast<const uint32_t *>(&b2);
            }
            *reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(a.out) + (size_t)m * a.N + nb) =
                make_uint4(w[0], w[1], w[2], w[3]);
            if (NPROJ == 2 && a.out_f16) {
#pragma unroll
              for (int e = 0; e < 4; ++e) w[e] = h2bits(__floats2half2_rn(v[2 * e], v[2 * e + 1]));
              *reinterpret_cast<uint4 *>(a.out_f16 + (size_t)m * a.ldo16 + nb) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
        } else {
          for (int e = 0; e < 8 && nb + e < a.N; ++e) {
            const size_t o = (size_t)m * a.N + nb + e;
            if (NPROJ == 1 && a.out_f32) {
              reinterpret_cast<float *>(a.out)[o] = v[e];
            } else {
              reinterpret_cast<__nv_bfloat16 *>(a.out)[o] = __float2bfloat16_rn(v[e]);
              if (NPROJ == 2 && a.out_f16) a.out_f16[(size_t)m * a.ldo16 + nb + e] = __half_as_ushort(__float2half_rn(v[e]));
            }
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
// A CTA takes kPrepTok tokens, staged in shared memory, so that every LoRA-A
// row it reads serves all of them; fixed-order reductions.
constexpr int kPrepTok = 4;

__global__ void __launch_bounds__(256) gemm_prep_kernel(const __nv_bfloat16 *x, int M, int K, int lda16,
                                                        const __nv_bfloat16 *lora_a, int r2, float lora_scale,
                                                        uint16_t *x16, float *rs, uint16_t *ta) {
  extern __shared__ __align__(16) __nv_bfloat16 xs[];  // [kPrepTok][K]
  __shared__ float red[kPrepTok][8];
  const int m0 = blockIdx.x * kPrepTok, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nt = min(kPrepTok, M - m0);
  float ss[kPrepTok];
#pragma unroll
  for (int t = 0; t < kPrepTok; ++t) ss[t] = 0.f;
#pragma unroll
  for (int t = 0; t < kPrepTok; ++t) {
    if (t >= nt) break;
    const __nv_bfloat16 *xr = x + (size_t)(m0 + t) * K;
    for (int k = tid; k < K; k += blockDim.x) {
      const __nv_bfloat16 bv = xr[k];
      const float v = __bfloat162float(bv);
      xs[t * K + k] = bv;
      ss[t] = fmaf(v, v, ss[t]);
      x16[(size_t)(m0 + t) * lda16 + k] = __half_as_ushort(__float2half_rn(v));
    }
    for (int k = K + tid; k < lda16; k += blockDim.x) x16[(size_t)(m0 + t) * lda16 + k] = 0;
  }
#pragma unroll
  for (int t = 0; t < kPrepTok; ++t) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss[t] += __shfl_xor_sync(0xffffffffu, ss[t], o);
    if (lane == 0) red[t][warp] = ss[t];
  }
  __syncthreads();
  if (tid < nt) {
    float tot = 0.f;
    for (int w = 0; w < 8; ++w) tot += red[tid][w];
    rs[m0 + tid] = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(tot, (float)K), kRmsEps)));
  }
  if (r2 > 0) {
    // warp w takes LoRA-A rows w, w + 8, ...: lanes stride the features, then the warp adds up
    for (int j = warp; j < r2; j += 8) {
      const __nv_bfloat16 *ar = lora_a + (size_t)j * K;
      float acc[kPrepTok];
#pragma unroll
      for (int t = 0; t < kPrepTok; ++t) acc[t] = 0.f;
      for (int k = lane; k < K; k += 32) {
        const float av = __bfloat162float(ar[k]);
#pragma unroll
        for (int t = 0; t < kPrepTok; ++t) acc[t] = fmaf(av, __bfloat162float(xs[t * K + k]), acc[t]);
      }
#pragma unroll
      for (int t = 0; t < kPrepTok; ++t) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[t] += __shfl_xor_sync(0xffffffffu, acc[t], o);
        if (lane == 0 && t < nt) ta[(size_t)(m0 + t) * r2 + j] = __half_as_ushort(__float2half_rn(lora_scale * acc[t]));
      }
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

// cuTensorMapEncodeTiled from the driver (looked up once).
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Tensor maps of a launch (zero fill outside every tensor):
//   activations [M][lda] binary16, boxes of 8 features x 128 tokens;
//   codes [RT][KB * BPK / 128][128 B], boxes of one block of 8 row tiles;
//   scales/zeros [RT][KB * GPB][64 B], boxes of one block of 8 row tiles.
cudaError_t make_maps(const GemmArgs &a, int nproj, int bits, GemmMaps *m) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint32_t e1[3] = {1, 1, 1};
  {
    const cuuint64_t dims[2] = {(cuuint64_t)a.K, (cuuint64_t)a.M};
    const cuuint64_t strides[1] = {(cuuint64_t)a.lda * 2};
    const cuuint32_t box[2] = {8, (cuuint32_t)kBM};
    if (fn(&m->act, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<uint16_t *>(a.act), dims, strides, box, e1,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const cuuint64_t RT = (cuuint64_t)(a.N + 15) / 16, KB = (cuuint64_t)(a.K + 127) / 128;
  const cuuint64_t bpk = bits == 2 ? 512 : 1024, gpb = 128 / a.group;
  for (int p = 0; p < 2; ++p) {
    const int src = p < nproj ? p : 0;  // unused second map of the down kernel: a copy of the first
    {
      const cuuint64_t dims[3] = {128, KB * bpk / 128, RT};
      const cuuint64_t strides[2] = {128, KB * bpk};
      const cuuint32_t box[3] = {128, (cuuint32_t)(bpk / 128), 8};
      if (fn(&m->codes[p], CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint32_t *>(a.codes[src]), dims, strides, box, e1,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    }
    {
      const cuuint64_t dims[3] = {64, KB * gpb, RT};
      const cuuint64_t strides[2] = {64, KB * gpb * 64};
      const cuuint32_t box[3] = {64, (cuuint32_t)gpb, 8};
      if (fn(&m->meta[p], CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint16_t *>(a.meta[src]), dims, strides, box, e1,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    }
  }
  return cudaSuccess;
}

template <int BITS, int NPROJ, int GROUP, bool EXACT>
cudaError_t launch_gemm_t(const GemmArgs &a, cudaStream_t s) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  auto kern = qgemm_kernel<BITS, NPROJ, GROUP, EXACT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  GemmMaps maps;
  if ((e = make_maps(a, NPROJ, BITS, &maps)) != cudaSuccess) return e;
  const dim3 grid((a.M + kBM - 1) / kBM, (a.N + kBN - 1) / kBN);
  kern<<<grid, kGemmThreads, C::SMEM, s>>>(a, maps);
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
  const size_t smem = (size_t)kPrepTok * K * 2;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(gemm_prep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  gemm_prep_kernel<<<(M + kPrepTok - 1) / kPrepTok, 256, smem, s>>>(
      reinterpret_cast<const __nv_bfloat16 *>(x), M, K, lda16, reinterpret_cast<const __nv_bfloat16 *>(lora_a), r2,
      lora_scale, x16, rs, ta);
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
