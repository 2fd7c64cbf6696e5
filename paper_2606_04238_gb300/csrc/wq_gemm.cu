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
// A CTA computes a tile of 128 or 256 tokens x 128 output rows (x 2
// projections for gate/up) over the whole feature axis, 64 features (half a
// block of the packed format) per pipeline stage; with 256 tokens the two
// halves of 128 multiply the same dequantized B tile into accumulators of
// their own, so each weight is dequantized once per 256 tokens.  Warp roles:
//   warps 0..15 dequantize the stage's codes: code q of row n, group j gives
//               the binary16 value s_nj (q - z_nj), rounded once; they write
//               it in the tcgen05 K-major layout (8-row x 16-byte core
//               matrices), then run the epilogue from TMEM;
//   warp 16     loads the binary16 activation tile with the tensor-memory
//               accelerator (TMA; one box of 64 features x 128 tokens in the
//               128-byte swizzled layout, zero fill outside the matrix);
//   warp 17     owns the TMEM allocation; its lane 0 issues the MMAs;
//   warp 18     loads the packed codes and scales/zeros of the CTA's 8 row
//               tiles (TMA, one box each per projection and block) into their
//               own ring.
// The activation tiles, the B tiles and the packed codes have rings of their
// own depths: each slot is released by what last reads it (the MMAs' commit,
// or the dequantizing warps for the codes).
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
constexpr int kHalves = 2;                       // token halves of kBM a CTA can take (GemmArgs::mt)
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
  static constexpr int BT = NB * kTileBytes;               // a stage's B tiles
  static constexpr int AT = kHalves * kTileBytes;          // a stage's activation tiles (both token halves)
  // 1 KB for the barriers, 1 KB to align the tiles on 1024 bytes
  static constexpr int AVAIL = (int)kGemmSmemLimit - 2048;
  // Three rings.  The activation tiles come from L2 with a long latency, so
  // their ring is the deepest (up to 8 stages); the B tiles are made on chip
  // and need only 3 (2 where 3 would leave fewer than 4 activation stages);
  // the packed codes (blocks of two stages) take what is left, at most 6.
  static constexpr int SB = (AVAIL - 3 * BT - 3 * RAW) / AT >= 4 ? 3 : 2;
  static constexpr int SA = std::min(8, (AVAIL - SB * BT - 3 * RAW) / AT);
  static constexpr int R = std::min(6, (AVAIL - SA * AT - SB * BT) / RAW);
  static_assert(SA >= 2 && R >= 2, "GEMM pipeline does not fit");
  static constexpr int OFF_A = 0;
  static constexpr int OFF_B = SA * AT;
  static constexpr int OFF_RAW = OFF_B + SB * BT;
  static constexpr int OFF_BAR = OFF_RAW + R * RAW;
  static constexpr int SMEM = OFF_BAR + (2 * SA + 2 * SB + 2 * R + 2) * 8 + 16 + 1024;  // + alignment slack
  static constexpr int NCH = NPROJ * kBN;                  // TMEM columns of a token half (fp32 accumulators)
  static constexpr int NCOLS = kHalves * NCH;
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
// on `bar` with its byte count.  x (the feature coordinate) is a multiple of 64.
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int x, int y, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

// The epilogue of one part of a tile (the 16 dequantizing warps, after the
// part's accumulators are complete; `have`: no timeout so far).  Warp w reads
// TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31 (the tokens of each half) and
// columns 32 (w / 4) .. 32 (w / 4) + 31.  A whole tile is finished from TMEM;
// a part of a split tile is written to its scratch slot, and the CTA that adds
// the tile's last part to its counter sums the parts in k order (their CTAs
// are consecutive) and finishes the tile.  Kept out of line so that the
// dequantization loop keeps its registers.
// ---------------------------------------------------------------------------
// Pieces shared by the two kernels below.
// ---------------------------------------------------------------------------

// Dequantizes the stage hb (features 64 hb .. 64 hb + 63) of a block of
// packed codes `raw` into the B tiles `Bs`; thread dt of the 16 dequantizing
// warps takes the items (projection, 16-row tile, lane of the fragment layout)
// dt, dt + 512, ...
template <int BITS, int NPROJ, int GROUP, bool EXACT>
__device__ __forceinline__ void gemm_deq_stage(const uint8_t *raw, uint8_t *Bs, int hb, int dt) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  constexpr int GPB = C::GPB, GS = GROUP / 16;
  for (int item = dt; item < NPROJ * 8 * 32; item += kDeqWarps * 32) {
    const int p = item >> 8, j = (item >> 5) & 7, L = item & 31;
    const int g = L >> 2;
    uint8_t *Bp = Bs + p * kTileBytes;
    // the lane's code words of this half block: 2-bit, words 2 hb, 2 hb + 1
    // of its 16 bytes; 4-bit, the 16 bytes of half hb
    uint32_t wds[BITS == 2 ? 2 : 4];
    const uint8_t *cb = raw + p * C::RAWP + j * C::BPK;               // codes of tile j
    const uint8_t *mb = raw + p * C::RAWP + 8 * C::BPK + j * GPB * 64;  // its scales/zeros
    if (BITS == 2) {
      const uint2 w0 = lds64(cb + L * 16 + hb * 8);
      wds[0] = w0.x;
      wds[1] = w0.y;
    } else {
      const uint4 w0 = lds128(cb + hb * 512 + L * 16);
      wds[0] = w0.x;
      wds[1] = w0.y;
      wds[2] = w0.z;
      wds[3] = w0.w;
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
      const __half2 t_lo = __half2half2(
          __hsub(__ushort_as_half((unsigned short)sg), __ushort_as_half((unsigned short)(sg & 0xfff0u))));
      const __half2 t_hi = __half2half2(
          __hsub(__ushort_as_half((unsigned short)sg8), __ushort_as_half((unsigned short)(sg8 & 0xfff0u))));
      // 1024 + z: the code read as 1024 + q minus this is q - z exactly
      const __half2 z_lo =
          __half2half2(__hadd(__ushort_as_half((unsigned short)(sz.y & 0xffffu)), __float2half(1024.f)));
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
        uint32_t w[4], wl[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __half2 v = bits2h(q[e] | 0x64006400u);  // 1024 + q, exact
          const bool hi_row = (e & 1) != 0;
          const __half2 qz = __hsub2(v, hi_row ? z_hi : z_lo);  // q - z, exact
          w[e] = h2bits(__hmul2(qz, hi_row ? s_hi : s_lo));
          if (EXACT) wl[e] = h2bits(__hmul2(qz, hi_row ? t_hi : t_lo));
        }
        // the four 8x8 blocks (rows +0/+8, k +0/+8) of this k-step are core
        // matrices of the K-major tile: one matrix store; lane L gives row
        // L % 8 of block L / 8
        const int blk = L >> 3;
        const uint32_t dst = smem_addr(Bp) + (uint32_t)(2 * j + (blk & 1)) * kSboTile +
                             (uint32_t)(2 * kl + (blk >> 1)) * 128u + (uint32_t)(L & 7) * 16u;
        stmatrix_x4(dst, w[0], w[1], w[2], w[3]);
        if (EXACT) stmatrix_x4(dst + NPROJ * kTileBytes, wl[0], wl[1], wl[2], wl[3]);
      }
    }
  }
}

// LoRA stage l, B side: rows n0 .. n0 + 127 of B_p (bf16 [N][r]), rank
// columns 32 l .. 32 l + 31 -> binary16, zeros past r.
template <int NPROJ>
__device__ __forceinline__ void gemm_lora_b_stage(const GemmArgs &a, uint8_t *Bs, int n0, int l, int dt) {
  constexpr uint32_t sbo = 4 * 128u;
  for (int i = dt; i < NPROJ * kBN * 4; i += kDeqWarps * 32) {
    const int p = i / (kBN * 4), rem = i - p * kBN * 4;
    const int nl = rem >> 2, c = rem & 3;
    const int n = n0 + nl, col = l * kLoraK + c * 8;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (n < a.N && col < a.r)
      v = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const uint8_t *>(a.lora_b[p]) +
                                                ((size_t)n * a.r + col) * 2));
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float lo = __uint_as_float(w[e] << 16), hi = __uint_as_float(w[e] & 0xffff0000u);
      o[e] = h2bits(__floats2half2_rn(lo, hi));
    }
    *reinterpret_cast<uint4 *>(Bs + p * (kBN * kLoraK * 2) + kmajor_off(nl, c * 8, sbo)) =
        make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// LoRA stage l, A side (one warp): lora_scale * t, rank columns 32 l .. 32 l
// + 31 of gate (first r columns of ta) and of up (next r) for the mth token
// halves from m0, zeros past r; lane 0 arrives on `full` once all landed.
template <int NPROJ>
__device__ __forceinline__ void gemm_lora_a_stage(const GemmArgs &a, uint8_t *As, int m0, int mth, int l, int lane,
                                                  uint64_t *full) {
  for (int i = lane; i < mth * NPROJ * kBM * 4; i += 32) {
    const int h = i / (NPROJ * kBM * 4), hr = i - h * NPROJ * kBM * 4;
    const int p = hr / (kBM * 4), rem = hr - p * kBM * 4;
    const int ml = rem >> 2, c = rem & 3;
    const int m = m0 + h * kBM + ml, col = l * kLoraK + c * 8;
    const bool in = m < a.M && col < a.r;
    const uint16_t *src = in ? a.ta + (size_t)m * 2 * a.r + p * a.r + col : a.ta;
    cp_async16_zfill(As + h * kTileBytes + p * (kBM * kLoraK * 2) + kmajor_off(ml, c * 8, 4 * 128u), src,
                     in ? 16u : 0u);
  }
  // once landed, each lane fences its generic-proxy writes against the tensor
  // cores' reads, then lane 0 arrives
  cp_async_wait_all();
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) mbar_arrive(full);
}

// The MMAs of one stage (one thread): every token half multiplies the same B
// tile into its own accumulators; `first` starts the accumulators.
template <int NPROJ, bool EXACT>
__device__ __forceinline__ void gemm_issue_stage(uint32_t tmem, uint32_t as0, uint32_t bs, int mth, bool wstage,
                                                 bool first) {
  constexpr int NCH = NPROJ * kBN;
  // gate/up: one MMA of N = 256 a k-step (the gate tile and the up tile are
  // adjacent, 256 rows), so the activation tile is read once
  constexpr uint32_t idesc = umma_idesc_f16(kBM, kBN);
  constexpr uint32_t idesc2 = umma_idesc_f16(kBM, 2 * kBN);
  for (int h = 0; h < mth; ++h) {
    const uint32_t as = as0 + h * kTileBytes, th = tmem + h * NCH;
    if (wstage && NPROJ == 2 && !EXACT) {
#pragma unroll
      for (int ks = 0; ks < 4; ++ks)
        umma_f16(th, umma_desc_kmajor_sw128(as + ks * 32, 1024), umma_desc_kmajor(bs + ks * 256, 128, kSboTile), idesc2,
                 (first && ks == 0) ? 0u : 1u);
    } else if (wstage) {
#pragma unroll
      for (int p = 0; p < NPROJ; ++p)
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          // A (swizzled TMA layout): k-step ks at byte 32 ks of each row
          umma_f16(th + p * kBN, umma_desc_kmajor_sw128(as + ks * 32, 1024),
                   umma_desc_kmajor(bs + p * kTileBytes + ks * 256, 128, kSboTile), idesc,
                   (first && ks == 0) ? 0u : 1u);
          if (EXACT)  // the low parts of the same weights
            umma_f16(th + p * kBN, umma_desc_kmajor_sw128(as + ks * 32, 1024),
                     umma_desc_kmajor(bs + (NPROJ + p) * kTileBytes + ks * 256, 128, kSboTile), idesc, 1u);
        }
    } else {
      constexpr uint32_t sbo = 4 * 128u;  // 32 rank columns a LoRA stage
      for (int p = 0; p < NPROJ; ++p)
        for (int ks = 0; ks < kLoraK / 16; ++ks)
          umma_f16(th + p * kBN, umma_desc_kmajor(as + p * (kBM * kLoraK * 2) + ks * 256, 128, sbo),
                   umma_desc_kmajor(bs + p * (kBN * kLoraK * 2) + ks * 256, 128, sbo), idesc,
                   (first && ks == 0) ? 0u : 1u);
    }
  }
}

// Output of 8 consecutive rows nb .. nb + 7 of token m from the fp32 sums g
// (and u for gate/up): h = SiLU(rs g) * (rs u),
// or y = rs g + residual in bf16 or fp32 (rs: the token's factor that undoes
// the power-of-two scale of its binary16 activations, times its RMSNorm scale
// for gate/up).  `vec`: 16-byte stores (N a multiple of 8).
template <int NPROJ>
__device__ __forceinline__ void gemm_finish(const GemmArgs &a, int m, int nb, float rs, const float (&g)[8],
                                            const float (&u)[8], bool vec) {
  if (m >= a.M || nb >= a.N) return;
  float v[8];
  if (NPROJ == 2) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float gv = rs * g[e], uv = rs * u[e];
      v[e] = __bfloat162float(__float2bfloat16_rn(__fdividef(gv, 1.f + __expf(-gv)) * uv));  // h as stored
    }
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = rs * g[e];
    if (a.residual) {
      if (vec) {
        const uint4 rv =
            *reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(a.residual) + (size_t)m * a.N + nb);
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
    }
  } else {
    for (int e = 0; e < 8 && nb + e < a.N; ++e) {
      const size_t o = (size_t)m * a.N + nb + e;
      if (NPROJ == 1 && a.out_f32) {
        reinterpret_cast<float *>(a.out)[o] = v[e];
      } else {
        reinterpret_cast<__nv_bfloat16 *>(a.out)[o] = __float2bfloat16_rn(v[e]);
      }
    }
  }
}

// Shared memory of a launch: the barriers behind the rings, then the TMEM
// base address, the abort flag and the stream-K "last part" flag.
template <class C>
struct GemmSmem {
  uint8_t *base;
  uint64_t *raw_full, *raw_empty, *a_full, *a_empty, *b_full, *b_empty, *acc_full;
  uint32_t *tmem_s;
  volatile int *abort_s, *last_s;
  __device__ explicit GemmSmem(uint8_t *smem_raw) {
    // the swizzled activation tiles need 1024-byte alignment
    base = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    raw_full = reinterpret_cast<uint64_t *>(base + C::OFF_BAR);
    raw_empty = raw_full + C::R;
    a_full = raw_empty + C::R;
    a_empty = a_full + C::SA;
    b_full = a_empty + C::SA;
    b_empty = b_full + C::SB;
    acc_full = b_empty + C::SB;
    tmem_s = reinterpret_cast<uint32_t *>(acc_full + 2);
    abort_s = reinterpret_cast<volatile int *>(tmem_s + 1);
    last_s = abort_s + 1;
  }
  // thread 0: barrier initialisation; the MMA warp: TMEM allocation
  __device__ void init(int tid, int warp) {
    if (tid == 0) {
      for (int q = 0; q < C::R; ++q) {
        mbar_init(&raw_full[q], 1);
        mbar_init(&raw_empty[q], kDeqWarps);
      }
      for (int s = 0; s < C::SA; ++s) {
        mbar_init(&a_full[s], 1);
        mbar_init(&a_empty[s], 1);
      }
      for (int s = 0; s < C::SB; ++s) {
        mbar_init(&b_full[s], kDeqWarps);
        mbar_init(&b_empty[s], 1);
      }
      mbar_init(acc_full, 1);
      *abort_s = 0;
      fence_barrier_init();
    }
    if (warp == kMmaWarp) tmem_alloc(tmem_s, C::NCOLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  }
};

// ---------------------------------------------------------------------------
// One tile a CTA: grid (token tiles, row tiles).
// ---------------------------------------------------------------------------
template <int BITS, int NPROJ, int GROUP, bool EXACT>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_tile_kernel(const GemmArgs a, const __grid_constant__ GemmMaps tm) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  constexpr int SA = C::SA, SB = C::SB, R = C::R, GPB = C::GPB;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  GemmSmem<C> sm(smem_raw);
  uint8_t *smem = sm.base;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * a.mt * kBM, n0 = blockIdx.y * kBN;
  const int mth = min(a.mt, (a.M - m0 + kBM - 1) / kBM);  // token halves with tokens in them
  const int KB = (a.K + 127) / 128;
  const int nws = 2 * KB;  // weight stages (64 features each)
  const int nlora = NPROJ == 2 && a.r > 0 ? (a.r + kLoraK - 1) / kLoraK : 0;
  const int nit = nws + nlora;
  sm.init(tid, warp);
  const uint32_t tmem = *sm.tmem_s;

  // bounded wait; a timeout (or an earlier one) makes the caller skip its work
  auto wait = [&](uint64_t *bar, uint32_t parity) -> bool {
    if (*sm.abort_s) return false;
    if (mbar_wait_sleep(bar, parity)) return true;
    *sm.abort_s = 1;
    if (lane == 0) gemm_timeout();
    return false;
  };

  if (warp == kRawWarp) {
    // ---- packed codes and scales/zeros (TMA) into their ring; row tiles
    // past the matrix read as zeros ----
    if (lane == 0)
      for (int it = 0; it < KB; ++it) {
        const int q = it % R;
        if (it >= R && !wait(&sm.raw_empty[q], (it / R - 1) & 1)) break;
        mbar_arrive_expect_tx(&sm.raw_full[q], (uint32_t)C::RAW);
        for (int p = 0; p < NPROJ; ++p) {
          uint8_t *dst = smem + C::OFF_RAW + q * C::RAW + p * C::RAWP;
          tma_load_3d(dst, &tm.codes[p], 0, it * (C::BPK / 128), n0 / 16, &sm.raw_full[q]);
          tma_load_3d(dst + 8 * C::BPK, &tm.meta[p], 0, it * GPB, n0 / 16, &sm.raw_full[q]);
        }
      }
    __syncwarp();
  } else if (warp == kProducerWarp) {
    // ---- activation tiles (TMA); the LoRA stages' by cp.async ----
    for (int it = 0; it < nit; ++it) {
      const int s = it % SA;
      if (it >= SA && !wait(&sm.a_empty[s], (it / SA - 1) & 1)) break;
      uint8_t *As = smem + C::OFF_A + s * C::AT;
      if (it < nws) {
        if (lane == 0) {
          // per token half one box of 64 features x 128 tokens, a 128-byte row
          // per token, swizzled (8-row groups 1 KB apart)
          mbar_arrive_expect_tx(&sm.a_full[s], (uint32_t)(mth * kTileBytes));
          for (int h = 0; h < mth; ++h) tma_load_2d(As + h * kTileBytes, &tm.act, it * 64, m0 + h * kBM, &sm.a_full[s]);
        }
      } else {
        gemm_lora_a_stage<NPROJ>(a, As, m0, mth, it - nws, lane, &sm.a_full[s]);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---- MMA issue ----
    if (lane == 0) {
      for (int it = 0; it < nit; ++it) {
        const int sa = it % SA, sb = it % SB;
        if (!wait(&sm.a_full[sa], (it / SA) & 1) || !wait(&sm.b_full[sb], (it / SB) & 1)) break;
        tc_fence_after();
        gemm_issue_stage<NPROJ, EXACT>(tmem, smem_addr(smem + C::OFF_A + sa * C::AT),
                                       smem_addr(smem + C::OFF_B + sb * C::BT), mth, it < nws, it == 0);
        // both slots are free once these MMAs have read them
        umma_commit(&sm.a_empty[sa]);
        umma_commit(&sm.b_empty[sb]);
      }
      umma_commit(sm.acc_full);
    }
    __syncwarp();
  } else {
    // ---- dequantization into the B tiles ----
    for (int it = 0; it < nit; ++it) {
      const int s = it % SB, kb = it >> 1, hb = it & 1, q = kb % R;
      if (it < nws && !wait(&sm.raw_full[q], (kb / R) & 1)) break;
      if (it >= SB && !wait(&sm.b_empty[s], (it / SB - 1) & 1)) break;
      uint8_t *Bs = smem + C::OFF_B + s * C::BT;
      if (it < nws)
        gemm_deq_stage<BITS, NPROJ, GROUP, EXACT>(smem + C::OFF_RAW + q * C::RAW, Bs, hb, tid);
      else
        gemm_lora_b_stage<NPROJ>(a, Bs, n0, it - nws, tid);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&sm.b_full[s]);
        if (it < nws && hb == 1) mbar_arrive(&sm.raw_empty[q]);  // both halves of this block's codes are read
      }
    }

    // ---- epilogue: warp w reads TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31
    // (the tokens of each half) and columns 32 (w / 4) .. 32 (w / 4) + 31 ----
    if (wait(sm.acc_full, 0)) {
      tc_fence_after();
      const int quarter = warp & 3, c0 = (warp >> 2) * 32;
      const bool vec = (a.N & 7) == 0;
      for (int h = 0; h < mth; ++h) {
        const int m = m0 + h * kBM + quarter * 32 + lane;
        const float rs = (a.rs != nullptr && m < a.M) ? a.rs[m] : 1.f;
        const uint32_t tl = tmem + h * C::NCH + ((uint32_t)(quarter * 32) << 16);
        for (int c = c0; c < c0 + 32; c += 8) {
          uint32_t gw[8], uw[8];
          tmem_ld8(tl + c, gw);
          if (NPROJ == 2) tmem_ld8(tl + kBN + c, uw);
          tmem_ld_wait();
          float g[8], u[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            g[e] = __uint_as_float(gw[e]);
            u[e] = NPROJ == 2 ? __uint_as_float(uw[e]) : 0.f;
          }
          gemm_finish<NPROJ>(a, m, n0 + c, rs, g, u, vec);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, C::NCOLS);
}

// ---------------------------------------------------------------------------
// Stream-K: gridDim.x persistent CTAs divide the T * U work units evenly.
// ---------------------------------------------------------------------------
// The tiles (mt * 128 tokens x 128 rows) are cut into units of one
// 128-feature block (plus one unit for the LoRA stages); CTA c takes units
// [c W / P, (c + 1) W / P) of the W = T * U in order, i.e. whole tiles and at
// most one part of a tile at each end of its range.

// The epilogue of one part of a tile (the 16 dequantizing warps, after the
// part's accumulators are complete; `have`: no timeout so far).  Warp w reads
// TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31 (the tokens of each half) and
// columns 32 (w / 4) .. 32 (w / 4) + 31.  A whole tile is finished from TMEM;
// a part of a split tile is written to its scratch slot, and the CTA that adds
// the tile's last part to its counter sums the parts in k order (their CTAs
// are consecutive) and finishes the tile.  Kept out of line so that the
// dequantization loop keeps its registers.
template <int BITS, int NPROJ, int GROUP, bool EXACT>
__device__ __noinline__ void gemm_part_epilogue(const GemmArgs &a, uint32_t tmem, int tile, int ub, int ue, int U,
                                                long long W, long long P, long long g0, bool have,
                                                volatile int *abort_s, volatile int *last_s) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, c0 = (warp >> 2) * 32;
  const int MT = (a.M + a.mt * kBM - 1) / (a.mt * kBM);
  const int m0 = (tile % MT) * a.mt * kBM, n0 = (tile / MT) * kBN;
  const int mth = min(a.mt, (a.M - m0 + kBM - 1) / kBM);
  const bool vec = (a.N & 7) == 0;
  constexpr int SLOT = kHalves * kBM * C::NCH;  // floats of a scratch slot: [half][NCH / 8][128 tokens][8]
  const bool whole = ub == 0 && ue == U;
  // a split part's scratch slot: the CTA's first part (0) or its last (1)
  float *mine = whole ? nullptr : a.sk_part + ((size_t)blockIdx.x * 2 + ((long long)tile * U + ub == g0 ? 0 : 1)) * SLOT;
  for (int h = 0; h < mth && have; ++h) {
    const int m = m0 + h * kBM + quarter * 32 + lane;
    const float rs = (a.rs != nullptr && m < a.M) ? a.rs[m] : 1.f;
    const uint32_t tl = tmem + h * C::NCH + ((uint32_t)(quarter * 32) << 16);
    for (int c = c0; c < c0 + 32; c += 8) {
      uint32_t gw[8], uw[8];
      tmem_ld8(tl + c, gw);
      if (NPROJ == 2) tmem_ld8(tl + kBN + c, uw);
      tmem_ld_wait();
      float g[8], u[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        g[e] = __uint_as_float(gw[e]);
        u[e] = NPROJ == 2 ? __uint_as_float(uw[e]) : 0.f;
      }
      if (whole) {
        gemm_finish<NPROJ>(a, m, n0 + c, rs, g, u, vec);
      } else {
        // fp32 partial sums, 32 bytes a (token, 8 columns): lanes contiguous
        float4 *pg = reinterpret_cast<float4 *>(mine + (((size_t)h * (C::NCH / 8) + c / 8) * kBM + quarter * 32 + lane) * 8);
        __stcg(pg, make_float4(g[0], g[1], g[2], g[3]));
        __stcg(pg + 1, make_float4(g[4], g[5], g[6], g[7]));
        if (NPROJ == 2) {
          float4 *pu = reinterpret_cast<float4 *>(
              mine + (((size_t)h * (C::NCH / 8) + (kBN + c) / 8) * kBM + quarter * 32 + lane) * 8);
          __stcg(pu, make_float4(u[0], u[1], u[2], u[3]));
          __stcg(pu + 1, make_float4(u[4], u[5], u[6], u[7]));
        }
      }
    }
  }
  if (whole) return;
  // the tile's parts lie in CTAs c_lo .. c_hi; the one that brings the
  // counter to their number sums them and finishes the tile
  const long long t0u = (long long)tile * U;
  const int c_lo = (int)(((t0u + 1) * P + W - 1) / W - 1), c_hi = (int)(((t0u + U) * P + W - 1) / W - 1);
  named_barrier_sync(1, kDeqWarps * 32);
  if (tid == 0) {
    int last = 0;
    if (!*abort_s) {
      __threadfence();
      last = atomicAdd(&a.sk_cnt[tile], 1u) == (unsigned)(c_hi - c_lo) ? 1 : 0;
      if (last) {
        a.sk_cnt[tile] = 0;  // ready for the next launch
        __threadfence();
      }
    }
    *last_s = last;
  }
  named_barrier_sync(1, kDeqWarps * 32);
  if (!*last_s) return;
  for (int h = 0; h < mth; ++h) {
    const int m = m0 + h * kBM + quarter * 32 + lane;
    const float rs = (a.rs != nullptr && m < a.M) ? a.rs[m] : 1.f;
    for (int c = c0; c < c0 + 32; c += 8) {
      float g[8], u[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) g[e] = u[e] = 0.f;
      for (int cc = c_lo; cc <= c_hi; ++cc) {
        // CTA cc's part of this tile is its first (slot 0) unless the tile began inside its range
        const float *src = a.sk_part + ((size_t)cc * 2 + (t0u <= W * cc / P ? 0 : 1)) * SLOT;
        const float4 *pg =
            reinterpret_cast<const float4 *>(src + (((size_t)h * (C::NCH / 8) + c / 8) * kBM + quarter * 32 + lane) * 8);
        const float4 g0v = __ldcg(pg), g1v = __ldcg(pg + 1);
        g[0] += g0v.x; g[1] += g0v.y; g[2] += g0v.z; g[3] += g0v.w;
        g[4] += g1v.x; g[5] += g1v.y; g[6] += g1v.z; g[7] += g1v.w;
        if (NPROJ == 2) {
          const float4 *pu = reinterpret_cast<const float4 *>(
              src + (((size_t)h * (C::NCH / 8) + (kBN + c) / 8) * kBM + quarter * 32 + lane) * 8);
          const float4 u0v = __ldcg(pu), u1v = __ldcg(pu + 1);
          u[0] += u0v.x; u[1] += u0v.y; u[2] += u0v.z; u[3] += u0v.w;
          u[4] += u1v.x; u[5] += u1v.y; u[6] += u1v.z; u[7] += u1v.w;
        }
      }
      gemm_finish<NPROJ>(a, m, n0 + c, rs, g, u, vec);
    }
  }
}

template <int BITS, int NPROJ, int GROUP, bool EXACT>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_sk_kernel(const __grid_constant__ GemmArgs a,
                                                                   const __grid_constant__ GemmMaps tm) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  constexpr int SA = C::SA, SB = C::SB, R = C::R, GPB = C::GPB;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  GemmSmem<C> sm(smem_raw);
  uint8_t *smem = sm.base;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int KB = (a.K + 127) / 128;
  const int nlora = NPROJ == 2 && a.r > 0 ? (a.r + kLoraK - 1) / kLoraK : 0;
  const int U = KB + (nlora > 0 ? 1 : 0);
  const int MT = (a.M + a.mt * kBM - 1) / (a.mt * kBM), NT = (a.N + kBN - 1) / kBN;
  const long long W = (long long)MT * NT * U, P = gridDim.x;
  const long long g0 = W * blockIdx.x / P, g1 = W * (blockIdx.x + 1) / P;
  sm.init(tid, warp);
  const uint32_t tmem = *sm.tmem_s;

  auto wait = [&](uint64_t *bar, uint32_t parity) -> bool {
    if (*sm.abort_s) return false;
    if (mbar_wait_sleep(bar, parity)) return true;
    *sm.abort_s = 1;
    if (lane == 0) gemm_timeout();
    return false;
  };
  // The parts of tiles in this CTA's range, in order: tile, units [ub, ue),
  // weight blocks wb, stages nit (two a block, then the LoRA stages); token
  // tiles vary fastest, so neighbouring CTAs share row tiles.
#define WQ_FOR_EACH_PART                                                         \
  for (long long g_ = g0; g_ < g1;)                                              \
    for (int tile = (int)(g_ / U), ub = (int)(g_ - (long long)tile * U),         \
             ue = (int)min((long long)U, ub + (g1 - g_)), wb = min(ue, KB) - ub, \
             nit = 2 * wb + (ue > KB ? nlora : 0), once_ = (g_ += ue - ub, 1);   \
         once_; once_ = 0)
  auto tile_m0 = [&](int tile) { return (tile % MT) * a.mt * kBM; };
  auto halves = [&](int m0) { return min(a.mt, (a.M - m0 + kBM - 1) / kBM); };

  if (warp == kRawWarp) {
    if (lane == 0) {
      int gr = 0;  // blocks loaded so far
      bool ok = true;
      WQ_FOR_EACH_PART {
        (void)nit;  // the codes ring follows the blocks only
        const int n0 = (tile / MT) * kBN;
        for (int kb = ub; kb < ub + wb && ok; ++kb, ++gr) {
          const int q = gr % R;
          if (gr >= R && !wait(&sm.raw_empty[q], (gr / R - 1) & 1)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&sm.raw_full[q], (uint32_t)C::RAW);
          for (int p = 0; p < NPROJ; ++p) {
            uint8_t *dst = smem + C::OFF_RAW + q * C::RAW + p * C::RAWP;
            tma_load_3d(dst, &tm.codes[p], 0, kb * (C::BPK / 128), n0 / 16, &sm.raw_full[q]);
            tma_load_3d(dst + 8 * C::BPK, &tm.meta[p], 0, kb * GPB, n0 / 16, &sm.raw_full[q]);
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == kProducerWarp) {
    int gs = 0;  // stages so far
    bool ok = true;
    WQ_FOR_EACH_PART {
      const int m0 = tile_m0(tile), mth = halves(m0);
      for (int it = 0; it < nit && ok; ++it, ++gs) {
        const int s = gs % SA;
        if (gs >= SA && !wait(&sm.a_empty[s], (gs / SA - 1) & 1)) {
          ok = false;
          break;
        }
        uint8_t *As = smem + C::OFF_A + s * C::AT;
        if (it < 2 * wb) {
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.a_full[s], (uint32_t)(mth * kTileBytes));
            for (int h = 0; h < mth; ++h)
              tma_load_2d(As + h * kTileBytes, &tm.act, (ub + (it >> 1)) * 128 + (it & 1) * 64, m0 + h * kBM,
                          &sm.a_full[s]);
          }
        } else {
          gemm_lora_a_stage<NPROJ>(a, As, m0, mth, it - 2 * wb, lane, &sm.a_full[s]);
        }
      }
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      int gs = 0;
      bool ok = true;
      WQ_FOR_EACH_PART {
        if (!ok) break;
        const int mth = halves(tile_m0(tile));
        for (int it = 0; it < nit; ++it, ++gs) {
          const int sa = gs % SA, sb = gs % SB;
          if (!wait(&sm.a_full[sa], (gs / SA) & 1) || !wait(&sm.b_full[sb], (gs / SB) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          gemm_issue_stage<NPROJ, EXACT>(tmem, smem_addr(smem + C::OFF_A + sa * C::AT),
                                         smem_addr(smem + C::OFF_B + sb * C::BT), mth, it < 2 * wb, it == 0);
          umma_commit(&sm.a_empty[sa]);
          umma_commit(&sm.b_empty[sb]);
        }
        if (ok) umma_commit(sm.acc_full);  // the part's accumulators are complete
      }
    }
    __syncwarp();
  } else {
    // dequantization, then each part's epilogue; a warp that met a timeout
    // skips its work but still passes the epilogue's named barriers
    int gs = 0, gr = 0, part = 0;
    bool ok = true;
    WQ_FOR_EACH_PART {
      const int n0 = (tile / MT) * kBN;
      for (int it = 0; it < nit; ++it, ++gs) {
        const int s = gs % SB, hb = it & 1, kr = gr + (it >> 1), q = kr % R;
        const bool wstage = it < 2 * wb;
        if (ok && wstage && !wait(&sm.raw_full[q], (kr / R) & 1)) ok = false;
        if (ok && gs >= SB && !wait(&sm.b_empty[s], (gs / SB - 1) & 1)) ok = false;
        if (!ok) continue;
        uint8_t *Bs = smem + C::OFF_B + s * C::BT;
        if (wstage)
          gemm_deq_stage<BITS, NPROJ, GROUP, EXACT>(smem + C::OFF_RAW + q * C::RAW, Bs, hb, tid);
        else
          gemm_lora_b_stage<NPROJ>(a, Bs, n0, it - 2 * wb, tid);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&sm.b_full[s]);
          if (wstage && hb == 1) mbar_arrive(&sm.raw_empty[q]);  // both halves of this block's codes are read
        }
      }
      gr += wb;
      const bool have = ok && wait(sm.acc_full, part & 1);
      ++part;
      tc_fence_after();
      gemm_part_epilogue<BITS, NPROJ, GROUP, EXACT>(a, tmem, tile, ub, ue, U, W, P, g0, have, sm.abort_s, sm.last_s);
      // the next part's MMAs overwrite the accumulators only after this warp's
      // b_full arrival, which follows its TMEM reads
      tc_fence_before();
    }
  }
#undef WQ_FOR_EACH_PART

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, C::NCOLS);
}

// Per token of x [M, K] (bf16, K a multiple of 32): the binary16 copy x16
// [M][lda16] (the GEMM's A operand, zeros past K), the RMSNorm scale
// rs = 1/sqrt(mean(x^2) + eps) and, with an adapter, ta = lora_scale * x A^T
// as binary16 [M][2r] (gate rows, then up rows).
// A CTA takes 16 tokens and 16 rows of A.  The products x A^T run on m16n8k16
// bf16 MMAs (exact products, fp32 sums); the 16 warps take interleaved chunks
// of 32 features, two chunks' loads in flight at a time, and their partial
// sums are added in warp order.  A lane loads 8 consecutive features of a row
// (16 bytes) and feeds features 0..3 and 4..7 of them to two k-steps in the
// slots of k 2t, 2t+1, 2t+8, 2t+9: the same permutation of k for x and A, so
// the sums are unchanged.  Every CTA sums x^2 of its tokens (row block 0
// writes rs) and converts the chunks c with c % gridDim.y == blockIdx.y.
constexpr int kPrepTok = 16, kPrepRows = 16, kPrepWarps = 16, kPrepUnroll = 2;

__global__ void __launch_bounds__(kPrepWarps * 32) gemm_prep_kernel(const __nv_bfloat16 *x, int M, int K, int lda16,
                                                                   const __nv_bfloat16 *lora_a, int r2,
                                                                   float lora_scale, int prenorm, uint16_t *x16,
                                                                   float *rs, uint16_t *ta) {
  __shared__ float part[kPrepWarps][kPrepTok][kPrepRows + 1];
  __shared__ float ssp[kPrepWarps][kPrepTok];
  __shared__ uint32_t mxp[kPrepWarps][kPrepTok];
  __shared__ float scl[kPrepTok];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, g = lane >> 2, t = lane & 3;
  const int m0 = blockIdx.x * kPrepTok, j0 = blockIdx.y * kPrepRows;
  const int nchunk = K / 32;
  const bool lora = r2 > 0;
  float acc[2][4];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i >> 2][i & 3] = 0.f;
  float ss[2] = {0.f, 0.f};  // tokens g and g + 8 of the block
  uint32_t mx[2] = {0u, 0u};  // their largest |x| (bit patterns of non-negative floats order like the values)
  const auto word = [](const uint4 &v, int q) { return q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w; };
  for (int cb = warp; cb < nchunk; cb += kPrepWarps * kPrepUnroll) {
    uint4 xa[kPrepUnroll][2], ab[kPrepUnroll][2];
#pragma unroll
    for (int u = 0; u < kPrepUnroll; ++u) {  // the loads of both chunks first
      const int c = cb + u * kPrepWarps, k = c * 32 + 8 * t;
      const bool in = c < nchunk;
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int m = m0 + g + 8 * i;
        xa[u][i] = in && m < M ? __ldg(reinterpret_cast<const uint4 *>(x + (size_t)m * K + k))
                               : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int n = 0; n < 2; ++n) {
        const int j = j0 + 8 * n + g;
        ab[u][n] = in && lora && j < r2 ? __ldg(reinterpret_cast<const uint4 *>(lora_a + (size_t)j * K + k))
                                        : make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int u = 0; u < kPrepUnroll; ++u) {
      const int c = cb + u * kPrepWarps;
      if (c >= nchunk) break;  // the same for the whole warp
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const uint32_t w[4] = {xa[u][i].x, xa[u][i].y, xa[u][i].z, xa[u][i].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float lo = __uint_as_float(w[e] << 16), hi = __uint_as_float(w[e] & 0xffff0000u);
          ss[i] = fmaf(lo, lo, ss[i]);
          ss[i] = fmaf(hi, hi, ss[i]);
          mx[i] = max(mx[i], max((w[e] << 16) & 0x7fffffffu, w[e] & 0x7fff0000u));
        }
      }
      if (lora) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          // rows g, g + 8 of the m-tile are tokens g (xa[u][0]) and g + 8 (xa[u][1])
          const uint32_t af[4] = {word(xa[u][0], 2 * h), word(xa[u][1], 2 * h), word(xa[u][0], 2 * h + 1),
                                  word(xa[u][1], 2 * h + 1)};
#pragma unroll
          for (int nt = 0; nt < 2; ++nt)
            mma_bf16_16816(acc[nt], af, word(ab[u][nt], 2 * h), word(ab[u][nt], 2 * h + 1));
        }
      }
    }
  }
  // sums of squares: the quad's lanes hold disjoint features of the same tokens
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    ss[i] += __shfl_xor_sync(0xffffffffu, ss[i], 1);
    ss[i] += __shfl_xor_sync(0xffffffffu, ss[i], 2);
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    mx[i] = max(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
    mx[i] = max(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
  }
  if (t == 0) {
    ssp[warp][g] = ss[0];
    ssp[warp][g + 8] = ss[1];
    mxp[warp][g] = mx[0];
    mxp[warp][g + 8] = mx[1];
  }
  if (lora) {
    // accumulator (row, col) of n-tile nt: rows g / g + 8, cols 2t, 2t+1
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      part[warp][g][8 * nt + 2 * t] = acc[nt][0];
      part[warp][g][8 * nt + 2 * t + 1] = acc[nt][1];
      part[warp][g + 8][8 * nt + 2 * t] = acc[nt][2];
      part[warp][g + 8][8 * nt + 2 * t + 1] = acc[nt][3];
    }
  }
  __syncthreads();
  // Per token an exact power of two 2^e puts its largest |x| in [2^4, 2^5):
  // the binary16 copies of x and of t = lora_scale x A^T are taken of the
  // values times 2^e (no overflow: 2^11 below the binary16 maximum even for
  // |t| up to 2^10 |x|; every element within 2^-22 of the largest stays
  // exact), and the epilogue multiplies the fp32 sums by rs 2^-e, which
  // undoes it exactly.
  if (tid < kPrepTok) {
    uint32_t mxb = 0u;
    for (int w = 0; w < kPrepWarps; ++w) mxb = max(mxb, mxp[w][tid]);
    const int be = (int)(mxb >> 23);
    const int e = mxb == 0u || be >= 255 ? 0 : max(-100, min(100, 131 - be));
    scl[tid] = __int_as_float((e + 127) << 23);
    if (blockIdx.y == 0 && m0 + tid < M) {
      float tot = 0.f;
      for (int w = 0; w < kPrepWarps; ++w) tot += ssp[w][tid];
      const float r = prenorm ? __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(tot, (float)K), kRmsEps))) : 1.f;
      rs[m0 + tid] = r * __int_as_float((127 - e) << 23);
    }
  }
  __syncthreads();
  // the binary16 copy of x (2^e x): this CTA's chunks c = blockIdx.y + cc
  // gridDim.y, 16 bytes an item, four loads in flight a thread
  {
    const int ncc = (nchunk - (int)blockIdx.y + (int)gridDim.y - 1) / (int)gridDim.y;
    const int items = kPrepTok * ncc * 4;
    constexpr int NT = kPrepWarps * 32;
    for (int i0 = tid; i0 < items; i0 += 4 * NT) {
      uint4 v[4];
      int tl[4];
      size_t dst[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * NT;
        tl[u] = i / (ncc * 4);
        const int rem = i % (ncc * 4), c = (int)blockIdx.y + (rem / 4) * (int)gridDim.y, k = c * 32 + 8 * (rem % 4);
        const int m = m0 + tl[u];
        const bool ok = i < items && m < M;
        dst[u] = ok ? (size_t)m * lda16 + k : ~(size_t)0;
        v[u] = ok ? __ldg(reinterpret_cast<const uint4 *>(x + (size_t)m * K + k)) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (dst[u] == ~(size_t)0) continue;
        const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
        const float sc = scl[tl[u]];
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e)
          o[e] = h2bits(__floats2half2_rn(__uint_as_float(w[e] << 16) * sc, __uint_as_float(w[e] & 0xffff0000u) * sc));
        *reinterpret_cast<uint4 *>(x16 + dst[u]) = make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
  }
  if (lora) {
    for (int o = tid; o < kPrepTok * kPrepRows; o += kPrepWarps * 32) {
      const int tl = o / kPrepRows, jl = o % kPrepRows;
      const int m = m0 + tl, j = j0 + jl;
      if (m >= M || j >= r2) continue;
      float v = 0.f;
      for (int w = 0; w < kPrepWarps; ++w) v += part[w][tl][jl];
      ta[(size_t)m * r2 + j] = __half_as_ushort(__float2half_rn(lora_scale * v * scl[tl]));
    }
  }
  // zeros past K
  if (blockIdx.y == 0)
    for (int i = tid; i < kPrepTok * (lda16 - K); i += kPrepWarps * 32) {
      const int tl = i / (lda16 - K), k = K + i % (lda16 - K);
      if (m0 + tl < M) x16[(size_t)(m0 + tl) * lda16 + k] = 0;
    }
}

// bf16 [M, K] -> binary16 [M, lda16] (zero padded), the down GEMM's A
// operand, one CTA per token: an exact power of two 2^e puts the token's
// largest |x| in [2^4, 2^5) (no overflow, every element within 2^-22 of the
// largest exact); sx[m] = 2^-e, by which the epilogue multiplies the sums.
// K a multiple of 8.
__global__ void __launch_bounds__(256) to_f16_kernel(const __nv_bfloat16 *x, int M, int K, int lda16, uint16_t *x16,
                                                     float *sx) {
  __shared__ uint32_t wmax[8];
  const int m = blockIdx.x, tid = threadIdx.x;
  if (m >= M) return;
  const uint4 *row = reinterpret_cast<const uint4 *>(x + (size_t)m * K);
  const int n8 = K / 8;
  uint32_t mx = 0u;
  for (int i = tid; i < n8; i += blockDim.x) {
    const uint4 v = __ldg(row + i);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) mx = max(mx, max((w[e] << 16) & 0x7fffffffu, w[e] & 0x7fff0000u));
  }
  mx = __reduce_max_sync(0xffffffffu, mx);
  if ((tid & 31) == 0) wmax[tid >> 5] = mx;
  __syncthreads();
  mx = 0u;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) mx = max(mx, wmax[w]);
  const int be = (int)(mx >> 23);
  const int e = mx == 0u || be >= 255 ? 0 : max(-100, min(100, 131 - be));
  const float sc = __int_as_float((e + 127) << 23);
  if (tid == 0) sx[m] = __int_as_float((127 - e) << 23);
  for (int i = tid; i < n8; i += blockDim.x) {
    const uint4 v = __ldg(row + i);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q)
      o[q] = h2bits(__floats2half2_rn(__uint_as_float(w[q] << 16) * sc, __uint_as_float(w[q] & 0xffff0000u) * sc));
    *reinterpret_cast<uint4 *>(x16 + (size_t)m * lda16 + 8 * i) = make_uint4(o[0], o[1], o[2], o[3]);
  }
  for (int k = K + tid; k < lda16; k += blockDim.x) x16[(size_t)m * lda16 + k] = 0;
}

// ---------------------------------------------------------------------------
// Few tokens (M <= 64): the operands swapped.  The dequantized weight tile is
// the MMA's A operand (M = 128 rows, the K-major no-swizzle layout the
// dequantizing warps already write) and the activation tile its B operand
// (N = NT tokens, NT = M rounded up to 16; one TMA box of 64 features x NT
// tokens a stage, 128-byte swizzled), so the tensor cores spend no work on
// padding tokens: with 128-token tiles a 16-token call did 8x the MMA work it
// needs.  TMEM holds D[row][token]: lane = output row, column = token (gate in
// columns 0..NT-1, up in NT..2NT-1).  The feature blocks are split KS ways
// (grid.y) when there are fewer row tiles than SMs: each split writes its fp32
// partial sums to the workspace and the split that brings the row tile's
// arrival counter to KS adds them in split order and finishes the tile
// (deterministic; the counter is left at zero).  The LoRA stages run in split
// 0.
// ---------------------------------------------------------------------------
constexpr int kSwapMaxTok = 64;

template <int BITS, int NPROJ, int GROUP, bool EXACT>
struct SwapCfg {
  using G = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  static constexpr int BPK = G::BPK, GPB = G::GPB, RAWP = G::RAWP, RAW = G::RAW, BT = G::BT;
  static constexpr int AT = kSwapMaxTok * 128;  // an activation stage: up to 64 token rows of 128 bytes
  static constexpr int AVAIL = (int)kGemmSmemLimit - 2048;
  static constexpr int SB = (AVAIL - 3 * BT - 3 * RAW) / AT >= 4 ? 3 : 2;
  static constexpr int SA = std::min(8, (AVAIL - SB * BT - 3 * RAW) / AT);
  static constexpr int R = std::min(6, (AVAIL - SA * AT - SB * BT) / RAW);
  static_assert(SA >= 2 && R >= 2, "swapped GEMM pipeline does not fit");
  static constexpr int OFF_A = 0;
  static constexpr int OFF_B = SA * AT;
  static constexpr int OFF_RAW = OFF_B + SB * BT;
  static constexpr int OFF_BAR = OFF_RAW + R * RAW;
  static constexpr int SMEM = OFF_BAR + (2 * SA + 2 * SB + 2 * R + 2) * 8 + 16 + 1024;
  static constexpr int NCOLS = 128;  // NPROJ x NT fp32 columns, NT <= 64
  static_assert(SMEM <= (int)kGemmSmemLimit, "swapped GEMM stage does not fit");
};

// LoRA stage l, token side: lora_scale * t of tokens 0 .. NT-1 (rank columns
// 32 l .. 32 l + 31 of gate, then of up), zeros past M and r; lane 0 arrives
// on `full` once all landed.
template <int NPROJ>
__device__ __forceinline__ void swap_lora_t_stage(const GemmArgs &a, uint8_t *As, int NT, int l, int lane,
                                                  uint64_t *full) {
  for (int i = lane; i < NPROJ * NT * 4; i += 32) {
    const int p = i / (NT * 4), rem = i - p * NT * 4;
    const int ml = rem >> 2, c = rem & 3;
    const int col = l * kLoraK + c * 8;
    const bool in = ml < a.M && col < a.r;
    const uint16_t *src = in ? a.ta + (size_t)ml * 2 * a.r + p * a.r + col : a.ta;
    cp_async16_zfill(As + p * (NT * kLoraK * 2) + kmajor_off(ml, c * 8, 4 * 128u), src, in ? 16u : 0u);
  }
  cp_async_wait_all();
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) mbar_arrive(full);
}

// The MMAs of one stage (one thread): per projection, D[p] (+)= W_p x^T over
// the stage's 4 k-steps (EXACT: the low parts of the weights as well).
template <int NPROJ, bool EXACT>
__device__ __forceinline__ void swap_issue_stage(uint32_t tmem, uint32_t as, uint32_t bs, int NT, bool wstage,
                                                 bool first) {
  const uint32_t idesc = umma_idesc_f16(128, NT);
  if (wstage) {
#pragma unroll
    for (int p = 0; p < NPROJ; ++p)
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        const uint64_t xdesc = umma_desc_kmajor_sw128(as + ks * 32, 1024);
        umma_f16(tmem + p * NT, umma_desc_kmajor(bs + p * kTileBytes + ks * 256, 128, kSboTile), xdesc, idesc,
                 (first && ks == 0) ? 0u : 1u);
        if (EXACT)  // the low parts of the same weights
          umma_f16(tmem + p * NT, umma_desc_kmajor(bs + (NPROJ + p) * kTileBytes + ks * 256, 128, kSboTile), xdesc,
                   idesc, 1u);
      }
  } else {
    constexpr uint32_t sbo = 4 * 128u;  // 32 rank columns a LoRA stage
    for (int p = 0; p < NPROJ; ++p)
      for (int ks = 0; ks < kLoraK / 16; ++ks)
        umma_f16(tmem + p * NT, umma_desc_kmajor(bs + p * (kBN * kLoraK * 2) + ks * 256, 128, sbo),
                 umma_desc_kmajor(as + p * (NT * kLoraK * 2) + ks * 256, 128, sbo), idesc,
                 (first && ks == 0) ? 0u : 1u);
  }
}

// Output row n for tokens mb .. mb + 7 from the fp32 sums g (and u):
// h = SiLU(rs g) * (rs u), or y = rs g + residual (bf16 or fp32); the lanes
// of a warp hold consecutive rows, so each token's stores are contiguous.
template <int NPROJ>
__device__ __forceinline__ void swap_finish(const GemmArgs &a, int n, int mb, const float (&g)[8],
                                            const float (&u)[8]) {
  if (n >= a.N) return;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int m = mb + e;
    if (m >= a.M) break;
    const float rs = a.rs != nullptr ? a.rs[m] : 1.f;
    const size_t o = (size_t)m * a.N + n;
    if (NPROJ == 2) {
      const float gv = rs * g[e], uv = rs * u[e];
      reinterpret_cast<__nv_bfloat16 *>(a.out)[o] = __float2bfloat16_rn(__fdividef(gv, 1.f + __expf(-gv)) * uv);
    } else {
      float v = rs * g[e];
      if (a.residual) v += __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(a.residual)[o]);
      if (a.out_f32)
        reinterpret_cast<float *>(a.out)[o] = v;
      else
        reinterpret_cast<__nv_bfloat16 *>(a.out)[o] = __float2bfloat16_rn(v);
    }
  }
}

template <int BITS, int NPROJ, int GROUP, bool EXACT>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_swap_kernel(const GemmArgs a, const __grid_constant__ GemmMaps tm,
                                                                     int NT, int KS) {
  using C = SwapCfg<BITS, NPROJ, GROUP, EXACT>;
  constexpr int SA = C::SA, SB = C::SB, R = C::R, GPB = C::GPB;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  GemmSmem<C> sm(smem_raw);
  uint8_t *smem = sm.base;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x, n0 = tile * kBN, ks = blockIdx.y;
  const int KB = (a.K + 127) / 128;
  const int kb0 = (int)((long long)KB * ks / KS), kb1 = (int)((long long)KB * (ks + 1) / KS);
  const int nws = 2 * (kb1 - kb0);  // weight stages (64 features each)
  const int nlora = NPROJ == 2 && a.r > 0 && ks == 0 ? (a.r + kLoraK - 1) / kLoraK : 0;
  const int nit = nws + nlora;
  sm.init(tid, warp);
  const uint32_t tmem = *sm.tmem_s;

  auto wait = [&](uint64_t *bar, uint32_t parity) -> bool {
    if (*sm.abort_s) return false;
    if (mbar_wait_sleep(bar, parity)) return true;
    *sm.abort_s = 1;
    if (lane == 0) gemm_timeout();
    return false;
  };

  if (warp == kRawWarp) {
    if (lane == 0)
      for (int it = 0; it < kb1 - kb0; ++it) {
        const int q = it % R;
        if (it >= R && !wait(&sm.raw_empty[q], (it / R - 1) & 1)) break;
        mbar_arrive_expect_tx(&sm.raw_full[q], (uint32_t)C::RAW);
        for (int p = 0; p < NPROJ; ++p) {
          uint8_t *dst = smem + C::OFF_RAW + q * C::RAW + p * C::RAWP;
          tma_load_3d(dst, &tm.codes[p], 0, (kb0 + it) * (C::BPK / 128), n0 / 16, &sm.raw_full[q]);
          tma_load_3d(dst + 8 * C::BPK, &tm.meta[p], 0, (kb0 + it) * GPB, n0 / 16, &sm.raw_full[q]);
        }
      }
    __syncwarp();
  } else if (warp == kProducerWarp) {
    for (int it = 0; it < nit; ++it) {
      const int s = it % SA;
      if (it >= SA && !wait(&sm.a_empty[s], (it / SA - 1) & 1)) break;
      uint8_t *As = smem + C::OFF_A + s * C::AT;
      if (it < nws) {
        if (lane == 0) {
          // one box of 64 features x NT tokens, a 128-byte swizzled row per token
          mbar_arrive_expect_tx(&sm.a_full[s], (uint32_t)(NT * 128));
          tma_load_2d(As, &tm.act, (2 * kb0 + it) * 64, 0, &sm.a_full[s]);
        }
      } else {
        swap_lora_t_stage<NPROJ>(a, As, NT, it - nws, lane, &sm.a_full[s]);
      }
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      for (int it = 0; it < nit; ++it) {
        const int sa = it % SA, sb = it % SB;
        if (!wait(&sm.a_full[sa], (it / SA) & 1) || !wait(&sm.b_full[sb], (it / SB) & 1)) break;
        tc_fence_after();
        swap_issue_stage<NPROJ, EXACT>(tmem, smem_addr(smem + C::OFF_A + sa * C::AT),
                                       smem_addr(smem + C::OFF_B + sb * C::BT), NT, it < nws, it == 0);
        umma_commit(&sm.a_empty[sa]);
        umma_commit(&sm.b_empty[sb]);
      }
      umma_commit(sm.acc_full);
    }
    __syncwarp();
  } else {
    // ---- dequantization into the weight tiles ----
    for (int it = 0; it < nit; ++it) {
      const int s = it % SB, lb = it >> 1, hb = it & 1, q = lb % R;
      if (it < nws && !wait(&sm.raw_full[q], (lb / R) & 1)) break;
      if (it >= SB && !wait(&sm.b_empty[s], (it / SB - 1) & 1)) break;
      uint8_t *Bs = smem + C::OFF_B + s * C::BT;
      if (it < nws)
        gemm_deq_stage<BITS, NPROJ, GROUP, EXACT>(smem + C::OFF_RAW + q * C::RAW, Bs, hb, tid);
      else
        gemm_lora_b_stage<NPROJ>(a, Bs, n0, it - nws, tid);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&sm.b_full[s]);
        if (it < nws && hb == 1) mbar_arrive(&sm.raw_empty[q]);
      }
    }

    // ---- epilogue: warp w reads TMEM lanes 32 (w % 4) .. (the rows) and the
    // token groups of 8 columns w / 4, w / 4 + 4, .. ----
    const bool ok = wait(sm.acc_full, 0);
    tc_fence_after();
    const int quarter = warp & 3, rl = quarter * 32 + lane, n = n0 + rl;
    constexpr int SLOT = NPROJ * kBN * kSwapMaxTok;  // floats of a split's partial tile: [p][128 rows][NT]
    float *mine = KS > 1 && a.sk_part ? a.sk_part + ((size_t)tile * KS + ks) * SLOT : nullptr;
    for (int tg = warp >> 2; tg * 8 < NT; tg += 4) {
      uint32_t gw[8], uw[8];
      const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16) + tg * 8;
      tmem_ld8(tl, gw);
      if (NPROJ == 2) tmem_ld8(tl + NT, uw);
      tmem_ld_wait();
      if (!ok) continue;
      float g[8], u[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        g[e] = __uint_as_float(gw[e]);
        u[e] = NPROJ == 2 ? __uint_as_float(uw[e]) : 0.f;
      }
      if (mine == nullptr) {
        swap_finish<NPROJ>(a, n, tg * 8, g, u);
      } else {
#pragma unroll
        for (int p = 0; p < NPROJ; ++p) {
          float4 *dst = reinterpret_cast<float4 *>(mine + ((size_t)p * kBN + rl) * kSwapMaxTok + tg * 8);
          const float *v = p == 0 ? g : u;
          __stcg(dst, make_float4(v[0], v[1], v[2], v[3]));
          __stcg(dst + 1, make_float4(v[4], v[5], v[6], v[7]));
        }
      }
    }
    if (mine != nullptr) {
      named_barrier_sync(1, kDeqWarps * 32);
      if (tid == 0) {
        int last = 0;
        if (ok && !*sm.abort_s) {
          __threadfence();
          last = atomicAdd(&a.sk_cnt[tile], 1u) == (unsigned)(KS - 1) ? 1 : 0;
          if (last) {
            a.sk_cnt[tile] = 0;  // ready for the next launch
            __threadfence();
          }
        }
        *sm.last_s = last;
      }
      named_barrier_sync(1, kDeqWarps * 32);
      if (*sm.last_s) {
        for (int tg = warp >> 2; tg * 8 < NT; tg += 4) {
          float g[8], u[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) g[e] = u[e] = 0.f;
          for (int k2 = 0; k2 < KS; ++k2) {  // the splits in order
            const float *src = a.sk_part + ((size_t)tile * KS + k2) * SLOT;
#pragma unroll
            for (int p = 0; p < NPROJ; ++p) {
              const float4 *pv = reinterpret_cast<const float4 *>(src + ((size_t)p * kBN + rl) * kSwapMaxTok + tg * 8);
              const float4 v0 = __ldcg(pv), v1 = __ldcg(pv + 1);
              float *d = p == 0 ? g : u;
              d[0] += v0.x; d[1] += v0.y; d[2] += v0.z; d[3] += v0.w;
              d[4] += v1.x; d[5] += v1.y; d[6] += v1.z; d[7] += v1.w;
            }
          }
          swap_finish<NPROJ>(a, n, tg * 8, g, u);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, C::NCOLS);
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
cudaError_t make_maps(const GemmArgs &a, int nproj, int bits, GemmMaps *m, int box_rows = kBM) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint32_t e1[3] = {1, 1, 1};
  {
    const cuuint64_t dims[2] = {(cuuint64_t)a.K, (cuuint64_t)a.M};
    const cuuint64_t strides[1] = {(cuuint64_t)a.lda * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    if (fn(&m->act, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<uint16_t *>(a.act), dims, strides, box, e1,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
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

cudaError_t num_sms_cached(int *sms) {
  static int cached[64] = {0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (cached[dev] == 0 && (e = cudaDeviceGetAttribute(&cached[dev], cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return e;
  *sms = cached[dev];
  return cudaSuccess;
}

// Work split of a launch.  A CTA takes two token halves (each weight
// dequantized once for 256 tokens) whenever there are more than 128 tokens.
// Tiles are mt * 128 tokens x 128 rows, U work units each (128-feature
// blocks, plus one for the LoRA stages).  Stream-K -- P CTAs (one per SM at
// most, 4 units each at least) dividing the T * U units evenly -- when it
// shortens the critical path by more than its own cost, which was measured at
// about 40 units (the split tiles' partial sums and fixups, and a slower main
// loop); one CTA per tile otherwise.
constexpr long long kStreamKCost = 40;  // work units

struct GemmSched {
  int mt, T, U, P;
  bool sk;
};
GemmSched gemm_schedule(int M, int N, int K, int nproj, int r, int sms) {
  GemmSched g;
  g.mt = M > kBM ? 2 : 1;
  g.T = (M + g.mt * kBM - 1) / (g.mt * kBM) * ((N + kBN - 1) / kBN);
  g.U = (K + 127) / 128 + (nproj == 2 && r > 0 ? 1 : 0);
  const long long W = (long long)g.T * g.U;
  const long long waves = (g.T + sms - 1) / sms, P = std::max(1LL, std::min((long long)sms, W / 4));
  g.sk = W >= 8 && waves * g.U > (W + P - 1) / P + kStreamKCost;
  g.P = g.sk ? (int)P : g.T;
  return g;
}

// The swapped-operand launch for few tokens: NT = M rounded up to 16; the
// feature blocks split KS ways when the row tiles alone leave SMs idle (each
// split at least 2 blocks).
struct SwapSched {
  int NT, KS, tiles;
};
SwapSched swap_schedule(int M, int N, int K, int sms) {
  SwapSched w;
  w.NT = (std::min(M, kSwapMaxTok) + 15) / 16 * 16;
  w.tiles = (N + kBN - 1) / kBN;
  const int KB = (K + 127) / 128;
  w.KS = std::max(1, std::min(sms / std::max(1, w.tiles), KB / 2));
  return w;
}

template <int BITS, int NPROJ, int GROUP, bool EXACT>
cudaError_t launch_gemm_t(const GemmArgs &a, cudaStream_t s) {
  using C = GemmCfg<BITS, NPROJ, GROUP, EXACT>;
  if (a.M <= kSwapMaxTok) {
    using SC = SwapCfg<BITS, NPROJ, GROUP, EXACT>;
    auto kern = qgemm_swap_kernel<BITS, NPROJ, GROUP, EXACT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SC::SMEM);
    if (e != cudaSuccess) return e;
    int sms = 0;
    if ((e = num_sms_cached(&sms)) != cudaSuccess) return e;
    SwapSched w = swap_schedule(a.M, a.N, a.K, sms);
    if (!(a.sk_part && a.sk_cnt)) w.KS = 1;
    GemmMaps maps;
    if ((e = make_maps(a, NPROJ, BITS, &maps, w.NT)) != cudaSuccess) return e;
    kern<<<dim3(w.tiles, w.KS), kGemmThreads, SC::SMEM, s>>>(a, maps, w.NT, w.KS);
    return cudaGetLastError();
  }
  auto tile_kern = qgemm_tile_kernel<BITS, NPROJ, GROUP, EXACT>;
  auto sk_kern = qgemm_sk_kernel<BITS, NPROJ, GROUP, EXACT>;
  cudaError_t e = cudaFuncSetAttribute(tile_kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(sk_kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  GemmMaps maps;
  if ((e = make_maps(a, NPROJ, BITS, &maps)) != cudaSuccess) return e;
  int sms = 0;
  if ((e = num_sms_cached(&sms)) != cudaSuccess) return e;
  const GemmSched g = gemm_schedule(a.M, a.N, a.K, NPROJ, a.r, sms);
  GemmArgs ka = a;
  ka.mt = g.mt;
  if (g.sk && a.sk_part && a.sk_cnt) {
    sk_kern<<<g.P, kGemmThreads, C::SMEM, s>>>(ka, maps);
  } else {
    ka.sk_part = nullptr;
    ka.sk_cnt = nullptr;
    tile_kern<<<dim3((a.M + g.mt * kBM - 1) / (g.mt * kBM), (a.N + kBN - 1) / kBN), kGemmThreads, C::SMEM, s>>>(ka, maps);
  }
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

size_t gemm_scratch_floats(int M, int N, int K, int nproj, int num_sms) {
  if (M <= 0 || N <= 0 || K <= 0 || num_sms <= 0) return 0;
  const GemmSched g = gemm_schedule(M, N, K, nproj, kMaxRank, num_sms);
  const size_t sk = g.sk ? (size_t)2 * g.P * kHalves * kBM * nproj * kBN : 0;
  // the swapped-operand launch of any token count up to this one (a
  // workspace serves every smaller call too)
  const SwapSched w = swap_schedule(M, N, K, num_sms);
  const size_t sw = w.KS > 1 ? (size_t)w.tiles * w.KS * nproj * kBN * kSwapMaxTok : 0;
  return std::max(sk, sw);
}

size_t gemm_counters(int M, int N) { return (size_t)((M + kBM - 1) / kBM) * ((N + kBN - 1) / kBN); }

cudaError_t launch_gemm_prep(const void *x, int M, int K, int lda16, const void *lora_a, int r2, float lora_scale,
                             int prenorm, uint16_t *x16, float *rs, uint16_t *ta, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (K % 32 != 0 || lda16 < K) return cudaErrorInvalidValue;
  const dim3 grid((M + kPrepTok - 1) / kPrepTok, r2 > 0 ? (r2 + kPrepRows - 1) / kPrepRows : 1);
  gemm_prep_kernel<<<grid, kPrepWarps * 32, 0, s>>>(
      reinterpret_cast<const __nv_bfloat16 *>(x), M, K, lda16, reinterpret_cast<const __nv_bfloat16 *>(lora_a), r2,
      lora_scale, prenorm, x16, rs, ta);
  return cudaGetLastError();
}
cudaError_t launch_to_f16(const void *x, int M, int K, int lda16, uint16_t *x16, float *sx, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (K % 8 != 0 || lda16 < K) return cudaErrorInvalidValue;
  to_f16_kernel<<<M, 256, 0, s>>>(reinterpret_cast<const __nv_bfloat16 *>(x), M, K, lda16, x16, sx);
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
    case 0: return GemmCfg<2, 2, 32, false>::SA;
    case 1: return GemmCfg<2, 2, 64, false>::SA;
    case 2: return GemmCfg<2, 2, 128, false>::SA;
    case 3: return GemmCfg<4, 2, 32, false>::SA;
    case 4: return GemmCfg<4, 2, 64, false>::SA;
    case 5: return GemmCfg<4, 2, 128, false>::SA;
    case 6: return GemmCfg<4, 1, 32, false>::SA;
    case 7: return GemmCfg<4, 1, 64, false>::SA;
    default: return GemmCfg<4, 1, 128, false>::SA;
  }
}

}  // namespace wq
