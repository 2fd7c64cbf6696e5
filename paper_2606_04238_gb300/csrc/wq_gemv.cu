// wq_gemv.cu -- decode-regime dequant-GEMV kernels (sm_103a).
//
// One templated kernel serves the three matrix products of the gated MLP
// with W4/W2-GateUp weights (Sec. 3.3):
//   * gate+up, 2-bit codes, unmerged LoRA (Eq. 1) and SiLU(gate)*up fused
//     into the epilogue, so the intermediate g/u never leave the chip
//     (Sec. 5 models the MLP operators as one fused kernel);
//   * gate+up, 4-bit codes (the uniform-W4 comparator);
//   * down, 4-bit codes, residual add fused into the epilogue, optionally
//     followed by the next layer's per-tile RMSNorm / LoRA-A partial sums.
//
// The decode step is a chain of these launches joined by programmatic
// dependent launch.  Everything a launch can do before its input exists is
// done before griddepcontrol.wait, so that it overlaps the previous launch:
//   1. each warp's lane 0 bulk-copies (TMA) the packed codes and binary16
//      scales/zeros of the warp's slice into shared memory; LoRA-B rows and
//      the next layer's LoRA-A columns are staged with plain loads;
//   2. after the wait, every input of the previous launch is requested in one
//      round trip: the activation panel (converted to binary16, one
//      128-feature block per warp item, with an exact power-of-two scale per
//      (block, token) and per code position class, below), the tile partials
//      of the input (sum x^2 and A x per 16 features, added up for the
//      epilogue) and the residual rows;
//   3. each warp owns one or two 16-row tiles and a share of the panel: a
//      16-byte shared load per lane yields the tensor-core A fragments of 64
//      (2-bit) or 32 (4-bit) codes; codes are isolated with a single AND each
//      -- the isolated bits read as a binary16 subnormal code * 4^c * 2^-24,
//      the 4^c (c = bit-position class) being cancelled by the activation's
//      class scale -- and fed to mma.sync m16n8k16 (fp32 accumulation);
//   4. per group: acc += s * sx * sum_k code*x (block scale sx); the
//      zero-point part -s * z * sum_k x of the affine dequantization s(q - z)
//      is added once per output row after the loop;
//   5. warps' partial sums are reduced in shared memory in a fixed order;
//      with several panels the last-arriving CTA of a row tile adds the
//      panel partials in panel order (deterministic), then the epilogue
//      (RMSNorm scale, LoRA-B expansion, SiLU(g)*u; or residual add and the
//      next layer's tile partials) stores the outputs.
#include <algorithm>
#include <climits>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>

#include "wq_internal.h"
#include "wq_ptx.cuh"

namespace wq {

// Device status word: WQ_OK (0) or WQ_ERR_TIMEOUT (-6) after a bounded wait ran out.
__device__ int g_device_status = 0;

// Debug builds only: first failed bounds/alignment check {site, line, value, count}.
__device__ long long g_debug_record[4] = {0, 0, 0, 0};

namespace {

__device__ __forceinline__ void record_timeout() { atomicExch(&g_device_status, -6); }

#ifdef WQ_DEBUG_CHECKS
__device__ __noinline__ void debug_fail(int site, int line, long long value) {
  if (atomicAdd(reinterpret_cast<unsigned long long *>(&g_debug_record[3]), 1ull) == 0ull) {
    g_debug_record[0] = site;
    g_debug_record[1] = line;
    g_debug_record[2] = value;
  }
}
// True when the access may proceed; records the first violation otherwise.
#define WQ_OK_IF(cond, site, value) ((cond) ? true : (debug_fail((site), __LINE__, (long long)(value)), false))
#else
#define WQ_OK_IF(cond, site, value) true
#endif
// [off, off + len) inside [0, size) and off aligned to `al`
#define WQ_RANGE(off, len, size, al) \
  ((long long)(off) >= 0 && (long long)(off) + (long long)(len) <= (long long)(size) && ((long long)(off) % (al)) == 0)

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

__device__ __forceinline__ void unpack_bf16x8(const uint4 v, float (&f)[8]) {
  f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
  f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
  f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
  f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

__device__ __forceinline__ uint32_t pack_half2(float a, float b) {
  const __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<const uint32_t *>(&h);
}

// 2^k for -126 <= k <= 127, built from the binary32 exponent field
__device__ __forceinline__ float exp2i(int k) { return __int_as_float((k + 127) << 23); }

// sum_{i < n} base[i * stride] from L2, added in index order, eight loads in
// flight at a time (the partial sums of split work).
__device__ __forceinline__ float sum_strided_cg(const float *base, size_t stride, int n) {
  float s = 0.f;
  for (int i0 = 0; i0 < n; i0 += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = i0 + u < n ? ldcg_f32(base + (size_t)(i0 + u) * stride) : 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (i0 + u < n) s += v[u];
  }
  return s;
}

// Scale exponent e of a block whose largest |x| has the bit pattern mxb:
// 2^e puts it in [2^14, 2^15).  mx = f 2^E with f in [0.5, 1) and E = (biased
// exponent) - 126, so e = 15 - E, clamped (subnormal mx: 100); 0 for a zero,
// infinite or nan mx.
__device__ __forceinline__ int block_exponent(uint32_t mxb) {
  const int be = (int)(mxb >> 23);
  return mxb == 0u || be >= 255 ? 0 : max(-100, min(100, 141 - be));
}

__device__ __forceinline__ float half_bits_to_float(uint32_t bits16) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(bits16 & 0xffffu)));
}

constexpr int kMaxThreads = 512;  // per CTA: up to 128 registers a thread

// ---------------------------------------------------------------------------
// The dequant-GEMV kernel.
//   BITS  2, 3 or 4 (code width; 3: two bit planes, below), NPROJ 2
//   (gate+up) or 1 (down),
//   GROUP 32/64/128 (quantization group), NT 1 or 2 (8-token MMA tiles per
//   token chunk: chunks of 8 tokens for m <= 8, of 16 otherwise), TPW 1 or 2
//   (row tiles per warp: with 2, each activation fragment feeds 2 tiles x
//   NPROJ projections).
// ---------------------------------------------------------------------------
template <int BITS, int NPROJ, int GROUP, int NT, int TPW>
__device__ __forceinline__ void qgemv_body(const GemvArgs &a, const GemvPlan &p) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int BPK = BITS == 2 ? 512 : BITS == 3 ? 768 : 1024;  // code bytes per (row tile, 128-feature block)
  constexpr int GPB = 128 / GROUP;             // groups per block
  constexpr int GS = GROUP / 16;               // k-steps (16 features) per group
  constexpr int TOK = 8 * NT;                  // tokens per chunk
  constexpr int LPG = GROUP / 4;               // conversion lanes per group (4 features a lane)
  // Down with one row tile per warp runs two accumulation chains, one per
  // 64-feature half of a block, and scales the activations per half
  // (HALF); the other kernels scale per 128-feature block.
  constexpr bool HALF = NPROJ * TPW < 2;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int rb = blockIdx.x / p.P, panel = blockIdx.x % p.P;
  const int rt0 = rb * p.RB;
  const int nrt = min(p.RB, p.RT - rt0);
  const int kb0 = panel * p.KP;
  const int nkb = min(p.KP, p.KB - kb0);
  const int NG = p.KB * GPB;
  const int M = a.M, MPAD = p.MPAD;
  const int r = a.r;
  const int Q = 1 + 2 * r;           // values per (tile, token) of the tile partials
  const int Qp = WQ_TP_STRIDE(r);     // their stride (zero padded)

  uint8_t *codes_s = smem + p.off_codes;
  uint8_t *meta_s = smem + p.off_meta;
  const __nv_bfloat16 *lorab_s = reinterpret_cast<const __nv_bfloat16 *>(smem + p.off_lorab);  // [NPROJ][RB*16][r]
  __nv_bfloat16 *an_s = reinterpret_cast<__nv_bfloat16 *>(smem + p.off_an);                    // [RB*16][2r]
  __half *xp_s = reinterpret_cast<__half *>(smem + p.off_xp);
  float *xs_s = reinterpret_cast<float *>(smem + p.off_xs);    // [KP*GPB][MPAD] group sums of x
  float *sc_s = reinterpret_cast<float *>(smem + p.off_sc);    // [2 KP][MPAD] half-block scales 2^(24-e)
  float *slot_s = reinterpret_cast<float *>(smem + p.off_slots);
  float *red_s = reinterpret_cast<float *>(smem + p.off_red);  // [4 * threads] chunk sums of tile partials
  float *rt_s = reinterpret_cast<float *>(smem + p.off_rt);    // [M][Qp] tile partials summed over tiles
  float *yv_s = reinterpret_cast<float *>(smem + p.off_yv);    // [RB*16][MPAD] residual, then stored outputs (down)
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + p.off_bar);
  int *last_s = reinterpret_cast<int *>(smem + p.off_last);

  // ---- 1. weight prefetch (independent of the previous kernel) ----
  // Warp (rg, wk) owns row tiles rg*TPW .. rg*TPW+TPW-1 of the block and
  // blocks [kbs, kbe) of the panel; its lane 0 bulk-copies exactly that
  // slice (every projection) on its own barrier, so each warp starts as soon
  // as its own weights have landed.
  const int RG = p.RB / TPW;
  const int rg = warp % RG, wk = warp / RG;
  const int kbs = wk * nkb / p.WK, kbe = (wk + 1) * nkb / p.WK;
  const int ntw = max(0, min(TPW, nrt - rg * TPW));  // row tiles of this warp inside the matrix
  const bool has_slice = ntw > 0 && kbe > kbs;
  if (lane == 0 && has_slice) {
    uint64_t *bar = &bars[warp];
    mbar_init(bar, 1);
    fence_barrier_init();
    const int nb = kbe - kbs;
    const uint64_t pol = l2_evict_first_policy();  // weights are read once a step
    mbar_arrive_expect_tx(bar, NPROJ * ntw * nb * (BPK + GPB * 64));
    for (int j = 0; j < ntw; ++j) {
      const int rl = rg * TPW + j, rt = rt0 + rl;
#pragma unroll
      for (int pj = 0; pj < NPROJ; ++pj) {
        const size_t cd = p.off_codes + ((size_t)(pj * p.RB + rl) * p.KP + kbs) * BPK;
        const size_t cs = ((size_t)rt * p.KB + kb0 + kbs) * BPK;
        if (WQ_OK_IF(WQ_RANGE(cd, nb * BPK, p.off_meta, 16), 1, cd) &&
            WQ_OK_IF(WQ_RANGE(cs, nb * BPK, a.nb_codes[pj], 16), 2, cs))
          bulk_g2s_hint(smem + cd, reinterpret_cast<const uint8_t *>(a.codes[pj]) + cs, nb * BPK, bar, pol);
        const size_t md = p.off_meta + ((size_t)(pj * p.RB + rl) * p.KP * GPB + (size_t)kbs * GPB) * 64;
        const size_t ms = ((size_t)rt * NG + (size_t)(kb0 + kbs) * GPB) * 64;
        if (WQ_OK_IF(WQ_RANGE(md, nb * GPB * 64, p.off_lorab, 16), 3, md) &&
            WQ_OK_IF(WQ_RANGE(ms, nb * GPB * 64, a.nb_meta[pj], 16), 4, ms))
          bulk_g2s_hint(smem + md, reinterpret_cast<const uint8_t *>(a.meta[pj]) + ms, nb * GPB * 64, bar, pol);
      }
    }
  }
  // LoRA-B rows of this CTA's row tiles (gate/up with an adapter).
  if (NPROJ == 2 && r > 0) {
    const int rows = nrt * 16, per_row = r / 8;
    for (int i = tid; i < NPROJ * rows * per_row; i += blockDim.x) {
      const int pj = i / (rows * per_row), rem = i % (rows * per_row);
      const int rl = rem / per_row, c = rem % per_row;
      const int n = rt0 * 16 + rl;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      const size_t src = ((size_t)n * r + (size_t)c * 8) * 2;
      const void *lb = pj == 0 ? a.lora_b[0] : a.lora_b[NPROJ - 1];  // no dynamic index into the arguments
      if (n < a.N && WQ_OK_IF(WQ_RANGE(src, 16, pj == 0 ? a.nb_lora_b[0] : a.nb_lora_b[NPROJ - 1], 16), 30, n))
        v = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const uint8_t *>(lb) + src));
      const size_t dst = p.off_lorab + (((size_t)pj * p.RB * 16 + rl) * r + (size_t)c * 8) * 2;
      if (WQ_OK_IF(WQ_RANGE(dst, 16, p.off_an, 16), 31, i)) *reinterpret_cast<uint4 *>(smem + dst) = v;
    }
  }
  // The next layer's LoRA-A columns for this CTA's output rows (down writing
  // tile partials), transposed to [row][2r]: the tile-partial loop reads the
  // 2r values of a row from consecutive addresses (no bank conflicts).
  if (NPROJ == 1 && a.tp_out != nullptr && r > 0) {
    const int per = nrt * 2;  // 16-byte chunks per LoRA-A row (16 columns a tile)
    for (int i = tid; i < 2 * r * per; i += blockDim.x) {
      const int j = i % (2 * r), c = i / (2 * r);
      const int col = rt0 * 16 + c * 8;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      const size_t src = ((size_t)j * a.N + col) * 2;
      if (col + 8 <= a.N && WQ_OK_IF(WQ_RANGE(src, 16, a.nb_an, 16), 32, i))
        v = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const uint8_t *>(a.lora_a_next) + src));
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const size_t e = (size_t)(c * 8 + t) * 2 * r + j;
        if (WQ_OK_IF(WQ_RANGE(p.off_an + e * 2, 2, p.off_xp, 2), 33, i))
          an_s[e] = __ushort_as_bfloat16(static_cast<unsigned short>(w[t >> 1] >> (16 * (t & 1))));
      }
    }
  }
  for (int i = tid; i < nkb * GPB * MPAD; i += blockDim.x) xs_s[i] = 0.f;
  for (int i = tid; i < 2 * nkb * MPAD; i += blockDim.x) sc_s[i] = 0.f;
  __syncthreads();  // barrier initialisation visible before any thread waits on it

  pdl_wait();  // activations and tile partials of the previous kernel are ready

  // ---- 2. inputs of the previous kernel, all requested in one round trip ----
  // (a) tile partials of the input (gate/up): work item = (chunk of tiles,
  // token, 4 values); its first 8 tiles are loaded now, added below.
  const bool use_tp = NPROJ == 2 && a.tp != nullptr;
  const int Q4 = Qp / 4;
  const int ntb8 = (a.ntp + 7) / 8;
  const int nchk = use_tp ? max(1, min((4 * (int)blockDim.x) / (M * Qp), ntb8)) : 1;
  const int tpc = (a.ntp + nchk - 1) / nchk;  // tiles per chunk
  const int tp_items = use_tp ? nchk * M * Q4 : 0;
  float4 tv[8];
  auto tp_item_load = [&](int item, int tb) {
    const int c = item / (M * Q4), rem = item - c * (M * Q4);
    const int m = rem / Q4, j = rem - m * Q4;
    const int t1 = min((c + 1) * tpc, a.ntp);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const size_t o = ((size_t)(tb + u) * M + m) * Qp + 4 * j;
      tv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (tb + u < t1 && WQ_OK_IF(WQ_RANGE(o * 4, 16, a.nb_tp, 16), 34, tb + u))
        tv[u] = __ldcg(reinterpret_cast<const float4 *>(a.tp + o));
    }
  };
  if (tid < tp_items) tp_item_load(tid, (tid / (M * Q4)) * tpc);
  // (b) residual rows of this CTA (down): the first RV per thread into
  // registers now, parked in shared memory after the conversion below
  constexpr int RV = 4;
  const int nres = (NPROJ == 1 && a.residual) ? nrt * 16 * M : 0;
  __nv_bfloat16 resv[RV];
#pragma unroll
  for (int k = 0; k < RV; ++k) {
    const int i = tid + k * (int)blockDim.x;
    resv[k] = __float2bfloat16_rn(0.f);
    if (i < nres) {
      const int rl = M == 1 ? i : i / M, m = M == 1 ? 0 : i - rl * M;
      const int n = rt0 * 16 + rl;
      if (n < a.N && WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * 2, 2, a.nb_res, 2), 29, n))
        resv[k] = __ldcg(reinterpret_cast<const __nv_bfloat16 *>(a.residual) + (size_t)m * a.N + n);
    }
  }
  // (c) the activation panel, staged by asynchronous 16-byte copies: the raw
  // bf16 rows in the natural order (converted in place below), or the
  // producer's ready binary16 panel
  const bool pre = HALF && NPROJ == 1 && a.pre_x != nullptr;
  const int kbeg = kb0 * 128;
  {
    const uint8_t *srcb = reinterpret_cast<const uint8_t *>(pre ? (const void *)a.pre_x : a.act);
    const size_t row = pre ? (size_t)a.pre_stride : (size_t)a.K;
    const size_t nb_src = pre ? a.nb_pre_x : a.nb_act;
    (void)nb_src;
    const int cpr = nkb * 16;  // 16-byte chunks per token row of the panel
    for (int i = tid; i < M * cpr; i += blockDim.x) {
      const int m = M == 1 ? 0 : i / cpr, c = i - m * cpr;
      const int feat = kbeg + c * 8;
      __half *dst = xp_s + (size_t)m * p.xstride + c * 8;
      const size_t src = ((size_t)m * row + feat) * 2;
      if (!WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)m * p.xstride + c * 8) * 2, 16, p.off_xs, 16), 7, i)) continue;
      if (feat < a.K && WQ_OK_IF(WQ_RANGE(src, 16, nb_src, 16), 8, src))
        cp_async16(dst, srcb + src);
      else
        *reinterpret_cast<uint4 *>(dst) = make_uint4(0u, 0u, 0u, 0u);
    }
    cp_async_commit();
  }
  // (d) with the ready panel: its half-block scales and the group sums
  // (from 32-feature sums, added in order)
  // Four items a thread per round, loads first, so that they are in
  // flight together.
  if (pre) {
    const int nsc = 2 * nkb * M;
    for (int i0 = tid; i0 < nsc; i0 += 4 * blockDim.x) {
      float v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * (int)blockDim.x, h = i / M, m = i - h * M, hb = 2 * kb0 + h;
        v[u] = 0.f;
        if (i < nsc && hb * 64 < a.K && WQ_OK_IF(WQ_RANGE(((size_t)hb * M + m) * 4, 4, a.nb_pre_sc, 4), 47, hb))
          v[u] = ldcg_f32(a.pre_sc + (size_t)hb * M + m);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * (int)blockDim.x, h = i / M, m = i - h * M;
        if (i < nsc && WQ_OK_IF(WQ_RANGE(p.off_sc + ((size_t)h * MPAD + m) * 4, 4, p.off_slots, 4), 48, h))
          sc_s[h * MPAD + m] = v[u];
      }
    }
    constexpr int QPG = GROUP / 32;
    const int nxs = nkb * GPB * M;
    for (int i0 = tid; i0 < nxs; i0 += 2 * blockDim.x) {
      float v[2][QPG];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int i = i0 + u * (int)blockDim.x, g = i / M, m = i - g * M;
        const int q0 = (kb0 * GPB + g) * QPG;
#pragma unroll
        for (int q = 0; q < QPG; ++q) {
          v[u][q] = 0.f;
          if (i < nxs && (q0 + q) * 32 < a.K &&
              WQ_OK_IF(WQ_RANGE(((size_t)(q0 + q) * M + m) * 4, 4, a.nb_pre_xs, 4), 49, q0 + q))
            v[u][q] = ldcg_f32(a.pre_xs + (size_t)(q0 + q) * M + m);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int i = i0 + u * (int)blockDim.x, g = i / M, m = i - g * M;
        float sum = 0.f;
#pragma unroll
        for (int q = 0; q < QPG; ++q) sum += v[u][q];
        if (i < nxs && WQ_OK_IF(WQ_RANGE(p.off_xs + ((size_t)g * MPAD + m) * 4, 4, p.off_sc, 4), 50, g))
          xs_s[g * MPAD + m] = sum;
      }
    }
  }
  // (a) continued: add the loaded tile partials (more rounds only when a
  // chunk has more than 8 tiles)
  for (int item = tid; item < tp_items; item += blockDim.x) {
    const int c = item / (M * Q4), rem = item - c * (M * Q4);
    const int t0 = c * tpc, t1 = min(t0 + tpc, a.ntp);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int tb = t0; tb < t1; tb += 8) {
      if (item != tid || tb != t0) tp_item_load(item, tb);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        acc.x += tv[u].x;
        acc.y += tv[u].y;
        acc.z += tv[u].z;
        acc.w += tv[u].w;
      }
    }
    // chunk sums: red_s[c][m][Qp] (several chunks) or directly rt_s[m][Qp]
    float *dst = (nchk > 1 ? red_s + (size_t)c * M * Qp : rt_s) + (size_t)rem * 4;
    if (WQ_OK_IF(nchk > 1 ? WQ_RANGE((size_t)(dst - red_s) * 4 + p.off_red, 16, p.off_rt, 16)
                          : WQ_RANGE((size_t)(dst - rt_s) * 4 + p.off_rt, 16, p.off_yv, 16), 36, item))
      *reinterpret_cast<float4 *>(dst) = acc;
  }
  cp_async_wait_all();
  __syncthreads();
  // The next launch may start now: its weight stream then runs while this
  // launch computes, not while its latency-bound input loads above are in
  // flight.
  pdl_launch_dependents();
  // The tile partials summed over the chunks (fixed order) and, with the
  // RMSNorm, each token's scale rs = 1/sqrt(mean(x^2) + eps) in place of its
  // sum of squares: their inputs are complete here, so this runs before the
  // dot products instead of behind two more barriers after them, on the
  // last threads (their warps convert the fewest items below).
  if (use_tp && (nchk > 1 || a.prenorm)) {
    const size_t cst = (size_t)M * Qp;  // stride between chunks
    for (int pair = (int)blockDim.x - 1 - tid; pair < M * Qp; pair += blockDim.x) {
      float s = 0.f;
      if (nchk > 1) {
        // four loads in flight, added in chunk order
        int c = 0;
        for (; c + 4 <= nchk; c += 4) {
          const float v0 = red_s[c * cst + pair], v1 = red_s[(c + 1) * cst + pair];
          const float v2 = red_s[(c + 2) * cst + pair], v3 = red_s[(c + 3) * cst + pair];
          s += v0;
          s += v1;
          s += v2;
          s += v3;
        }
        for (; c < nchk; ++c) s += red_s[c * cst + pair];
      } else {
        s = rt_s[pair];
      }
      if (a.prenorm && pair % Qp == 0) s = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(s, (float)a.K), kRmsEps)));
      if (WQ_OK_IF(WQ_RANGE(p.off_rt + (size_t)pair * 4, 4, p.off_yv, 4), 37, pair)) rt_s[pair] = s;
    }
  }
  // Activation panel -> binary16 in place, one (block, token) item per warp.
  // Scale 2^e puts the block's max|x| in [2^14, 2^15): binary16 then holds
  // every scaled bf16 value exactly (bf16 has 8 significant bits), far from
  // overflow.  Lane L holds features 4L..4L+3 of the block, i.e. k-step L/4,
  // and writes them in the order the B fragments read them.
  // A warp converts CU consecutive (block, token) items together -- the
  // tokens of a block, or consecutive blocks of one token: independent
  // dependency chains (load, max reduction, shuffles) in flight at once.
  constexpr int CU = NPROJ == 2 ? 4 : 2;  // fewer for the down kernel (64 registers)
  const int nitems = pre ? 0 : nkb * M;
  const int st = lane >> 2, hi = (lane >> 1) & 1;
  // bit-position class of the codes that meet these features: 4^c for 2-bit
  // codes (c from the k-step parity and the feature half), 16^c for 4-bit
  // codes (c from the feature half)
  const int sh = BITS != 4 ? 4 * (st & 1) + 2 * hi : 4 * hi;
  const int u0 = 4 * (lane & 1) + hi;  // features (2j, 2j+1) of a half sit in word 2j + half
  const bool lo_half = lane < 16;      // features 0..63 of the block
  for (int it0 = warp * CU; it0 < nitems; it0 += CU * nwarps) {
    float f[CU][4];
    int kbv[CU], mv[CU], e0v[CU], e1v[CU];
#pragma unroll
    for (int u = 0; u < CU; ++u) {
      const int it = it0 + u;  // warp-uniform
      kbv[u] = M == 1 ? it : it / M;
      mv[u] = M == 1 ? 0 : it - kbv[u] * M;
      uint2 raw = make_uint2(0u, 0u);
      if (it < nitems &&
          WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)mv[u] * p.xstride + kbv[u] * 128 + 4 * lane) * 2, 8, p.off_xs, 8), 11,
                   it))
        raw = lds64(xp_s + (size_t)mv[u] * p.xstride + (size_t)kbv[u] * 128 + 4 * lane);
      f[u][0] = bf16_lo(raw.x);
      f[u][1] = bf16_hi(raw.x);
      f[u][2] = bf16_lo(raw.y);
      f[u][3] = bf16_hi(raw.y);
    }
#pragma unroll
    for (int u = 0; u < CU; ++u) {
      // max |x| of the block or of each half: non-negative floats order like
      // their bit patterns
      const uint32_t v = __float_as_uint(fmaxf(fmaxf(fabsf(f[u][0]), fabsf(f[u][1])), fmaxf(fabsf(f[u][2]), fabsf(f[u][3]))));
      const uint32_t mx0 = __reduce_max_sync(0xffffffffu, HALF ? (lo_half ? v : 0u) : v);
      const uint32_t mx1 = HALF ? __reduce_max_sync(0xffffffffu, lo_half ? 0u : v) : mx0;
      e0v[u] = block_exponent(mx0);
      e1v[u] = block_exponent(mx1);
    }
    __syncwarp();  // every lane has read its raw features before the blocks are overwritten
#pragma unroll
    for (int u = 0; u < CU; ++u) {
      const int it = it0 + u;
      if (it >= nitems) break;  // warp-uniform
      const float mul = exp2i((lo_half ? e0v[u] : e1v[u]) - sh);
      uint32_t *slot = reinterpret_cast<uint32_t *>(xp_s + (size_t)mv[u] * p.xstride + (size_t)kbv[u] * 128 + st * 16);
      slot[u0] = pack_half2(f[u][0] * mul, f[u][1] * mul);
      slot[u0 + 2] = pack_half2(f[u][2] * mul, f[u][3] * mul);
      // per-group sums of x (natural units) for the zero-point term
      float gs = (f[u][0] + f[u][1]) + (f[u][2] + f[u][3]);
#pragma unroll
      for (int o = 1; o < LPG; o <<= 1) gs += __shfl_xor_sync(0xffffffffu, gs, o);
      if ((lane % LPG) == 0) {
        const int gl = kbv[u] * GPB + lane / LPG;
        if (WQ_OK_IF(WQ_RANGE(p.off_xs + ((size_t)gl * MPAD + mv[u]) * 4, 4, p.off_sc, 4), 14, it))
          xs_s[gl * MPAD + mv[u]] = gs;
      }
      if (lane < 2 && WQ_OK_IF(WQ_RANGE(p.off_sc + ((size_t)(2 * kbv[u] + lane) * MPAD + mv[u]) * 4, 4, p.off_slots, 4), 12, it))
        sc_s[(2 * kbv[u] + lane) * MPAD + mv[u]] = exp2i(24 - (lane == 0 ? e0v[u] : e1v[u]));
    }
  }
  for (int i = tid; i < nres; i += blockDim.x) {
    const int k = (i - tid) / (int)blockDim.x;
    const int rl = M == 1 ? i : i / M, m = M == 1 ? 0 : i - rl * M;
    float v = 0.f;
    if (k < RV) {
#pragma unroll
      for (int kk = 0; kk < RV; ++kk)
        if (kk == k) v = __bfloat162float(resv[kk]);
    } else {
      const int n = rt0 * 16 + rl;
      if (n < a.N && WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * 2, 2, a.nb_res, 2), 29, n))
        v = __bfloat162float(__ldcg(reinterpret_cast<const __nv_bfloat16 *>(a.residual) + (size_t)m * a.N + n));
    }
    if (WQ_OK_IF(WQ_RANGE(p.off_yv + ((size_t)rl * MPAD + m) * 4, 4, p.off_bar, 4), 39, i))
      yv_s[(size_t)rl * MPAD + m] = v;
  }
  __syncthreads();

  // ---- 3./4. tensor-core dot products ----
  if (ntw > 0) {
    const bool ok = !has_slice || mbar_wait(&bars[warp], 0);
    if (!ok && lane == 0) record_timeout();
    // tile j of this warp: codes at + j*KP*BPK, meta at + j*KP*GPB*64.  A
    // missing tile (ragged row end, j >= ntw) multiplies whatever its shared
    // memory holds and is never stored.
    const uint8_t *cbase = codes_s + (size_t)(rg * TPW * p.KP) * BPK + lane * 16;
    const uint8_t *mbase = meta_s + (size_t)(rg * TPW * p.KP * GPB) * 64 + (lane >> 2) * 8;
    const size_t cproj = (size_t)p.RB * p.KP * BPK;
    const size_t mproj = (size_t)p.RB * p.KP * GPB * 64;
    for (int tc = 0; tc * TOK < M; ++tc) {
      float ctot[NPROJ][TPW][NT][4];
#pragma unroll
      for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
        for (int j = 0; j < TPW; ++j)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int q = 0; q < 4; ++q) ctot[pj][j][nt][q] = 0.f;
      for (int kb = ok ? kbs : kbe; kb < kbe; ++kb) {
        uint32_t b[8][NT][2];
        float2 scv[2][NT];  // activation scales of the block's two halves
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int col = tc * TOK + nt * 8 + 2 * (lane & 3);
            scv[h][nt] = make_float2(0.f, 0.f);
            if ((HALF || h == 0) &&
                WQ_OK_IF(WQ_RANGE(p.off_sc + ((size_t)(2 * kb + h) * MPAD + col) * 4, 8, p.off_slots, 8), 18, col))
              scv[h][nt] = *reinterpret_cast<const float2 *>(sc_s + (2 * kb + h) * MPAD + col);
            if (!HALF && h == 1) scv[1][nt] = scv[0][nt];
          }
#pragma unroll
        for (int ks = 0; ks < 8; ++ks)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int m = tc * TOK + nt * 8 + (lane >> 2);
            b[ks][nt][0] = 0u;
            b[ks][nt][1] = 0u;
            if (m < M && WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)m * p.xstride + (kb * 8 + ks) * 16 + 4 * (lane & 3)) * 2,
                                           8, p.off_xs, 8), 15, kb)) {
              const uint2 v = lds64(xp_s + (size_t)m * p.xstride + (kb * 8 + ks) * 16 + 4 * (lane & 3));
              b[ks][nt][0] = v.x;
              b[ks][nt][1] = v.y;
            }
          }
        constexpr int NW = BITS == 2 ? 4 : BITS == 3 ? 6 : 8;  // code words a lane holds per (tile, block)
        uint32_t wds[NPROJ][TPW][NW];
#pragma unroll
        for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
          for (int j = 0; j < TPW; ++j) {
            const uint8_t *cb = cbase + pj * cproj + ((size_t)j * p.KP + kb) * BPK;
#pragma unroll
            for (int q = 0; q < NW; ++q) wds[pj][j][q] = 0u;
            if (WQ_OK_IF(WQ_RANGE(cb - smem, BITS == 2 ? 16 : BITS == 3 ? 520 - 8 * lane : 528, p.off_meta, 16),
                         16, kb)) {
              const uint4 w0 = lds128(cb);
              wds[pj][j][0] = w0.x; wds[pj][j][1] = w0.y; wds[pj][j][2] = w0.z; wds[pj][j][3] = w0.w;
              if (BITS == 3) {  // the lane's two words of the high bit plane, at 512 + 8 lane in the block
                const uint2 w1 = lds64(cb + 512 - 8 * lane);
                wds[pj][j][4] = w1.x; wds[pj][j][5] = w1.y;
              }
              if (BITS == 4) {
                const uint4 w1 = lds128(cb + 512);
                wds[pj][j][NW - 4] = w1.x; wds[pj][j][NW - 3] = w1.y;
                wds[pj][j][NW - 2] = w1.z; wds[pj][j][NW - 1] = w1.w;
              }
            }
          }
        // Accumulation chains per (projection, tile): one, or (HALF) two, one
        // per half of the block, issued alternately (k-steps 0,4,1,5,..).
        // The first MMA of a chain in a group starts from zero.
        constexpr int NCH = HALF ? 2 : 1;
        constexpr int GH = GS < 4 ? GS : 4;  // k-steps of a group inside one chain (HALF)
        float acc[NCH][NPROJ][TPW][NT][4];
        // per group: ctot += s * (sx * sum_k code * x' - z * sum_k x) for the
        // chains (c0, c1) of the group, the affine dequantization s (q - z)
        // with x' = x / sx (sx of the chain's half)
        auto group_epi = [&](const int gl, const int c0, const int c1) {
          float2 xs[NT];
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int col = tc * TOK + nt * 8 + 2 * (lane & 3);
            xs[nt] = make_float2(0.f, 0.f);
            if (WQ_OK_IF(WQ_RANGE(p.off_xs + ((size_t)gl * MPAD + col) * 4, 8, p.off_sc, 8), 14, gl))
              xs[nt] = *reinterpret_cast<const float2 *>(xs_s + gl * MPAD + col);
          }
#pragma unroll
          for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
            for (int j = 0; j < TPW; ++j) {
              const uint8_t *mp = mbase + pj * mproj + ((size_t)j * p.KP * GPB + gl) * 64;
              uint2 sz = make_uint2(0u, 0u);
              if (WQ_OK_IF(WQ_RANGE(mp - smem, 8, p.off_lorab, 8), 17, gl)) sz = lds64(mp);
              const float s_lo = half_bits_to_float(sz.x), s_hi = half_bits_to_float(sz.x >> 16);
              const float zs_lo = -s_lo * half_bits_to_float(sz.y), zs_hi = -s_hi * half_bits_to_float(sz.y >> 16);
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                float *ct = ctot[pj][j][nt];
                const float2 sa = scv[c0][nt];
                const float *ga = acc[c0][pj][j][nt];
                ct[0] = fmaf(s_lo * sa.x, ga[0], ct[0]);
                ct[1] = fmaf(s_lo * sa.y, ga[1], ct[1]);
                ct[2] = fmaf(s_hi * sa.x, ga[2], ct[2]);
                ct[3] = fmaf(s_hi * sa.y, ga[3], ct[3]);
                if (c1 != c0) {
                  const float2 sb = scv[c1][nt];
                  const float *gb = acc[c1][pj][j][nt];
                  ct[0] = fmaf(s_lo * sb.x, gb[0], ct[0]);
                  ct[1] = fmaf(s_lo * sb.y, gb[1], ct[1]);
                  ct[2] = fmaf(s_hi * sb.x, gb[2], ct[2]);
                  ct[3] = fmaf(s_hi * sb.y, gb[3], ct[3]);
                }
                ct[0] = fmaf(zs_lo, xs[nt].x, ct[0]);
                ct[1] = fmaf(zs_lo, xs[nt].y, ct[1]);
                ct[2] = fmaf(zs_hi, xs[nt].x, ct[2]);
                ct[3] = fmaf(zs_hi, xs[nt].y, ct[3]);
              }
            }
        };
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int ks = NCH == 2 ? (i >> 1) + 4 * (i & 1) : i;
          const int ch = NCH == 2 ? (i & 1) : 0;
          const bool first = (ks % (NCH == 2 ? GH : GS)) == 0;  // first k-step of this chain in the group
#pragma unroll
          for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
            for (int j = 0; j < TPW; ++j) {
              uint32_t af[4];
              if (BITS == 2) {
                const uint32_t x = wds[pj][j][(ks >> 1) & 3];
                const uint32_t x8 = x >> 8;
                const int s4 = (ks & 1) * 4;
                af[0] = x & (0x00030003u << s4);   // rows g,   features 2t..2t+1
                af[1] = x8 & (0x00030003u << s4);  // rows g+8
                af[2] = x & (0x000C000Cu << s4);   // rows g,   features 2t+8..2t+9
                af[3] = x8 & (0x000C000Cu << s4);  // rows g+8
              } else if (BITS == 3) {
                // the low two bits as for 2-bit codes; the high bit of the same
                // code from the plane word, shifted to bit 2c + 2 (c the class):
                // << 2 / << 1 for rows g / g+8 of an even 2-bit word, >> 6 / >> 7
                // of an odd one.  A half then reads q 4^c 2^-24, q < 8.
                const int wi = (ks >> 1) & 3;
                const uint32_t x = wds[pj][j][wi];
                const uint32_t x8 = x >> 8;
                const uint32_t hw = wds[pj][j][4 + (wi >> 1)];
                const uint32_t h0 = (wi & 1) ? hw >> 6 : hw << 2, h1 = (wi & 1) ? hw >> 7 : hw << 1;
                const int s4 = (ks & 1) * 4;
                af[0] = (x & (0x00030003u << s4)) | (h0 & (0x00040004u << s4));
                af[1] = (x8 & (0x00030003u << s4)) | (h1 & (0x00040004u << s4));
                af[2] = (x & (0x000C000Cu << s4)) | (h0 & (0x00100010u << s4));
                af[3] = (x8 & (0x000C000Cu << s4)) | (h1 & (0x00100010u << s4));
              } else {
                const uint32_t x = wds[pj][j][ks & (NW - 1)];
                const uint32_t x8 = x >> 8;
                af[0] = x & 0x000F000Fu;
                af[1] = x8 & 0x000F000Fu;
                af[2] = x & 0x00F000F0u;
                af[3] = x8 & 0x00F000F0u;
              }
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                if (first)
                  mma_f16_16816_zc(acc[ch][pj][j][nt], af, b[ks][nt][0], b[ks][nt][1]);
                else
                  mma_f16_16816(acc[ch][pj][j][nt], af, b[ks][nt][0], b[ks][nt][1]);
              }
            }
          if (NCH == 1) {
            if ((ks + 1) % GS == 0) group_epi(kb * GPB + ks / GS, 0, 0);
          } else if (GS == 8) {
            if (i == 7) group_epi(kb, 0, 1);  // a group spans both halves
          } else if ((ks + 1) % GS == 0) {
            group_epi(kb * GPB + ks / GS, ch, ch);
          }
        }
      }
      // per-warp partial -> shared slot [wk][row tile][pj][16][M] (valid tokens only)
#pragma unroll
      for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
        for (int j = 0; j < TPW; ++j) {
          if (j >= ntw) continue;
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int col = tc * TOK + nt * 8 + 2 * (lane & 3), r0 = lane >> 2;
            float *sl = slot_s + (size_t)((wk * p.RB + rg * TPW + j) * NPROJ + pj) * 16 * M;
#pragma unroll
            for (int c = 0; c < 2; ++c) {
              if (col + c >= M) continue;
              if (!WQ_OK_IF(WQ_RANGE((uint8_t *)(sl + (r0 + 8) * M + col + c) - smem, 4, p.off_red, 4), 20, col))
                continue;
              sl[r0 * M + col + c] = ctot[pj][j][nt][c];
              sl[(r0 + 8) * M + col + c] = ctot[pj][j][nt][2 + c];
            }
          }
        }
    }
  }
  __syncthreads();

  // ---- 5. add up the k-split warps' partial sums (fixed order) ----
  const int per_rt = NPROJ * 16 * M;
  if (p.WK > 1) {
    const int nel = nrt * per_rt;
    const size_t wst = (size_t)p.RB * per_rt;  // slot stride between warps
    for (int i = tid; i < nel; i += blockDim.x) {
      if (!WQ_OK_IF(WQ_RANGE(p.off_slots + ((size_t)(p.WK - 1) * wst + i) * 4, 4, p.off_red, 4), 21, i)) continue;
      // four loads in flight, added in warp order
      float s = 0.f;
      int w = 0;
      for (; w + 4 <= p.WK; w += 4) {
        const float v0 = slot_s[w * wst + i], v1 = slot_s[(w + 1) * wst + i];
        const float v2 = slot_s[(w + 2) * wst + i], v3 = slot_s[(w + 3) * wst + i];
        s += v0;
        s += v1;
        s += v2;
        s += v3;
      }
      for (; w < p.WK; ++w) s += slot_s[w * wst + i];
      slot_s[i] = s;
    }
    __syncthreads();
  }

  if (p.P > 1) {
    for (int i = tid; i < nrt * per_rt; i += blockDim.x) {
      const int rti = i / per_rt, rem = i % per_rt;
      const size_t po = ((size_t)(rt0 + rti) * p.P + panel) * per_rt + rem;
      if (WQ_OK_IF(WQ_RANGE(po * 4, 4, a.nb_part, 4), 22, po)) a.partials[po] = slot_s[i];
    }
    __threadfence();
    __syncthreads();
    if (tid < nrt && WQ_OK_IF(WQ_RANGE((size_t)(rt0 + tid) * 4, 4, a.nb_cnt, 4), 23, rt0 + tid)) {
      const unsigned prev = atomicAdd(&a.counters[rt0 + tid], 1u);
      last_s[tid] = prev == (unsigned)(p.P - 1);
    }
    __syncthreads();
    __threadfence();
    for (int i = tid; i < nrt * per_rt; i += blockDim.x) {
      const int rti = i / per_rt, rem = i % per_rt;
      if (!last_s[rti]) continue;
      const float *src = a.partials + (size_t)(rt0 + rti) * p.P * per_rt + rem;
      float s = 0.f;
      if (WQ_OK_IF(WQ_RANGE((src - a.partials + (size_t)(p.P - 1) * per_rt) * 4, 4, a.nb_part, 4), 24, i))
        s = sum_strided_cg(src, per_rt, p.P);
      slot_s[i] = s;
    }
    if (tid < nrt && last_s[tid]) a.counters[rt0 + tid] = 0u;
    __syncthreads();
  }  // one panel: every row tile is finished here (last_s is not read)

  // ---- epilogue: RMSNorm scale, LoRA-B + SiLU(g) * u; or residual add ----
  const int rows = nrt * 16;
  // gate/up output of local row rl, token m (before the bf16 store)
  auto gateup_h = [&](int rl, int m) -> float {
    const int rti = rl >> 4, r16 = rl & 15;
    float g = slot_s[(size_t)(rti * NPROJ) * 16 * M + r16 * M + m];
    float u = slot_s[(size_t)(rti * NPROJ + 1) * 16 * M + r16 * M + m];
    // xin = x * rs (Sec. 3.3 MLP input after RMSNorm, never stored):
    // g = rs * (x deq(Wg)^T + lora_scale * (x A_g^T) B_g^T)
    const float rs = use_tp && a.prenorm ? rt_s[(size_t)m * Qp] : 1.f;
    if (use_tp && r > 0) {
      const float *tg = rt_s + (size_t)m * Qp + 1;
      const float *tu = tg + r;
      const __nv_bfloat16 *bg = lorab_s + (size_t)rl * r;
      const __nv_bfloat16 *bu = lorab_s + ((size_t)p.RB * 16 + rl) * r;
      float lg = 0.f, lu = 0.f;
      const bool lora_ok =
          WQ_OK_IF(WQ_RANGE(p.off_rt + ((size_t)m * Qp + Q) * 4 - 4, 4, p.off_yv, 4), 25, m) &&
          WQ_OK_IF(WQ_RANGE(p.off_lorab + (((size_t)p.RB * 16 + rl) * r + r) * 2 - 16, 16, p.off_an, 16), 26, rl);
      for (int q = 0; lora_ok && q < r; q += 8) {
        float fg[8], fu[8];
        unpack_bf16x8(lds128(bg + q), fg);
        unpack_bf16x8(lds128(bu + q), fu);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          lg = fmaf(tg[q + e], fg[e], lg);
          lu = fmaf(tu[q + e], fu[e], lu);
        }
      }
      g = fmaf(a.lora_scale, lg, g);
      u = fmaf(a.lora_scale, lu, u);
    }
    g *= rs;
    u *= rs;
    return g / (1.f + __expf(-g)) * u;
  };
  if (NPROJ == 2 && a.hq_out != nullptr) {
    // Decode chain (P = 1, RB a multiple of 4): h is also written as the
    // down launch's binary16 panel.  A pair of warps per (token, 64-row
    // half), one row a lane: each warp reduces its 32 rows (largest |h|, sum),
    // the pair swaps maxima through shared memory behind a named barrier.
    const int nhalf = p.RB / 4, npair = nwarps >> 1;
    const int pair = warp >> 1, sub = warp & 1;
    uint32_t *xch = reinterpret_cast<uint32_t *>(red_s);  // [2][npair][2], alternating by iteration
    for (int item = pair, it = 0; item < nhalf * M; item += npair, ++it) {
      const int m = item / nhalf, hh = item - m * nhalf;
      const int rl = hh * 64 + sub * 32 + lane;
      const int n = rt0 * 16 + rl;
      float hv = 0.f;
      if (n < a.N) {
        const __nv_bfloat16 hb = __float2bfloat16_rn(gateup_h(rl, m));
        if (WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * 2, 2, a.nb_out, 2), 27, n))
          reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = hb;
        hv = __bfloat162float(hb);
      }
      const uint32_t mq = __reduce_max_sync(0xffffffffu, __float_as_uint(fabsf(hv)));
      float sq = hv;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
      const int nq = rt0 * 16 + hh * 64 + sub * 32;  // first feature of this warp's 32
      if (lane == 0) {
        const int xi = ((it & 1) * npair + pair) * 2 + sub;
        if (WQ_OK_IF(WQ_RANGE(p.off_red + (size_t)xi * 4, 4, p.off_rt, 4), 51, xi)) xch[xi] = mq;
        if (nq < a.N && WQ_OK_IF(WQ_RANGE(((size_t)(nq >> 5) * M + m) * 4, 4, a.nb_hxs, 4), 52, nq))
          a.hxs_out[(size_t)(nq >> 5) * M + m] = sq;
      }
      named_barrier_sync(1 + pair, 64);
      const int xb = ((it & 1) * npair + pair) * 2;
      const int e = block_exponent(max(xch[xb], xch[xb + 1]));
      const int n0 = rt0 * 16 + hh * 64;
      if (sub == 0 && lane == 0 && WQ_OK_IF(WQ_RANGE(((size_t)(n0 >> 6) * M + m) * 4, 4, a.nb_hsc, 4), 54, n0))
        a.hsc_out[(size_t)(n0 >> 6) * M + m] = exp2i(24 - e);
      if (n < a.N) {
        // position in the B-fragment order of the 4-bit down kernel: k-step
        // st, feature pair pr -> word 4((pr >> 1) & 1) + (pr >> 2) + 2(pr & 1);
        // features 8..15 of a k-step scaled by 16^-1 (their code class)
        const int st = (n >> 4) & 7, pr = (n & 15) >> 1;
        const int w = 4 * ((pr >> 1) & 1) + (pr >> 2) + 2 * (pr & 1);
        const size_t o = (size_t)m * a.hq_stride + (size_t)(n >> 7) * 128 + st * 16 + 2 * w + (n & 1);
        const __half hq = __float2half_rn(hv * exp2i(e - 4 * ((n >> 3) & 1)));
        if (WQ_OK_IF(WQ_RANGE(o * 2, 2, a.nb_hq, 2), 53, n)) a.hq_out[o] = __half_as_ushort(hq);
      }
    }
  } else {
    for (int i = tid; i < rows * M; i += blockDim.x) {
      const int m = i / rows, rl = i % rows;
      const int rti = rl >> 4, r16 = rl & 15;
      if (p.P > 1 && !last_s[rti]) continue;
      const int n = (rt0 + rti) * 16 + r16;
      if (n >= a.N) continue;
      if (NPROJ == 2) {
        const float h = gateup_h(rl, m);
        if (WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * 2, 2, a.nb_out, 2), 27, n))
          reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = __float2bfloat16_rn(h);
      } else {
        float y = slot_s[(size_t)(rti * NPROJ) * 16 * M + r16 * M + m];
        if (!WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * (a.out_f32 ? 4 : 2), a.out_f32 ? 4 : 2, a.nb_out, 2), 28, n))
          continue;
        if (a.residual) y += yv_s[(size_t)rl * MPAD + m];
        if (a.out_f32) {
          reinterpret_cast<float *>(a.out)[(size_t)m * a.N + n] = y;
        } else {
          const __nv_bfloat16 yb = __float2bfloat16_rn(y);
          reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = yb;
          y = __bfloat162float(yb);
        }
        if (WQ_OK_IF(WQ_RANGE(p.off_yv + ((size_t)rl * MPAD + m) * 4, 4, p.off_bar, 4), 38, rl))
          yv_s[(size_t)rl * MPAD + m] = y;
      }
    }
  }

  // ---- the next layer's tile partials of the stored output (down) ----
  // Same arithmetic and order as tile_prep_kernel: s = fma(w_c, y_c, s) over
  // the tile's 16 features, w = y (sum of squares) or a LoRA-A row.
  if (NPROJ == 1 && a.tp_out != nullptr) {
    __syncthreads();
    for (int i = tid; i < nrt * M * Qp; i += blockDim.x) {
      const int rti = i / (M * Qp), rem = i % (M * Qp);
      const int m = rem / Qp, q = rem % Qp;
      if (p.P > 1 && !last_s[rti]) continue;
      const int tile = rt0 + rti;
      const int nv = q < Q ? max(0, min(16, a.N - tile * 16)) : 0;  // rows of the tile inside the matrix
      float vv[16], wv[16];
#pragma unroll
      for (int r16 = 0; r16 < 16; ++r16) {
        const int rl = rti * 16 + r16;
        vv[r16] = yv_s[(size_t)rl * MPAD + m];
        wv[r16] = q == 0 ? vv[r16] : (q < Q ? __bfloat162float(an_s[(size_t)rl * 2 * r + (q - 1)]) : 0.f);
      }
      float s = 0.f;
#pragma unroll
      for (int r16 = 0; r16 < 16; ++r16)
        if (r16 < nv) s = fmaf(wv[r16], vv[r16], s);
      const size_t o = ((size_t)tile * M + m) * Qp + q;
      if (WQ_OK_IF(WQ_RANGE(o * 4, 4, a.nb_tp_out, 4), 35, o)) a.tp_out[o] = s;
    }
  }
}

template <int BITS, int NPROJ, int GROUP, int NT, int TPW>
__global__ void __launch_bounds__(kMaxThreads, NPROJ == 1 && NT == 1 && TPW == 1 ? 2 : 1)
    qgemv_kernel(const GemvArgs a, const GemvPlan p) {
  qgemv_body<BITS, NPROJ, GROUP, NT, TPW>(a, p);
}

// ---------------------------------------------------------------------------
// The same kernel over the routed experts of a mixture-of-experts block
// (Sec. 5's MoE model reads only the experts a token selects).  grid.y runs
// over slots (token t, choice j) -> slot t*top_k + j, one token each; the
// experts' matrices are stacked row-wise ([E*N, K] packed as one matrix, so
// expert e owns row tiles e*RT .. e*RT+RT-1) and slot s computes with expert
// e = slot_expert[s], written by the routing kernel of the same step.  When
// the routing kernel is the previous launch (gate/up), the expert is known
// only after the wait, so the wait comes first and the weight stream follows
// it.  When it ran two launches earlier (down, `slot_expert_ready`), it has
// completed before this launch could start -- the gate/up launch lets its
// dependents start only after its own wait on the routing kernel -- so the
// index is read at once and the weights stream before the wait, overlapping
// the gate/up launch.  Per slot: input row s / slot_div of act, tile
// partials and panel partials / counters of its own, output row s.
// ---------------------------------------------------------------------------
template <int BITS, int NPROJ, int GROUP, int TPW>
__global__ void __launch_bounds__(kMaxThreads, NPROJ == 1 && TPW == 1 ? 2 : 1)
    qgemv_slots_kernel(const GemvArgs a0, const GemvPlan p) {
  if (!a0.slot_expert_ready) pdl_wait();  // slot_expert comes from the previous launch
  const int slot = blockIdx.y;
  const int e = __ldcg(a0.slot_expert + slot);
  if (e < 0 || e >= a0.n_experts) {
    if (threadIdx.x == 0) atomicExch(&g_device_status, -1);  // WQ_ERR_ARG: an expert index outside [0, E)
    return;
  }
  constexpr int WPB = BITS == 2 ? 128 : 256;  // code words per (row tile, 128-feature block)
  const size_t rt = (size_t)p.RT, ng = (size_t)p.KB * (128 / GROUP);
  const int Qp = WQ_TP_STRIDE(a0.r);
  GemvArgs a = a0;
#pragma unroll
  for (int pj = 0; pj < NPROJ; ++pj) {
    a.codes[pj] = a0.codes[pj] + (size_t)e * rt * p.KB * WPB;
    a.meta[pj] = a0.meta[pj] + (size_t)e * rt * ng * 32;
    a.nb_codes[pj] = rt * p.KB * WPB * 4;
    a.nb_meta[pj] = rt * ng * 64;
    if (NPROJ == 2 && a0.r > 0) {
      a.lora_b[pj] = reinterpret_cast<const uint8_t *>(a0.lora_b[pj]) + (size_t)e * a0.N * a0.r * 2;
      a.nb_lora_b[pj] = (size_t)a0.N * a0.r * 2;
    }
  }
  a.act = reinterpret_cast<const uint8_t *>(a0.act) + (size_t)(slot / a0.slot_div) * a0.K * 2;
  a.nb_act = (size_t)a0.K * 2;
  if (a0.tp != nullptr) {
    a.tp = a0.tp + (size_t)slot * a0.ntp * Qp;
    a.nb_tp = (size_t)a0.ntp * Qp * 4;
  }
  const size_t osz = a0.out_f32 ? 4 : 2;
  a.out = reinterpret_cast<uint8_t *>(a0.out) + (size_t)slot * a0.N * osz;
  a.nb_out = (size_t)a0.N * osz;
  if (p.P > 1) {
    const size_t per = rt * p.P * NPROJ * 16;
    a.partials = a0.partials + (size_t)slot * per;
    a.counters = a0.counters + (size_t)slot * rt;
    a.nb_part = per * 4;
    a.nb_cnt = rt * 4;
  }
  qgemv_body<BITS, NPROJ, GROUP, 1, TPW>(a, p);
}

// ---------------------------------------------------------------------------
// Tile partials of an input x [M, d] (d a multiple of 16), one warp per tile
// of 16 features: tp[tile][m][0] = sum_c x_c^2, tp[tile][m][1 + j] =
// sum_c A[j, c] x_c, each as s = fma(w_c, x_c, s) over c in order.  The
// gate/up kernel adds them up into the RMSNorm scale and the LoRA-A
// products x A^T of Eq. 1.  A lane takes the values lane, lane + 32, ..
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) tile_prep_kernel(const __nv_bfloat16 *x, int M, int d,
                                                         const __nv_bfloat16 *lora_a, int r2, float *tp,
                                                         size_t nb_x, size_t nb_a, size_t nb_tp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ntp = d / 16;
  const int tile = blockIdx.x * (blockDim.x >> 5) + warp;
  const int Q = 1 + r2, Qp = (Q + 3) & ~3;
  constexpr int QI = (1 + 2 * kMaxRank + 3) / 32 + 1;  // values a lane takes, at most
  pdl_launch_dependents();
  // The LoRA-A rows of this lane's values (weights, not written by the
  // previous kernel) are loaded before the wait; only x waits for it.
  const uint8_t *x8 = reinterpret_cast<const uint8_t *>(x);
  const uint8_t *a8 = reinterpret_cast<const uint8_t *>(lora_a);
  (void)nb_x;
  (void)nb_a;
  (void)nb_tp;
  uint4 av[QI][2];
#pragma unroll
  for (int i = 0; i < QI; ++i) {
    const int q = lane + 32 * i;
    av[i][0] = av[i][1] = make_uint4(0u, 0u, 0u, 0u);
    if (tile < ntp && q >= 1 && q < Q) {
      const size_t ao = ((size_t)(q - 1) * d + (size_t)tile * 16) * 2;
      if (WQ_OK_IF(WQ_RANGE(ao, 32, nb_a, 16), 45, ao)) {
        av[i][0] = __ldg(reinterpret_cast<const uint4 *>(a8 + ao));
        av[i][1] = __ldg(reinterpret_cast<const uint4 *>(a8 + ao + 16));
      }
    }
  }
  pdl_wait();
  if (tile >= ntp) return;
  for (int m = 0; m < M; ++m) {
    float v[16];
    const size_t xo = ((size_t)m * d + (size_t)tile * 16) * 2;
    uint4 x0 = make_uint4(0u, 0u, 0u, 0u), x1 = x0;
    if (WQ_OK_IF(WQ_RANGE(xo, 32, nb_x, 16), 44, xo)) {
      x0 = ldg_cg128(x8 + xo);
      x1 = ldg_cg128(x8 + xo + 16);
    }
    unpack_bf16x8(x0, *reinterpret_cast<float(*)[8]>(v));
    unpack_bf16x8(x1, *reinterpret_cast<float(*)[8]>(v + 8));
#pragma unroll
    for (int i = 0; i < QI; ++i) {
      const int q = lane + 32 * i;
      if (q >= Qp) break;
      float s = 0.f;
      if (q == 0) {
#pragma unroll
        for (int c = 0; c < 16; ++c) s = fmaf(v[c], v[c], s);
      } else if (q < Q) {
        float w[16];
        unpack_bf16x8(av[i][0], *reinterpret_cast<float(*)[8]>(w));
        unpack_bf16x8(av[i][1], *reinterpret_cast<float(*)[8]>(w + 8));
#pragma unroll
        for (int c = 0; c < 16; ++c) s = fmaf(w[c], v[c], s);
      }  // else padding: 0
      const size_t o = ((size_t)tile * M + m) * Qp + q;
      if (WQ_OK_IF(WQ_RANGE(o * 4, 4, nb_tp, 4), 46, o)) tp[o] = s;
    }
  }
}

// ---------------------------------------------------------------------------
// Host side: planning and launching.
// ---------------------------------------------------------------------------
uint32_t align_up(uint32_t v, uint32_t a) { return (v + a - 1) / a * a; }

int kind_bits(GemvKind k) { return k == kGateUpW2 ? 2 : k == kGateUpW3 ? 3 : 4; }
int kind_nproj(GemvKind k) { return k == kDownW4 ? 1 : 2; }

void compute_layout(GemvKind kind, int group, int r, GemvPlan *p) {
  const int nproj = kind_nproj(kind);
  const int BPK = kind_bits(kind) * 256, GPB = 128 / group;
  uint32_t off = 0;
  p->r = r;
  p->off_codes = off;
  off = align_up(off + (uint32_t)nproj * p->RB * p->KP * BPK, 128);
  p->off_meta = off;
  off = align_up(off + (uint32_t)nproj * p->RB * p->KP * GPB * 64, 128);
  p->off_lorab = off;  // gate/up: LoRA-B rows [2][RB*16][r] bf16
  off = align_up(off + (nproj == 2 ? (uint32_t)nproj * p->RB * 16 * r * 2 : 0u), 128);
  p->off_an = off;  // down: next layer's LoRA-A columns [2r][RB*16] bf16
  off = align_up(off + (nproj == 1 ? (uint32_t)2 * r * p->RB * 16 * 2 : 0u), 128);
  p->xstride = p->KP * 128 + 16;  // row bytes = 256 KP + 32: conflict-free 8-byte fragment loads
  p->off_xp = off;
  off = align_up(off + (uint32_t)p->M * p->xstride * 2, 128);
  p->off_xs = off;
  off = align_up(off + (uint32_t)p->KP * GPB * p->MPAD * 4, 128);
  p->off_sc = off;  // [2 KP][MPAD] half-block activation scales
  off = align_up(off + (uint32_t)2 * p->KP * p->MPAD * 4, 128);
  p->off_slots = off;
  off = align_up(off + (uint32_t)p->WK * p->RB * nproj * 16 * p->M * 4, 128);
  p->off_red = off;  // gate/up: chunk sums of the tile partials [nchk][M][Qp], or the panel epilogue's maxima
  {
    const int Qp = WQ_TP_STRIDE(r);
    const int nchk = std::max(1, std::min(4 * p->threads / (p->M * Qp), p->KB));
    const uint32_t red = (uint32_t)std::max(nchk * p->M * Qp, 4 * (p->threads / 64) + 4) * 4;
    off = align_up(off + (nproj == 2 ? red : 0u), 128);
  }
  p->off_rt = off;
  off = align_up(off + (nproj == 2 ? (uint32_t)p->M * WQ_TP_STRIDE(r) * 4 : 0u), 128);
  p->off_yv = off;
  off = align_up(off + (nproj == 1 ? (uint32_t)p->RB * 16 * p->MPAD * 4 : 0u), 128);
  p->off_bar = off;  // one weight barrier per warp
  off = align_up(off + (uint32_t)p->RB * p->WK * 8, 128);
  p->off_last = off;
  off = align_up(off + (uint32_t)p->RB * 4, 128);
  p->smem = off;
}

constexpr uint32_t kSmemLimit = 232448;       // 227 KB opt-in dynamic shared memory per CTA
constexpr uint32_t kSmemPerSm = 233472;       // 228 KB shared memory per SM
constexpr uint32_t kCoResident = 114 * 1024;  // shared memory per SM that leaves room for the next kernel

bool search_plan(GemvKind kind, int N, int K, int M, int group, int r, int num_sms, GemvPlan *out) {
  const int nproj = kind_nproj(kind);
  const int RT = (N + 15) / 16, KB = (K + 127) / 128;
  const int NT = M <= 8 ? 1 : 2;
  const int tok = 8 * NT;
  const int MPAD = (M + tok - 1) / tok * tok;
  const int chunks = MPAD / tok;
  const double blk_bytes = 256.0 * kind_bits(kind) + 64.0 * (128 / group);
  const double total_bytes = (double)RT * KB * nproj * blk_bytes;
  const int max_warps = kMaxThreads / 32;
  bool found = false;
  double best = 1e300;
  GemvPlan bp{};
  for (int TPW = 1; TPW <= (NT == 1 ? 2 : 1); ++TPW)
  for (int KP = 1; KP <= KB; ++KP) {
    const int P = (KB + KP - 1) / KP;
    if ((KB + P - 1) / P != KP) continue;  // one canonical KP per panel count
    for (int RB = TPW; RB <= std::min((RT + TPW - 1) / TPW * TPW, max_warps * TPW); RB += TPW) {
      const int NRB = (RT + RB - 1) / RB;
      if ((long long)NRB * P > 8LL * num_sms) continue;  // more than 8 CTAs an SM never pays
      for (int WK = 1; WK <= std::min(KP, max_warps / (RB / TPW)); ++WK) {
        GemvPlan p{};
        p.RT = RT; p.KB = KB; p.RB = RB; p.KP = KP; p.WK = WK; p.P = P;
        p.NRB = NRB;
        p.M = M; p.MPAD = MPAD; p.NT = NT; p.TPW = TPW;
        const int warps = RB / TPW * WK;
        p.threads = warps * 32;
        p.units = NRB * P;
        compute_layout(kind, group, r, &p);
        if (p.smem > kSmemLimit) continue;
        const int regs = p.threads * ((kernel_regs(kind, group, NT, TPW) + 7) & ~7);  // registers of a CTA
        const int occ = std::max(1, std::min({(int)(kSmemPerSm / (p.smem + 1024)), 65536 / regs, 2048 / p.threads, 32}));
        const int per_sm = (p.units + num_sms - 1) / num_sms;  // CTAs landing on the busiest SM
        const int waves = (p.units + num_sms * occ - 1) / (num_sms * occ);
        // CTAs resident on a typical SM (a grid up to 10% larger than the SM
        // count leaves only a few SMs with a second CTA)
        const int res = p.units <= num_sms + num_sms / 10 ? 1 : std::min(per_sm, occ);
        // Cycle estimates, calibrated on GB300 timings of the decode chain:
        // after the wait, one L2 round trip for the inputs (~1500), ~250 per
        // converted (block, token) item a warp handles, the MMA loop at ~8
        // cycles per m16n8k16 per scheduler when each scheduler has four
        // warps to switch between (proportionally slower with fewer), ~3000
        // of reduction and epilogue, ~1000 per further CTA on the SM, ~5000
        // for a split-panel fixup (three dependent round trips) plus ~100 per
        // partial a thread adds up, ~3000 between the end of one launch and
        // the release of the next.  The weight stream runs at ~21 B/cycle per
        // SM (HBM over the SMs), at most ~64 B/cycle into one SM.
        const double mma_cta = (double)RB * KP * nproj * 8.0 * NT * chunks;  // RB counts padded tiles
        const double eff = std::min(1.0, (double)warps * std::min(occ, per_sm) / 16.0);  // CTAs of an SM run together
        const double imb = (double)((warps + 3) / 4 * 4) / warps;  // schedulers with one warp more than others
        const double t_mma = per_sm * mma_cta * 8.0 / 4.0 * imb / eff;
        const double items = std::ceil((double)KP * M / warps);
        const double conv = 1500.0 + items * 250.0;
        const double epi = 3000.0 + (r > 0 ? 8.0 * r : 0.0) + std::ceil((double)RB * 16 * M / p.threads) * 20.0;
        // the last-arriving CTA of a row tile loads P partials per output
        const double fix = P > 1 ? 5000.0 + std::ceil((double)RB * 16 * nproj * M / p.threads) * P * 100.0 : 0.0;
        const double W = conv + t_mma + epi + fix + 1000.0 * (per_sm - 1);
        const double sm_bytes = (double)per_sm * RB * KP * nproj * blk_bytes;
        const double stream = std::max(total_bytes / (21.3 * num_sms), sm_bytes / 64.0);
        // The chain alternates gate/up and down launches; the next launch's
        // CTAs can prefetch their weights during this one only if both fit
        // on an SM at once: a gate/up launch may take 5/8 of an SM's
        // registers, a down launch 1/4 (measured: down launches of more
        // than 8 warps a CTA delay the next gate/up launch), and each about
        // half its shared memory.
        const int reg_budget = kind == kDownW4 ? 16384 : 40960;
        const bool room = (uint32_t)res * (p.smem + 1024) <= kCoResident && res * regs <= reg_budget;
        double cost = room ? std::max(stream, 3000.0 + W) : stream + 3000.0 + W;
        if (waves > 1) cost += (waves - 1) * (W + 3000.0);
        cost += 0.5 * p.units;  // ties: fewer, larger CTAs
        if (cost < best) {
          best = cost;
          bp = p;
          found = true;
        }
      }
    }
  }
  if (found) *out = bp;
  return found;
}

}  // namespace

bool plan_gemv(GemvKind kind, int N, int K, int M, int group, int r, int num_sms, GemvPlan *out) {
  if (N <= 0 || K <= 0 || M <= 0 || M > kMaxTokens || num_sms <= 0 || r < 0 || r > kMaxRank) return false;
  if (kind == kDownW4 && r > 0 && N % 8 != 0) return false;  // next-layer LoRA-A columns load 8 at a time
  using Key = std::tuple<int, int, int, int, int, int, int>;
  static std::mutex mu;
  static std::map<Key, std::pair<bool, GemvPlan>> cache;
  const Key key{(int)kind, N, K, M, group, r, num_sms};
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      if (it->second.first) *out = it->second.second;
      return it->second.first;
    }
  }
  GemvPlan p{};
  const bool ok = search_plan(kind, N, K, M, group, r, num_sms, &p);
  {
    std::lock_guard<std::mutex> lock(mu);
    cache[key] = {ok, p};
  }
  if (ok) *out = p;
  return ok;
}

namespace {

template <int BITS, int NPROJ, int GROUP, int NT, int TPW>
cudaError_t launch_t(const GemvPlan &p, const GemvArgs &a, cudaStream_t s, bool pdl) {
  auto kern = qgemv_kernel<BITS, NPROJ, GROUP, NT, TPW>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.units);
  cfg.blockDim = dim3(p.threads);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, a, p);
}

template <int BITS, int NPROJ, int GROUP, int TPW>
cudaError_t launch_slots_t(const GemvPlan &p, const GemvArgs &a, int slots, cudaStream_t s, bool pdl) {
  auto kern = qgemv_slots_kernel<BITS, NPROJ, GROUP, TPW>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.units, slots);
  cfg.blockDim = dim3(p.threads);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, a, p);
}

template <int BITS, int NPROJ>
cudaError_t launch_slots_g(const GemvPlan &p, const GemvArgs &a, int slots, cudaStream_t s, bool pdl) {
  if (p.NT != 1 || p.M != 1) return cudaErrorInvalidValue;
  const bool t2 = p.TPW == 2;
  switch (a.group) {
    case 32: return t2 ? launch_slots_t<BITS, NPROJ, 32, 2>(p, a, slots, s, pdl) : launch_slots_t<BITS, NPROJ, 32, 1>(p, a, slots, s, pdl);
    case 64: return t2 ? launch_slots_t<BITS, NPROJ, 64, 2>(p, a, slots, s, pdl) : launch_slots_t<BITS, NPROJ, 64, 1>(p, a, slots, s, pdl);
    case 128: return t2 ? launch_slots_t<BITS, NPROJ, 128, 2>(p, a, slots, s, pdl) : launch_slots_t<BITS, NPROJ, 128, 1>(p, a, slots, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

template <int BITS, int NPROJ, int GROUP>
const void *kernel_ptr(int NT, int TPW) {
  if (NT == 2) return reinterpret_cast<const void *>(qgemv_kernel<BITS, NPROJ, GROUP, 2, 1>);
  return TPW == 2 ? reinterpret_cast<const void *>(qgemv_kernel<BITS, NPROJ, GROUP, 1, 2>)
                  : reinterpret_cast<const void *>(qgemv_kernel<BITS, NPROJ, GROUP, 1, 1>);
}

template <int BITS, int NPROJ, int GROUP>
cudaError_t launch_v(const GemvPlan &p, const GemvArgs &a, cudaStream_t s, bool pdl) {
  if (p.NT == 2) return p.TPW == 1 ? launch_t<BITS, NPROJ, GROUP, 2, 1>(p, a, s, pdl) : cudaErrorInvalidValue;
  return p.TPW == 2 ? launch_t<BITS, NPROJ, GROUP, 1, 2>(p, a, s, pdl) : launch_t<BITS, NPROJ, GROUP, 1, 1>(p, a, s, pdl);
}

template <int BITS, int NPROJ>
cudaError_t launch_g(const GemvPlan &p, const GemvArgs &a, cudaStream_t s, bool pdl) {
  switch (a.group) {
    case 32: return launch_v<BITS, NPROJ, 32>(p, a, s, pdl);
    case 64: return launch_v<BITS, NPROJ, 64>(p, a, s, pdl);
    case 128: return launch_v<BITS, NPROJ, 128>(p, a, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int kernel_regs(GemvKind kind, int group, int NT, int TPW) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, int, int>, int> cache;
  const auto key = std::make_tuple((int)kind, group, NT, TPW);
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  const int gi = group == 32 ? 0 : group == 64 ? 1 : 2;
  const void *fn = nullptr;
  switch (kind * 3 + gi) {
    case 0: fn = kernel_ptr<2, 2, 32>(NT, TPW); break;
    case 1: fn = kernel_ptr<2, 2, 64>(NT, TPW); break;
    case 2: fn = kernel_ptr<2, 2, 128>(NT, TPW); break;
    case 3: fn = kernel_ptr<4, 2, 32>(NT, TPW); break;
    case 4: fn = kernel_ptr<4, 2, 64>(NT, TPW); break;
    case 5: fn = kernel_ptr<4, 2, 128>(NT, TPW); break;
    case 6: fn = kernel_ptr<4, 1, 32>(NT, TPW); break;
    case 7: fn = kernel_ptr<4, 1, 64>(NT, TPW); break;
    case 8: fn = kernel_ptr<4, 1, 128>(NT, TPW); break;
    case 9: fn = kernel_ptr<3, 2, 32>(NT, TPW); break;
    case 10: fn = kernel_ptr<3, 2, 64>(NT, TPW); break;
    default: fn = kernel_ptr<3, 2, 128>(NT, TPW); break;
  }
  cudaFuncAttributes attr{};
  const int regs = cudaFuncGetAttributes(&attr, fn) == cudaSuccess && attr.numRegs > 0 ? attr.numRegs : 128;
  cache[key] = regs;
  return regs;
}

cudaError_t launch_gemv(GemvKind kind, const GemvPlan &plan, const GemvArgs &args, cudaStream_t stream, bool pdl) {
  if (plan.r != args.r) return cudaErrorInvalidValue;  // shared-memory layout sized for another rank
  switch (kind) {
    case kGateUpW2: return launch_g<2, 2>(plan, args, stream, pdl);
    case kGateUpW4: return launch_g<4, 2>(plan, args, stream, pdl);
    case kDownW4: return launch_g<4, 1>(plan, args, stream, pdl);
    case kGateUpW3: return launch_g<3, 2>(plan, args, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemv_slots(GemvKind kind, const GemvPlan &plan, const GemvArgs &args, int slots,
                              cudaStream_t stream, bool pdl) {
  if (plan.r != args.r || args.slot_expert == nullptr || slots <= 0 || slots > 65535) return cudaErrorInvalidValue;
  switch (kind) {
    case kGateUpW2: return launch_slots_g<2, 2>(plan, args, slots, stream, pdl);
    case kGateUpW4: return launch_slots_g<4, 2>(plan, args, slots, stream, pdl);
    case kDownW4: return launch_slots_g<4, 1>(plan, args, slots, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_tile_prep(const void *x, int M, int d, const void *lora_a, int r2, float *tp, cudaStream_t stream,
                             bool pdl) {
  const int ntp = d / 16;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((ntp + 7) / 8);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const size_t nb_x = (size_t)M * d * 2, nb_a = (size_t)r2 * d * 2, nb_tp = (size_t)ntp * M * ((1 + r2 + 3) & ~3) * 4;
  return cudaLaunchKernelEx(&cfg, tile_prep_kernel, reinterpret_cast<const __nv_bfloat16 *>(x), M, d,
                            reinterpret_cast<const __nv_bfloat16 *>(lora_a), r2, tp, nb_x, nb_a, nb_tp);
}

cudaError_t read_debug_record(long long rec[4]) {
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(rec, g_debug_record, 4 * sizeof(long long));
  if (e != cudaSuccess) return e;
  const long long zero[4] = {0, 0, 0, 0};
  return cudaMemcpyToSymbol(g_debug_record, zero, sizeof zero);
}

cudaError_t read_device_status(int *status) {
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(status, g_device_status, sizeof(int));
  if (e != cudaSuccess) return e;
  const int zero = 0;
  return cudaMemcpyToSymbol(g_device_status, &zero, sizeof(int));
}

}  // namespace wq
