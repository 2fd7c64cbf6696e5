// wq_gemv.cu -- decode-regime dequant-GEMV kernels (sm_103a).
//
// One templated kernel serves the three matrix products of the gated MLP
// with W4/W2-GateUp weights (Sec. 3.3):
//   * gate+up, 2-bit codes, unmerged LoRA (Eq. 1) and SiLU(gate)*up fused
//     into the epilogue, so the intermediate g/u never leave the chip
//     (Sec. 5 models the MLP operators as one fused kernel);
//   * gate+up, 4-bit codes (the uniform-W4 comparator);
//   * down, 4-bit codes, residual add fused into the epilogue.
//
// Data path of one CTA (one row block x one feature panel):
//   1. one thread issues bulk (TMA) copies of the packed codes and binary16
//      scales/zeros of its row tiles into shared memory -- before waiting on
//      the previous kernel (programmatic dependent launch), so the weight
//      stream of this kernel overlaps the tail of the previous one;
//   2. after griddepcontrol.wait, each token's activation panel is loaded
//      (plain 16-byte loads) and converted in place to binary16 with an exact
//      power-of-two scale per token (and per code position class, see below),
//      and per-group activation sums are formed;
//   3. each warp owns one 16-row tile and a share of the panel: a 16-byte
//      shared load per lane yields the tensor-core A fragments of 64 (2-bit)
//      or 32 (4-bit) codes; codes are isolated with a single AND each -- the
//      isolated bits read as a binary16 subnormal code * 4^c * 2^-24, the
//      4^c (c = bit-position class) being cancelled by the activation's
//      class scale -- and fed to mma.sync m16n8k16 (fp32 accumulation);
//   4. per group: acc += s * (sum_k code*x - z * sum_k x), i.e. the affine
//      dequantization s(q - z) is applied once per group, not per weight;
//   5. warps' partial sums are reduced in shared memory in a fixed order;
//      with several panels the last-arriving CTA of a row tile adds the
//      panel partials in panel order (deterministic), then the epilogue
//      (LoRA-B expansion, SiLU(g)*u, or residual add) stores the outputs.
#include <algorithm>
#include <climits>
#include <cmath>

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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ uint32_t pack_half2(float a, float b) {
  const __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<const uint32_t *>(&h);
}

__device__ __forceinline__ float half_bits_to_float(uint32_t bits16) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(bits16 & 0xffffu)));
}

// ---------------------------------------------------------------------------
// The dequant-GEMV kernel.
//   BITS  2 or 4 (code width), NPROJ 2 (gate+up) or 1 (down),
//   GROUP 32/64/128 (quantization group), NT 1 or 2 (8-token MMA tiles per
//   token chunk: chunks of 8 tokens for m <= 8, of 16 otherwise).
// ---------------------------------------------------------------------------
template <int BITS, int NPROJ, int GROUP, int NT>
__global__ void __launch_bounds__(NT == 1 ? 1024 : 512) qgemv_kernel(const GemvArgs a, const GemvPlan p) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int BPK = BITS == 2 ? 512 : 1024;  // code bytes per (row tile, 128-feature block)
  constexpr int GPB = 128 / GROUP;             // groups per block
  constexpr int GS = GROUP / 16;               // k-steps (16 features) per group
  constexpr int TOK = 8 * NT;                  // tokens per chunk

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rb = blockIdx.x / p.P, panel = blockIdx.x % p.P;
  const int rt0 = rb * p.RB;
  const int nrt = min(p.RB, p.RT - rt0);
  const int kb0 = panel * p.KP;
  const int nkb = min(p.KP, p.KB - kb0);
  const int NG = p.KB * GPB;
  const int M = a.M, MPAD = p.MPAD;

  uint8_t *codes_s = smem + p.off_codes;
  uint8_t *meta_s = smem + p.off_meta;
  __half *xp_s = reinterpret_cast<__half *>(smem + p.off_xp);
  float *xs_s = reinterpret_cast<float *>(smem + p.off_xs);
  float *scale_s = reinterpret_cast<float *>(smem + p.off_scale);
  float *slot_s = reinterpret_cast<float *>(smem + p.off_slots);
  float *t_s = reinterpret_cast<float *>(smem + p.off_t);
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + p.off_bar);
  int *last_s = reinterpret_cast<int *>(smem + p.off_last);

  // ---- 1. weight prefetch (independent of the previous kernel) ----
  // Warp (rw, wk) owns row tile rw and blocks [kbs, kbe) of the panel; its
  // lane 0 bulk-copies exactly that slice (both projections) on its own
  // barrier, so each warp starts as soon as its own weights have landed.
  const int rw = warp % p.RB, wk = warp / p.RB;
  const int kbs = wk * nkb / p.WK, kbe = (wk + 1) * nkb / p.WK;
  const bool has_slice = rw < nrt && kbe > kbs;
  if (lane == 0 && has_slice) {
    uint64_t *bar = &bars[warp];
    mbar_init(bar, 1);
    fence_barrier_init();
    const int rt = rt0 + rw, nb = kbe - kbs;
    mbar_arrive_expect_tx(bar, NPROJ * nb * (BPK + GPB * 64));
#pragma unroll
    for (int pj = 0; pj < NPROJ; ++pj) {
      const size_t cd = p.off_codes + ((size_t)(pj * p.RB + rw) * p.KP + kbs) * BPK;
      const size_t cs = ((size_t)rt * p.KB + kb0 + kbs) * BPK;
      if (WQ_OK_IF(WQ_RANGE(cd, nb * BPK, p.off_meta, 16), 1, cd) &&
          WQ_OK_IF(WQ_RANGE(cs, nb * BPK, a.nb_codes[pj], 16), 2, cs))
        bulk_g2s(smem + cd, reinterpret_cast<const uint8_t *>(a.codes[pj]) + cs, nb * BPK, bar);
      const size_t md = p.off_meta + ((size_t)(pj * p.RB + rw) * p.KP * GPB + (size_t)kbs * GPB) * 64;
      const size_t ms = ((size_t)rt * NG + (size_t)(kb0 + kbs) * GPB) * 64;
      if (WQ_OK_IF(WQ_RANGE(md, nb * GPB * 64, p.off_lorab, 16), 3, md) &&
          WQ_OK_IF(WQ_RANGE(ms, nb * GPB * 64, a.nb_meta[pj], 16), 4, ms))
        bulk_g2s(smem + md, reinterpret_cast<const uint8_t *>(a.meta[pj]) + ms, nb * GPB * 64, bar);
    }
  }
  int *tokmax_s = reinterpret_cast<int *>(scale_s + MPAD);
  for (int i = tid; i < nkb * GPB * MPAD; i += blockDim.x) xs_s[i] = 0.f;
  for (int i = tid; i < MPAD; i += blockDim.x) {
    scale_s[i] = 0.f;
    tokmax_s[i] = 0;
  }
  __syncthreads();  // barrier initialisation visible before any thread waits on it

  pdl_launch_dependents();
  pdl_wait();  // activations (and LoRA-A products) of the previous kernel are ready

  // ---- 2. activation panel -> binary16 with per-token power-of-two scale ----
  const int kbeg = kb0 * 128;
  const int kvalid = min(nkb * 128, a.K - kbeg);  // a multiple of 8
  // Activations are staged with ordinary loads, not a bulk copy: the panel is
  // converted in place below, and shared memory filled by the async (bulk
  // copy) proxy is only ever read afterwards in this kernel.
  {
    const __nv_bfloat16 *act = reinterpret_cast<const __nv_bfloat16 *>(a.act);
    const int nch = kvalid / 8;  // 16-byte chunks per token row
    for (int i = tid; i < M * nch; i += blockDim.x) {
      const int m = i / nch, c = i % nch;
      const size_t src = ((size_t)m * a.K + kbeg + (size_t)c * 8) * 2;
      if (WQ_OK_IF(WQ_RANGE(src, 16, a.nb_act, 16), 8, src) &&
          WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)m * p.xstride + c * 8) * 2, 16, p.off_xs, 16), 7, i))
        *reinterpret_cast<uint4 *>(xp_s + (size_t)m * p.xstride + c * 8) = ldg_cg128(act + (size_t)m * a.K + kbeg + c * 8);
    }
  }
  if (NPROJ == 2 && a.r > 0) {
    for (int i = tid; i < M * 2 * a.r; i += blockDim.x)
      if (WQ_OK_IF(WQ_RANGE((size_t)i * 4, 4, a.nb_t, 4), 9, i) &&
          WQ_OK_IF(WQ_RANGE(p.off_t + (size_t)i * 4, 4, p.off_bar, 4), 10, i))
        t_s[i] = ldcg_f32(a.t + i);
  }
  __syncthreads();
  {
    // Work item = 16 features of one token (one MMA k-step).  Pass 1: per
    // token max|x|.  Pass 2: in place, bf16 -> scaled binary16 in the order
    // the B fragments read it, plus per-group sums of x.
    const int nsteps = nkb * 8;
    const int total = M * nsteps;
    for (int i = tid; i < total; i += blockDim.x) {
      const int m = i / nsteps, st = i % nsteps;
      if (st * 16 < kvalid &&
          WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)m * p.xstride + st * 16) * 2, 32, p.off_xs, 16), 11, i)) {
        const __nv_bfloat16 *src = reinterpret_cast<const __nv_bfloat16 *>(xp_s + (size_t)m * p.xstride + st * 16);
        float f[16];
        unpack_bf16x8(lds128(src), *reinterpret_cast<float(*)[8]>(f));
        unpack_bf16x8(lds128(src + 8), *reinterpret_cast<float(*)[8]>(f + 8));
        const int nv = min(16, kvalid - st * 16);
        float mx = 0.f;
#pragma unroll
        for (int e = 0; e < 16; ++e)
          if (e < nv) mx = fmaxf(mx, fabsf(f[e]));
        if (WQ_OK_IF(m < MPAD, 12, m)) atomicMax(&tokmax_s[m], __float_as_int(mx));
      }
    }
    __syncthreads();
    constexpr int LG = GROUP / 16;  // lanes (work items) per group
    for (int base = warp * 32; base < total; base += blockDim.x) {
      const int i = base + lane;
      const bool valid = i < total;
      const int m = valid ? i / nsteps : 0, st = valid ? i % nsteps : 0;
      float f[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) f[e] = 0.f;
      __half *slot = xp_s + (size_t)m * p.xstride + st * 16;
      const bool slot_ok = !valid || WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)m * p.xstride + st * 16) * 2, 32,
                                                       p.off_xs, 16), 13, i);
      if (valid && slot_ok && st * 16 < kvalid) {
        const __nv_bfloat16 *src = reinterpret_cast<const __nv_bfloat16 *>(slot);
        unpack_bf16x8(lds128(src), *reinterpret_cast<float(*)[8]>(f));
        unpack_bf16x8(lds128(src + 8), *reinterpret_cast<float(*)[8]>(f + 8));
        if (st * 16 + 8 > kvalid) {
#pragma unroll
          for (int e = 8; e < 16; ++e) f[e] = 0.f;
        }
      }
      float gs = 0.f;
#pragma unroll
      for (int e = 0; e < 16; ++e) gs += f[e];
      // scale 2^e puts max|x| in [2^14, 2^15): binary16 holds every scaled
      // value exactly (bf16 has 8 significant bits), far from overflow.
      const float mx = __int_as_float(valid ? tokmax_s[m] : 0);
      int e = 0;
      if (mx > 0.f && mx <= 3.4e38f) {
        int E;
        frexpf(mx, &E);
        e = max(-100, min(100, 15 - E));
      }
      if (valid && slot_ok) {
        const float up = ldexpf(1.f, e);
        if (st == 0) scale_s[m] = ldexpf(1.f, 24 - e);
        // bit-position class of the codes feeding features 0-7 / 8-15 of this step
        const int sh_lo = BITS == 2 ? 4 * (st & 1) : 0;
        const int sh_hi = BITS == 2 ? sh_lo + 2 : 4;
        const float mul_lo = up * ldexpf(1.f, -sh_lo), mul_hi = up * ldexpf(1.f, -sh_hi);
        uint32_t w[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          w[2 * j] = pack_half2(f[2 * j] * mul_lo, f[2 * j + 1] * mul_lo);
          w[2 * j + 1] = pack_half2(f[8 + 2 * j] * mul_hi, f[9 + 2 * j] * mul_hi);
        }
        uint4 *dst = reinterpret_cast<uint4 *>(slot);
        dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
        dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
      }
#pragma unroll
      for (int o = 1; o < LG; o <<= 1) gs += __shfl_xor_sync(0xffffffffu, gs, o);
      if (valid && (lane % LG) == 0 &&
          WQ_OK_IF(WQ_RANGE(p.off_xs + ((size_t)(st / LG) * MPAD + m) * 4, 4, p.off_scale, 4), 14, i))
        xs_s[(st / LG) * MPAD + m] = gs * ldexpf(1.f, e - 24);
    }
  }
  __syncthreads();

  // ---- 3./4. tensor-core dot products ----
  if (rw < nrt) {
    const bool ok = !has_slice || mbar_wait(&bars[warp], 0);
    if (!ok && lane == 0) record_timeout();
    const uint8_t *cbase = codes_s + (size_t)(rw * p.KP) * BPK + lane * 16;
    const uint8_t *mbase = meta_s + (size_t)(rw * p.KP * GPB) * 64 + (lane >> 2) * 8;
    const size_t cproj = (size_t)p.RB * p.KP * BPK;
    const size_t mproj = (size_t)p.RB * p.KP * GPB * 64;
    for (int tc = 0; tc * TOK < M; ++tc) {
      float ctot[NPROJ][NT][4];
#pragma unroll
      for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int q = 0; q < 4; ++q) ctot[pj][nt][q] = 0.f;
      for (int kb = ok ? kbs : kbe; kb < kbe; ++kb) {
        uint32_t b[8][NT][2];
#pragma unroll
        for (int ks = 0; ks < 8; ++ks)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int m = tc * TOK + nt * 8 + (lane >> 2);
            if (m < M && WQ_OK_IF(WQ_RANGE(p.off_xp + ((size_t)m * p.xstride + (kb * 8 + ks) * 16 + 4 * (lane & 3)) * 2,
                                           8, p.off_xs, 8), 15, kb)) {
              const uint2 v = lds64(xp_s + (size_t)m * p.xstride + (kb * 8 + ks) * 16 + 4 * (lane & 3));
              b[ks][nt][0] = v.x;
              b[ks][nt][1] = v.y;
            } else {
              b[ks][nt][0] = 0u;
              b[ks][nt][1] = 0u;
            }
          }
#pragma unroll
        for (int pj = 0; pj < NPROJ; ++pj) {
          const uint8_t *cb = cbase + pj * cproj + (size_t)kb * BPK;
          uint32_t wds[BITS == 2 ? 4 : 8];
          wds[0] = wds[1] = wds[2] = wds[3] = 0u;
          if (BITS == 4) wds[BITS == 4 ? 4 : 0] = wds[BITS == 4 ? 5 : 1] = wds[BITS == 4 ? 6 : 2] = wds[BITS == 4 ? 7 : 3] = 0u;
          if (WQ_OK_IF(WQ_RANGE(cb - smem, BPK == 512 ? 16 : 528, p.off_meta, 16), 16, kb)) {
            const uint4 w0 = lds128(cb);
            wds[0] = w0.x; wds[1] = w0.y; wds[2] = w0.z; wds[3] = w0.w;
            if (BITS == 4) {
              const uint4 w1 = lds128(cb + 512);
              wds[BITS == 4 ? 4 : 0] = w1.x; wds[BITS == 4 ? 5 : 1] = w1.y;
              wds[BITS == 4 ? 6 : 2] = w1.z; wds[BITS == 4 ? 7 : 3] = w1.w;
            }
          }
          // two independent accumulator chains (even / odd k-steps) per group
          float cg[NT][4], ch[NT][4];
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int q = 0; q < 4; ++q) cg[nt][q] = ch[nt][q] = 0.f;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            uint32_t af[4];
            if (BITS == 2) {
              const uint32_t x = wds[(ks >> 1) & 3];
              const uint32_t x8 = x >> 8;
              const int s4 = (ks & 1) * 4;
              af[0] = x & (0x00030003u << s4);   // rows g,   features 2t..2t+1
              af[1] = x8 & (0x00030003u << s4);  // rows g+8
              af[2] = x & (0x000C000Cu << s4);   // rows g,   features 2t+8..2t+9
              af[3] = x8 & (0x000C000Cu << s4);  // rows g+8
            } else {
              const uint32_t x = wds[ks & (BITS == 2 ? 3 : 7)];
              const uint32_t x8 = x >> 8;
              af[0] = x & 0x000F000Fu;
              af[1] = x8 & 0x000F000Fu;
              af[2] = x & 0x00F000F0u;
              af[3] = x8 & 0x00F000F0u;
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              if (ks & 1)
                mma_f16_16816(ch[nt], af, b[ks][nt][0], b[ks][nt][1]);
              else
                mma_f16_16816(cg[nt], af, b[ks][nt][0], b[ks][nt][1]);
            }
            if ((ks + 1) % GS == 0) {
              const int gl = kb * GPB + ks / GS;
              uint2 mt = make_uint2(0u, 0u);
              if (WQ_OK_IF(WQ_RANGE(mbase + pj * mproj + (size_t)gl * 64 - smem, 8, p.off_lorab, 8), 17, gl))
                mt = lds64(mbase + pj * mproj + (size_t)gl * 64);
              const float s_lo = half_bits_to_float(mt.x), s_hi = half_bits_to_float(mt.x >> 16);
              const float z_lo = half_bits_to_float(mt.y), z_hi = half_bits_to_float(mt.y >> 16);
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                const int col = tc * TOK + nt * 8 + 2 * (lane & 3);
                float2 xs = make_float2(0.f, 0.f);
                if (WQ_OK_IF(WQ_RANGE(p.off_xs + ((size_t)gl * MPAD + col) * 4, 8, p.off_scale, 8), 18, col))
                  xs = *reinterpret_cast<const float2 *>(xs_s + gl * MPAD + col);
                ctot[pj][nt][0] = fmaf(s_lo, fmaf(-z_lo, xs.x, cg[nt][0] + ch[nt][0]), ctot[pj][nt][0]);
                ctot[pj][nt][1] = fmaf(s_lo, fmaf(-z_lo, xs.y, cg[nt][1] + ch[nt][1]), ctot[pj][nt][1]);
                ctot[pj][nt][2] = fmaf(s_hi, fmaf(-z_hi, xs.x, cg[nt][2] + ch[nt][2]), ctot[pj][nt][2]);
                ctot[pj][nt][3] = fmaf(s_hi, fmaf(-z_hi, xs.y, cg[nt][3] + ch[nt][3]), ctot[pj][nt][3]);
#pragma unroll
                for (int q = 0; q < 4; ++q) cg[nt][q] = ch[nt][q] = 0.f;
              }
            }
          }
        }
      }
      // per-warp partial -> shared slot [wk][rw][pj][16][MPAD]
#pragma unroll
      for (int pj = 0; pj < NPROJ; ++pj)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const int col = tc * TOK + nt * 8 + 2 * (lane & 3), r0 = lane >> 2;
          float *sl = slot_s + (size_t)((wk * p.RB + rw) * NPROJ + pj) * 16 * MPAD;
          if (!WQ_OK_IF(WQ_RANGE((uint8_t *)(sl + (r0 + 8) * MPAD + col) - smem, 8, p.off_t, 4), 19, col)) continue;
          sl[r0 * MPAD + col] = ctot[pj][nt][0];
          sl[r0 * MPAD + col + 1] = ctot[pj][nt][1];
          sl[(r0 + 8) * MPAD + col] = ctot[pj][nt][2];
          sl[(r0 + 8) * MPAD + col + 1] = ctot[pj][nt][3];
        }
    }
  }
  __syncthreads();

  // ---- 5. reduce the k-split warps (fixed order) and undo the token scale ----
  const int per_rt = NPROJ * 16 * MPAD;
  for (int i = tid; i < nrt * per_rt; i += blockDim.x) {
    float s = 0.f;
    for (int w = 0; w < p.WK; ++w)
      if (WQ_OK_IF(WQ_RANGE(p.off_slots + ((size_t)w * p.RB * per_rt + i) * 4, 4, p.off_t, 4), 20, i))
        s += slot_s[(size_t)w * p.RB * per_rt + i];
    const int m = i % MPAD;
    slot_s[i] = m < M ? s * scale_s[m] : 0.f;
  }
  __syncthreads();

  if (p.P > 1) {
    for (int i = tid; i < nrt * per_rt; i += blockDim.x) {
      const int rti = i / per_rt, rem = i % per_rt;
      const size_t po = ((size_t)(rt0 + rti) * p.P + panel) * per_rt + rem;
      if (WQ_OK_IF(WQ_RANGE(po * 4, 4, a.nb_part, 4), 21, po)) a.partials[po] = slot_s[i];
    }
    __threadfence();
    __syncthreads();
    if (tid < nrt && WQ_OK_IF(WQ_RANGE((size_t)(rt0 + tid) * 4, 4, a.nb_cnt, 4), 22, rt0 + tid)) {
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
      for (int pp = 0; pp < p.P; ++pp)
        if (WQ_OK_IF(WQ_RANGE((src - a.partials + (size_t)pp * per_rt) * 4, 4, a.nb_part, 4), 23, pp))
          s += ldcg_f32(src + (size_t)pp * per_rt);
      slot_s[i] = s;
    }
    if (tid < nrt && last_s[tid]) a.counters[rt0 + tid] = 0u;
    __syncthreads();
  } else {
    if (tid < nrt) last_s[tid] = 1;
    __syncthreads();
  }

  // ---- epilogue: LoRA-B + SiLU(g) * u, or residual add ----
  const int rows = nrt * 16;
  for (int i = tid; i < rows * M; i += blockDim.x) {
    const int m = i / rows, rl = i % rows;
    const int rti = rl >> 4, r16 = rl & 15;
    if (!last_s[rti]) continue;
    const int n = (rt0 + rti) * 16 + r16;
    if (n >= a.N) continue;
    const float v0 = slot_s[(size_t)(rti * NPROJ) * 16 * MPAD + r16 * MPAD + m];
    if (NPROJ == 2) {
      float g = v0;
      float u = slot_s[(size_t)(rti * NPROJ + 1) * 16 * MPAD + r16 * MPAD + m];
      if (a.r > 0) {
        const int r = a.r;
        const __nv_bfloat16 *bg = reinterpret_cast<const __nv_bfloat16 *>(a.lora_b[0]) + (size_t)n * r;
        const __nv_bfloat16 *bu = reinterpret_cast<const __nv_bfloat16 *>(a.lora_b[1]) + (size_t)n * r;
        const float *tg = t_s + (size_t)m * 2 * r;
        const float *tu = tg + r;
        float lg = 0.f, lu = 0.f;
        const bool lora_ok =
            WQ_OK_IF(WQ_RANGE(((size_t)m * 2 * r + 2 * r) * 4 + p.off_t - 4, 4, p.off_bar, 4), 24, m) &&
            WQ_OK_IF(WQ_RANGE(((size_t)n * r + r) * 2 - 16, 16, a.nb_lora_b[1], 16), 26, n);
        for (int q = 0; lora_ok && q < r; q += 8) {
          float fg[8], fu[8];
          unpack_bf16x8(__ldg(reinterpret_cast<const uint4 *>(bg + q)), fg);
          unpack_bf16x8(__ldg(reinterpret_cast<const uint4 *>(bu + q)), fu);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            lg = fmaf(tg[q + e], fg[e], lg);
            lu = fmaf(tu[q + e], fu[e], lu);
          }
        }
        g = fmaf(a.lora_scale, lg, g);
        u = fmaf(a.lora_scale, lu, u);
      }
      const float h = g / (1.f + __expf(-g)) * u;
      if (WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * 2, 2, a.nb_out, 2), 27, n))
        reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = __float2bfloat16_rn(h);
    } else {
      float y = v0;
      if (!WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * (a.out_f32 ? 4 : 2), a.out_f32 ? 4 : 2, a.nb_out, 2), 28, n))
        continue;
      if (a.residual && WQ_OK_IF(WQ_RANGE(((size_t)m * a.N + n) * 2, 2, a.nb_res, 2), 29, n))
        y += __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(a.residual)[(size_t)m * a.N + n]);
      if (a.out_f32)
        reinterpret_cast<float *>(a.out)[(size_t)m * a.N + n] = y;
      else
        reinterpret_cast<__nv_bfloat16 *>(a.out)[(size_t)m * a.N + n] = __float2bfloat16_rn(y);
    }
  }
}

// ---------------------------------------------------------------------------
// Prologue kernel: unit-weight RMSNorm of the MLP input (rounded to bf16,
// written by CTA 0) and the LoRA-A products t[m, rho] = xin[m] . A[rho]
// (CTA rho).  Every CTA computes the norm scale of each token with the same
// fixed-order reduction, so all CTAs see bit-identical xin.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) prep_kernel(const __nv_bfloat16 *x, int M, int d,
                                                    const __nv_bfloat16 *lora_a, int r2, int prenorm,
                                                    __nv_bfloat16 *xhat, float *t, uint32_t smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const uint32_t arow_bytes = ((uint32_t)d * 2 + 127u) & ~127u;
  __nv_bfloat16 *arow = reinterpret_cast<__nv_bfloat16 *>(smem);
  float *rs_s = reinterpret_cast<float *>(smem + arow_bytes);   // [kMaxTokens]
  float *red_s = rs_s + kMaxTokens;                              // [32]
  const int rho = blockIdx.x;
  const bool lora = r2 > 0;

  if (lora && WQ_OK_IF(rho < r2 && (d * 2) % 16 == 0, 41, rho)) {
    // the LoRA-A row does not depend on the previous kernel: load it first
    for (int c = tid; c < d / 8; c += blockDim.x)
      *reinterpret_cast<uint4 *>(arow + c * 8) = __ldg(reinterpret_cast<const uint4 *>(lora_a + (size_t)rho * d) + c);
  }
  (void)smem_bytes;
  pdl_launch_dependents();
  pdl_wait();

  const int nch = d / 8;
  for (int m = warp; m < M; m += nwarps) {
    float rs = 1.f;
    if (prenorm) {
      float ss = 0.f;
      for (int c = lane; c < nch; c += 32) {
        float f[8];
        unpack_bf16x8(ldg_cg128(x + (size_t)m * d + c * 8), f);
#pragma unroll
        for (int e = 0; e < 8; ++e) ss = fmaf(f[e], f[e], ss);
      }
      ss = warp_sum(ss);
      rs = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)d), kRmsEps)));
    }
    if (lane == 0 && WQ_OK_IF(m < kMaxTokens, 42, m)) rs_s[m] = rs;
  }
  __syncthreads();

  if (lora) {
    for (int m = 0; m < M; ++m) {
      const float rs = rs_s[m];
      float acc = 0.f;
      for (int c = tid; c < nch; c += blockDim.x) {
        float f[8], av[8];
        unpack_bf16x8(ldg_cg128(x + (size_t)m * d + c * 8), f);
        unpack_bf16x8(*reinterpret_cast<const uint4 *>(arow + c * 8), av);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float xv = prenorm ? __bfloat162float(__float2bfloat16_rn(__fmul_rn(f[e], rs))) : f[e];
          acc = fmaf(xv, av[e], acc);
        }
      }
      acc = warp_sum(acc);
      if (lane == 0) red_s[warp] = acc;
      __syncthreads();
      if (tid == 0) {
        float s = 0.f;
        for (int w = 0; w < nwarps; ++w) s += red_s[w];
        if (WQ_OK_IF((size_t)m * r2 + rho < (size_t)M * r2, 43, m)) t[(size_t)m * r2 + rho] = s;
      }
      __syncthreads();
    }
  }

  if (prenorm && blockIdx.x == 0) {
    for (int i = tid; i < M * nch; i += blockDim.x) {
      const int m = i / nch, c = i % nch;
      float f[8];
      unpack_bf16x8(ldg_cg128(x + (size_t)m * d + c * 8), f);
      const float rs = rs_s[m];
      uint32_t o[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const __nv_bfloat162 h2 = __floats2bfloat162_rn(__fmul_rn(f[2 * j], rs), __fmul_rn(f[2 * j + 1], rs));
        o[j] = *reinterpret_cast<const uint32_t *>(&h2);
      }
      *reinterpret_cast<uint4 *>(xhat + (size_t)m * d + c * 8) = make_uint4(o[0], o[1], o[2], o[3]);
    }
  }
}

// ---------------------------------------------------------------------------
// Host side: planning and launching.
// ---------------------------------------------------------------------------
uint32_t align_up(uint32_t v, uint32_t a) { return (v + a - 1) / a * a; }

int kind_bits(GemvKind k) { return k == kGateUpW2 ? 2 : 4; }
int kind_nproj(GemvKind k) { return k == kDownW4 ? 1 : 2; }

void compute_layout(GemvKind kind, int group, int r, GemvPlan *p) {
  const int nproj = kind_nproj(kind);
  const int BPK = kind_bits(kind) == 2 ? 512 : 1024, GPB = 128 / group;
  uint32_t off = 0;
  p->off_codes = off;
  off = align_up(off + (uint32_t)nproj * p->RB * p->KP * BPK, 128);
  p->off_meta = off;
  off = align_up(off + (uint32_t)nproj * p->RB * p->KP * GPB * 64, 128);
  p->off_lorab = off;
  if (p->lora_smem) off = align_up(off + (uint32_t)nproj * p->RB * 16 * r * 2, 128);
  p->xstride = p->KP * 128 + 16;  // row bytes = 256 KP + 32: conflict-free 8-byte fragment loads
  p->off_xp = off;
  off = align_up(off + (uint32_t)p->M * p->xstride * 2, 128);
  p->off_xs = off;
  off = align_up(off + (uint32_t)p->KP * GPB * p->MPAD * 4, 128);
  p->off_scale = off;  // token scales, then token max|x| bits
  off = align_up(off + (uint32_t)p->MPAD * 8, 128);
  p->off_slots = off;
  off = align_up(off + (uint32_t)p->WK * p->RB * nproj * 16 * p->MPAD * 4, 128);
  p->off_t = off;
  off = align_up(off + (nproj == 2 ? (uint32_t)p->M * 2 * r * 4 : 0u), 128);
  p->off_bar = off;  // one weight barrier per warp
  off = align_up(off + (uint32_t)p->RB * p->WK * 8, 128);
  p->off_last = off;
  off = align_up(off + (uint32_t)p->RB * 4, 128);
  p->smem = off;
}

}  // namespace

constexpr uint32_t kSmemLimit = 232448;  // 227 KB opt-in dynamic shared memory per CTA

bool plan_gemv(GemvKind kind, int N, int K, int M, int group, int r, int num_sms, GemvPlan *out) {
  if (N <= 0 || K <= 0 || M <= 0 || M > kMaxTokens || num_sms <= 0) return false;
  const int nproj = kind_nproj(kind);
  const int RT = (N + 15) / 16, KB = (K + 127) / 128;
  const int NT = M <= 8 ? 1 : 2;
  const int tok = 8 * NT;
  const int MPAD = (M + tok - 1) / tok * tok;
  const int chunks = MPAD / tok;
  bool found = false;
  double best = 1e300;
  GemvPlan bp{};
  for (int KP = 1; KP <= KB; ++KP) {
    const int P = (KB + KP - 1) / KP;
    if ((KB + P - 1) / P != KP) continue;  // one canonical KP per panel count
    for (int RB = 1; RB <= std::min(RT, kMaxWarps); ++RB) {
      for (int WK = 1; WK <= 8; WK *= 2) {
        if (WK > KP || RB * WK > (NT == 1 ? kMaxWarps : kMaxWarps / 2)) continue;
        GemvPlan p{};
        p.RT = RT; p.KB = KB; p.RB = RB; p.KP = KP; p.WK = WK; p.P = P;
        p.NRB = (RT + RB - 1) / RB;
        p.M = M; p.MPAD = MPAD; p.NT = NT;
        p.threads = RB * WK * 32;
        p.units = p.NRB * P;
        p.lora_smem = 0;
        compute_layout(kind, group, r, &p);
        if (p.smem > kSmemLimit) continue;
        const int occ = std::max(1, std::min({(int)(233472 / (p.smem + 1024)), 2048 / p.threads, 32}));
        const int per_sm = (p.units + num_sms - 1) / num_sms;           // units landing on the busiest SM
        const int waves = (p.units + num_sms * occ - 1) / (num_sms * occ);
        // Cycle estimates: a tile-projection (16 rows x 128 features of one
        // matrix) costs ~45 issue slots, spread over the SM's 4 schedulers;
        // one warp's chain of tile-projections costs ~120 cycles each of MMA
        // and shared-memory latency; each CTA wave adds a fixed prologue /
        // epilogue latency, and a split-panel fixup an L2 round trip.
        const double tiles = (double)per_sm * RB * KP * nproj * chunks;
        const double thr = tiles * 45.0 / 4.0;
        const double lat = (double)((KP + WK - 1) / WK) * nproj * chunks * 120.0 * waves;
        // the busiest SM's share of the weight stream at ~22 B/cycle (HBM / SMs)
        const double mem = (double)per_sm * RB * KP * nproj * (kind_bits(kind) == 2 ? 640.0 : 1088.0) / 22.0;
        // the weight stream (or the issue rate) bounds the bulk; the last
        // warp's dependent chain after its slice lands is added as a tail
        double cost = std::max(thr, mem) + lat + 800.0 * waves + (P > 1 ? 1500.0 : 0.0);
        cost += (p.smem > 113 * 1024 ? 300.0 : 0.0);  // no room to overlap the next kernel's prologue
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

template <int BITS, int NPROJ, int GROUP, int NT>
cudaError_t launch_t(const GemvPlan &p, const GemvArgs &a, cudaStream_t s, bool pdl) {
  auto kern = qgemv_kernel<BITS, NPROJ, GROUP, NT>;
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

template <int BITS, int NPROJ>
cudaError_t launch_g(const GemvPlan &p, const GemvArgs &a, cudaStream_t s, bool pdl) {
  const bool two = p.NT == 2;
  switch (a.group) {
    case 32: return two ? launch_t<BITS, NPROJ, 32, 2>(p, a, s, pdl) : launch_t<BITS, NPROJ, 32, 1>(p, a, s, pdl);
    case 64: return two ? launch_t<BITS, NPROJ, 64, 2>(p, a, s, pdl) : launch_t<BITS, NPROJ, 64, 1>(p, a, s, pdl);
    case 128: return two ? launch_t<BITS, NPROJ, 128, 2>(p, a, s, pdl) : launch_t<BITS, NPROJ, 128, 1>(p, a, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemv(GemvKind kind, const GemvPlan &plan, const GemvArgs &args, cudaStream_t stream, bool pdl) {
  switch (kind) {
    case kGateUpW2: return launch_g<2, 2>(plan, args, stream, pdl);
    case kGateUpW4: return launch_g<4, 2>(plan, args, stream, pdl);
    case kDownW4: return launch_g<4, 1>(plan, args, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_prep(const void *x, int M, int d, const void *lora_a, int r, int prenorm, void *xhat, float *t,
                        cudaStream_t stream, bool pdl) {
  const uint32_t smem = (((uint32_t)d * 2 + 127u) & ~127u) + (kMaxTokens + 32) * 4 + 16;
  cudaError_t e = cudaFuncSetAttribute(prep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(r > 0 ? 2 * r : 1);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, prep_kernel, reinterpret_cast<const __nv_bfloat16 *>(x), M, d,
                            reinterpret_cast<const __nv_bfloat16 *>(lora_a), 2 * r, prenorm,
                            reinterpret_cast<__nv_bfloat16 *>(xhat), t, smem);
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
