// wq_stack.cu -- the whole decode MLP stack (Sec. 3.3 gated MLP with
// W4/W2-GateUp weights and the unmerged adapters of Eq. 1, layer after layer)
// as ONE persistent launch on sm_103a.
//
// A launch chain pays, per layer, two kernel boundaries and runs the 4-bit
// down projection on 160 row tiles over 152 SMs.  Here one CTA per SM stays
// resident for the whole stack:
//
//   * one warp streams every layer's packed weights, in the order the math
//     consumes them, into a ring of shared-memory stages (1-D bulk copies,
//     one mbarrier pair per stage).  Weights do not depend on activations, so
//     the stream runs ahead of the math by the ring's size (about one layer
//     of the Qwen3-4B shape) and is never held up by a layer boundary;
//   * 16 warps do the math of each layer in three phases:
//       gate/up: the CTA's 16-row tiles of gate and up over all d features
//                (exact code x binary16 products on mma.sync, fp32 sums per
//                group, as the decode GEMV kernels), LoRA-B, RMSNorm scale,
//                SiLU(g) * u -> h (bf16);
//       down:    a K-slice of the down projection: 64-feature half blocks of
//                h times ALL d rows, so that on layer shapes whose gate/up
//                rows and down slices coincide (e.g. d 2560, inter 9728 on
//                152 SMs) each CTA multiplies its own h and waits for no
//                other CTA; the fp32 partial sums of y go to global memory;
//       owner:   after a grid barrier, each CTA adds up the partial sums of
//                its 16-row tiles of y over the half blocks in a fixed order
//                (deterministic), adds the residual, stores y in bf16 and the
//                next layer's per-tile RMSNorm / LoRA-A partial sums; a
//                second grid barrier opens the next layer;
//   * grid barriers are one 64-bit arrival counter in the workspace (measured
//     on GB300: ~1.2 us a barrier over 152 CTAs; per-CTA flags polled by every
//     CTA were ~3x slower); every wait is bounded and a timeout records
//     WQ_ERR_TIMEOUT and lets the launch run to its end.
//
// Layer shapes whose down K-slices do not coincide with the CTA's gate/up
// rows add a third barrier per layer before the down phase (h read back from
// global memory).
#include <algorithm>
#include <climits>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>

#include <cudaTypedefs.h>

#include "wq_internal.h"
#include "wq_ptx.cuh"
#include "wq_stack.h"

namespace wq {

// Status word of the stack kernel: WQ_OK (0) or WQ_ERR_TIMEOUT (-6) after a
// bounded wait ran out (read and cleared by read_stack_status).
__device__ int g_stack_status = 0;

namespace {

constexpr int kSW = 16;                    // math warps
constexpr int kSThreads = (kSW + 1) * 32;  // + the weight-stream warp
constexpr int kSMathThreads = kSW * 32;

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }
__device__ __forceinline__ uint32_t pack_half2(float a, float b) {
  const __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<const uint32_t *>(&h);
}
__device__ __forceinline__ float exp2i(int k) { return __int_as_float((k + 127) << 23); }
// 2^e puts a block's largest |v| (bit pattern mxb) in [2^14, 2^15); 0 for a
// zero, infinite or nan maximum; clamped to [-100, 100].
__device__ __forceinline__ int block_exp(uint32_t mxb) {
  const int be = (int)(mxb >> 23);
  return mxb == 0u || be >= 255 ? 0 : max(-100, min(100, 141 - be));
}
__device__ __forceinline__ float half_bits(uint32_t b) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(b & 0xffffu)));
}
__device__ __forceinline__ void record_timeout() { atomicExch(&g_stack_status, -6); }

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long *p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_add_u64(unsigned long long *p, unsigned long long v) {
  asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
// named barrier over the 16 math warps (the stream warp never joins it)
__device__ __forceinline__ void math_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kSMathThreads) : "memory"); }

}  // namespace

namespace {

// The CTA's share of each phase.
struct Share {
  int g0, T;      // gate/up row tiles [g0, g0 + T)
  int e0, ne;     // down cells [e0, e0 + ne)
  int j0, nj;     // half blocks its cells touch
  int o0, no;     // owned y tiles [o0, o0 + no)
};
__host__ __device__ inline Share cta_share(const StackPlan &p, int c) {
  Share s;
  s.g0 = (int)((long long)c * p.RTg / p.G);
  s.T = (int)((long long)(c + 1) * p.RTg / p.G) - s.g0;
  s.e0 = (int)((long long)c * p.cells / p.G);
  s.ne = (int)((long long)(c + 1) * p.cells / p.G) - s.e0;
  s.j0 = s.e0 / p.RTd;
  s.nj = s.ne > 0 ? (s.e0 + s.ne - 1) / p.RTd - s.j0 + 1 : 0;
  s.o0 = (int)((long long)c * p.RTd / p.G);
  s.no = (int)((long long)(c + 1) * p.RTd / p.G) - s.o0;
  return s;
}

template <int BITS>
struct GuConst {
  static constexpr int BPK = BITS == 2 ? 512 : 1024;  // code bytes per (row tile, 128-feature block)
};

// 3-D TMA load (coordinates innermost first) with an L2 cache policy,
// completing on `bar` with the box's byte count.
__device__ __forceinline__ void tma3(void *dst, const CUtensorMap *map, int x, int y, int z, uint64_t *bar,
                                     uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, %3, "
      "%4}], [%5], %6;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

// The down stages of a CTA: its cells [e0, e0 + ne) in half-block-major order,
// cut at half-block ends and into runs of at most RPS row tiles (one TMA box).
__device__ __forceinline__ int dn_stage_count(const StackPlan &p, const Share &sh) {
  int n = 0;
  for (int jl = 0; jl < sh.nj; ++jl) {
    const int j = sh.j0 + jl;
    const int rb = max(sh.e0 - j * p.RTd, 0), re = min(sh.e0 + sh.ne - j * p.RTd, p.RTd);
    n += (re - rb + p.RPS - 1) / p.RPS;
  }
  return n;
}
// Walks the down stages in order: (half block j, first row tile, row tiles).
struct DnWalk {
  int jl, rt, re;
  __device__ __forceinline__ void start(const StackPlan &p, const Share &sh) {
    jl = 0;
    const int j = sh.j0;
    rt = max(sh.e0 - j * p.RTd, 0);
    re = min(sh.e0 + sh.ne - j * p.RTd, p.RTd);
  }
  // the current stage; then advance
  __device__ __forceinline__ void next(const StackPlan &p, const Share &sh, int *j, int *rt0, int *nrt) {
    *j = sh.j0 + jl;
    *rt0 = rt;
    *nrt = min(p.RPS, re - rt);
    rt += p.RPS;
    if (rt >= re) {
      ++jl;
      const int jn = sh.j0 + jl;
      rt = max(sh.e0 - jn * p.RTd, 0);
      re = min(sh.e0 + sh.ne - jn * p.RTd, p.RTd);
    }
  }
};

// Weight-stream warp: walks the stage sequence of every layer and fills the
// ring by TMA (lane 0 arms each stage's barrier and issues its boxes).
//   gate/up stage: k-blocks [kb0, kb0 + kps) of the CTA's T row tiles, both
//     projections: codes [pj][t][kps][BPK], then meta [pj][t][gmy][64] (blocks
//     past the matrix zero-filled);
//   down stage: half block j, row tiles [rt0, rt0 + RPS): codes [RPS][512],
//     then meta [RPS][GPH * 64] (rows past the matrix zero-filled).
template <int BITS_GU, int GG, int GD>
__device__ void stream_weights(const StackArgs &a, const StackPlan &p, const StackMaps &maps, const Share &sh,
                               uint8_t *smem, volatile int *abort_flag, volatile int *issued) {
  constexpr int BPK = GuConst<BITS_GU>::BPK;
  constexpr int GPBg = 128 / GG;
  constexpr int GPH = GD == 32 ? 2 : 1;  // down groups a half block touches
  const int lane = threadIdx.x & 31;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + p.off_full);
  uint64_t *empty = reinterpret_cast<uint64_t *>(smem + p.off_empty);
  uint8_t *ring = smem + p.off_ring;
  const uint64_t pol = l2_evict_first_policy();
  const int nsg = (p.KBg + p.kps - 1) / p.kps;
  const int nsd = dn_stage_count(p, sh);
  const uint32_t cbytes = (uint32_t)(2 * sh.T * p.kps * BPK);
  const uint32_t gu_bytes = cbytes + (uint32_t)(2 * sh.T * p.gmy * 64);
  const uint32_t dn_bytes = (uint32_t)(p.RPS * (512 + GPH * 64));
  if (lane != 0) return;
  int q = 0;
  for (int l = 0; l < a.n_layers; ++l) {
    const CUtensorMap *mp = maps.m[l];
    DnWalk w;
    w.start(p, sh);
    for (int s = 0; s < nsg + nsd; ++s, ++q) {
      const int slot = q % p.NS;
      if (q >= p.NS && !mbar_wait(&empty[slot], ((q / p.NS) - 1) & 1)) {
        record_timeout();
        *abort_flag = 1;
      }
      if (*abort_flag) {
        *issued = q;
        return;
      }
      uint8_t *st = ring + (size_t)slot * p.SB;
      if (s < nsg) {
        const int kb0 = s * p.kps;
        mbar_arrive_expect_tx(&full[slot], gu_bytes);
        for (int pj = 0; pj < 2; ++pj)
          for (int t0 = 0; t0 < sh.T; t0 += p.Tbox) {
            tma3(st + (size_t)(pj * sh.T + t0) * p.kps * BPK, &mp[pj], 0, kb0 * (BPK / 128), sh.g0 + t0, &full[slot], pol);
            tma3(st + cbytes + (size_t)(pj * sh.T + t0) * p.gmy * 64, &mp[2 + pj], 0, kb0 * GPBg, sh.g0 + t0,
                 &full[slot], pol);
          }
      } else {
        int j, rt0, nrt;
        w.next(p, sh, &j, &rt0, &nrt);
        const int g = GD == 32 ? 2 * j : GD == 64 ? j : (j >> 1);
        mbar_arrive_expect_tx(&full[slot], dn_bytes);
        tma3(st, &mp[4], 0, 4 * j, rt0, &full[slot], pol);
        tma3(st + p.RPS * 512, &mp[5], 0, g, rt0, &full[slot], pol);
      }
    }
  }
  *issued = q;
}

// Grid barrier: arrive (after the CTA's writes) / wait for generation `gen`.
__device__ __forceinline__ void grid_arrive(unsigned long long *ctr) {
  // caller: math_sync() first, so that every math thread's writes precede this
  if (threadIdx.x == 0) {
    __threadfence();
    red_add_u64(ctr, 1ull);
  }
}
__device__ __forceinline__ void grid_wait(const unsigned long long *ctr, unsigned long long target, volatile int *abort_flag) {
  if (threadIdx.x == 0 && !*abort_flag) {
    const unsigned long long t0 = global_timer_ns();
    unsigned it = 0;
    while (ld_acquire_u64(ctr) < target) {
      if ((++it & 255u) == 0u && global_timer_ns() - t0 > kWaitLimitNs) {
        record_timeout();
        *abort_flag = 1;
        break;
      }
    }
  }
  math_sync();
}

// The dot products of NB k-blocks of one row tile, both projections, their
// MMA chains interleaved (2 NB independent accumulators): per k-step the
// exact products code x binary16 activation on mma.sync, per group
//   ctot += s * (sx * sum q x' - z * sum x)
// (the affine dequantization s (q - z), x' = x / sx with the block's scale
// sx).  Codes [pj][T][kps][BPK], meta [pj][T][gmy][64] in the stage.
template <int BITS_GU, int GG, int NB>
__device__ __forceinline__ void gu_blocks(float (&ctot)[2][4], const int (&kb)[NB], const int (&kbl)[NB],
                                          const uint8_t *stg, uint32_t cbytes, int T, int tl, int kps, int gmy,
                                          const __half *xp, int xstride, const float *xsc, const float *xs, int M,
                                          int lane) {
  constexpr int BPK = BITS_GU == 2 ? 512 : 1024;
  constexpr int GPBg = 128 / GG, GSg = GG / 16;
  constexpr int NW = BITS_GU == 2 ? 4 : 8;
  const int col = 2 * (lane & 3);
  uint32_t b[NB][8][2];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      uint2 v = make_uint2(0u, 0u);  // tokens past M: zero columns
      if ((lane >> 2) < M) v = lds64(xp + (size_t)(lane >> 2) * xstride + (kb[nb] * 8 + ks) * 16 + 4 * (lane & 3));
      b[nb][ks][0] = v.x;
      b[nb][ks][1] = v.y;
    }
  uint32_t wds[NB][2][NW];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int pj = 0; pj < 2; ++pj) {
      const uint8_t *cb = stg + ((size_t)(pj * T + tl) * kps + kbl[nb]) * BPK + lane * 16;
      const uint4 w0 = lds128(cb);
      wds[nb][pj][0] = w0.x; wds[nb][pj][1] = w0.y; wds[nb][pj][2] = w0.z; wds[nb][pj][3] = w0.w;
      if (BITS_GU == 4) {
        const uint4 w1 = lds128(cb + 512);
        wds[nb][pj][NW - 4] = w1.x; wds[nb][pj][NW - 3] = w1.y; wds[nb][pj][NW - 2] = w1.z; wds[nb][pj][NW - 1] = w1.w;
      }
    }
  float acc[NB][2][4];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
    for (int nb = 0; nb < NB; ++nb)
#pragma unroll
      for (int pj = 0; pj < 2; ++pj) {
        uint32_t af[4];
        if (BITS_GU == 2) {
          const uint32_t x = wds[nb][pj][(ks >> 1) & 3], x8 = x >> 8;
          const int s4 = (ks & 1) * 4;
          af[0] = x & (0x00030003u << s4);
          af[1] = x8 & (0x00030003u << s4);
          af[2] = x & (0x000C000Cu << s4);
          af[3] = x8 & (0x000C000Cu << s4);
        } else {
          const uint32_t x = wds[nb][pj][ks], x8 = x >> 8;
          af[0] = x & 0x000F000Fu;
          af[1] = x8 & 0x000F000Fu;
          af[2] = x & 0x00F000F0u;
          af[3] = x8 & 0x00F000F0u;
        }
        if (ks % GSg == 0)
          mma_f16_16816_zc(acc[nb][pj], af, b[nb][ks][0], b[nb][ks][1]);
        else
          mma_f16_16816(acc[nb][pj], af, b[nb][ks][0], b[nb][ks][1]);
      }
    if ((ks + 1) % GSg == 0) {
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int gl = kb[nb] * GPBg + ks / GSg;
        const float2 gsum = *reinterpret_cast<const float2 *>(xs + gl * 8 + col);
        const float2 sc = *reinterpret_cast<const float2 *>(xsc + kb[nb] * 8 + col);
#pragma unroll
        for (int pj = 0; pj < 2; ++pj) {
          const uint2 sz = lds64(stg + cbytes + ((size_t)(pj * T + tl) * gmy + kbl[nb] * GPBg + ks / GSg) * 64 +
                                 (lane >> 2) * 8);
          const float s_lo = half_bits(sz.x), s_hi = half_bits(sz.x >> 16);
          const float zs_lo = -s_lo * half_bits(sz.y), zs_hi = -s_hi * half_bits(sz.y >> 16);
          float *ct = ctot[pj];
          ct[0] = fmaf(s_lo * sc.x, acc[nb][pj][0], ct[0]);
          ct[1] = fmaf(s_lo * sc.y, acc[nb][pj][1], ct[1]);
          ct[2] = fmaf(s_hi * sc.x, acc[nb][pj][2], ct[2]);
          ct[3] = fmaf(s_hi * sc.y, acc[nb][pj][3], ct[3]);
          ct[0] = fmaf(zs_lo, gsum.x, ct[0]);
          ct[1] = fmaf(zs_lo, gsum.y, ct[1]);
          ct[2] = fmaf(zs_hi, gsum.x, ct[2]);
          ct[3] = fmaf(zs_hi, gsum.y, ct[3]);
        }
      }
    }
  }
}

using bf16 = __nv_bfloat16;
__device__ __forceinline__ const bf16 *B16(const uint16_t *p) { return reinterpret_cast<const bf16 *>(p); }
__device__ __forceinline__ bf16 *B16(uint16_t *p) { return reinterpret_cast<bf16 *>(p); }

template <int BITS_GU, int GG, int GD>
__global__ void __launch_bounds__(kSThreads, 1) stack_kernel(const __grid_constant__ StackArgs a, const StackPlan p,
                                                              const __grid_constant__ StackMaps maps) {
  extern __shared__ __align__(1024) uint8_t smem[];
  constexpr int BPK = GuConst<BITS_GU>::BPK;
  constexpr int GPBg = 128 / GG;      // gate/up groups per block
  constexpr int LPG = GG / 4;         // conversion lanes per gate/up group (4 features a lane)
  constexpr int GPH = GD == 32 ? 2 : 1;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int M = a.M, r = a.r, Q = 1 + 2 * r, Qp = p.Qp;
  const Share sh = cta_share(p, blockIdx.x);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + p.off_full);
  uint64_t *empty = reinterpret_cast<uint64_t *>(smem + p.off_empty);
  volatile int *misc = reinterpret_cast<volatile int *>(smem + p.off_misc);  // [0] abort, [1] issued
  unsigned long long *base_s = reinterpret_cast<unsigned long long *>(smem + p.off_misc + 16);
  __half *xp = reinterpret_cast<__half *>(smem + p.off_x);         // [M][xstride] activation panel
  float *xsc = reinterpret_cast<float *>(smem + p.off_xsc);        // [KBg][8] 2^(24-e)
  float *xs = reinterpret_cast<float *>(smem + p.off_xs);          // [KBg*GPB][8] group sums of x
  float *slot = reinterpret_cast<float *>(smem + p.off_slot);      // [T][WPT][2][16][M]
  float *hs = reinterpret_cast<float *>(smem + p.off_h);           // [M][Tmax*16] h of the CTA's rows
  uint2 *hp = reinterpret_cast<uint2 *>(smem + p.off_hp);          // [nj][4 k-steps][8 tokens][4] down B fragments
  float *hsc = reinterpret_cast<float *>(smem + p.off_hsc);        // [nj][8] 2^(24-e)
  float *hxs = reinterpret_cast<float *>(smem + p.off_hxs);        // [nj][2][8] sums of h over 32 features
  __nv_bfloat16 *lb = reinterpret_cast<__nv_bfloat16 *>(smem + p.off_lb);  // [2][Tmax*16][r]
  __nv_bfloat16 *la = reinterpret_cast<__nv_bfloat16 *>(smem + p.off_la);  // [own_max*16][2r]
  float *rt = reinterpret_cast<float *>(smem + p.off_rt);          // [M][Qp] tile partials summed
  float *yo = reinterpret_cast<float *>(smem + p.off_yo);          // [own][M][16] the owned tiles of y
  float *red = reinterpret_cast<float *>(smem + p.off_red);        // [512 x 4] scratch of the reductions
  uint8_t *ring = smem + p.off_ring;

  if (tid == 0) {
    for (int s = 0; s < p.NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kSW);
    }
    fence_barrier_init();
    misc[0] = 0;
    misc[1] = -1;
    // barrier generations of this launch count from the counter's value at
    // the start: every barrier takes exactly G arrivals, and no CTA passes
    // the first barrier before all have arrived, so this is base * G exactly
    base_s[0] = ld_acquire_u64(a.ctr) / (unsigned long long)p.G * (unsigned long long)p.G;
  }
  __syncthreads();
  if (warp == kSW) {
    stream_weights<BITS_GU, GG, GD>(a, p, maps, sh, smem, &misc[0], &misc[1]);
    return;
  }
  const unsigned long long base = base_s[0];
  unsigned long long gen = 0;
  const int KBd = (a.inter + 127) / 128;
  (void)KBd;
  const int nsg = (p.KBg + p.kps - 1) / p.kps;
  const int nsd = dn_stage_count(p, sh);
  int q = 0;  // stage sequence position

  // ---- the first layer's tile partials of x_in (owned tiles), barrier ----
  auto owner_stats = [&](const __nv_bfloat16 *y, const __nv_bfloat16 *A) {
    // tp[t][m][q] = sum over the tile's 16 features of w * y, w = y (q = 0) or A[q - 1]
    for (int i = tid; i < sh.no * M * Qp; i += kSMathThreads) {
      const int tl = i / (M * Qp), rem = i % (M * Qp), m = rem / Qp, qq = rem % Qp;
      const int t = sh.o0 + tl;
      float s = 0.f;
      if (qq < Q) {
        const uint4 y0 = ldg_cg128(y + (size_t)m * a.d + t * 16), y1 = ldg_cg128(y + (size_t)m * a.d + t * 16 + 8);
        const uint32_t yv[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
        uint32_t wv[8];
        if (qq == 0) {
#pragma unroll
          for (int u = 0; u < 8; ++u) wv[u] = yv[u];
        } else {
          const uint4 w0 = __ldg(reinterpret_cast<const uint4 *>(A + (size_t)(qq - 1) * a.d + t * 16));
          const uint4 w1 = __ldg(reinterpret_cast<const uint4 *>(A + (size_t)(qq - 1) * a.d + t * 16 + 8));
          wv[0] = w0.x; wv[1] = w0.y; wv[2] = w0.z; wv[3] = w0.w;
          wv[4] = w1.x; wv[5] = w1.y; wv[6] = w1.z; wv[7] = w1.w;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          s = fmaf(bf16_lo(wv[u]), bf16_lo(yv[u]), s);
          s = fmaf(bf16_hi(wv[u]), bf16_hi(yv[u]), s);
        }
      }
      a.tp[((size_t)t * M + m) * Qp + qq] = s;
    }
  };
  // the LoRA-B rows of layer l's gate/up tiles, by cp.async (waited for with
  // the activation panel): issued before the barrier that opens the layer
  auto prefetch_lb = [&](int l) {
    if (r <= 0) return;
    const int per_row = r / 8, rows = sh.T * 16;
    for (int i = tid; i < 2 * rows * per_row; i += kSMathThreads) {
      const int pj = i / (rows * per_row), rem = i % (rows * per_row), rl = rem / per_row, c = rem % per_row;
      cp_async16(lb + ((size_t)pj * p.Tmax * 16 + rl) * r + c * 8,
                 B16(a.L[l].lora_b[pj]) + (size_t)(sh.g0 * 16 + rl) * r + c * 8);
    }
    cp_async_commit();
  };
  owner_stats(B16(a.x_in), B16(a.L[0].lora_a));
  prefetch_lb(0);
  math_sync();
  grid_arrive(a.ctr);
  ++gen;

  for (int l = 0; l < a.n_layers; ++l) {
    const StackLayerDev &Ly = a.L[l];
    const bool last = l == a.n_layers - 1;
    const bf16 *cur = l == 0 ? B16(a.x_in) : B16(a.xw);
    grid_wait(a.ctr, base + (unsigned long long)p.G * gen, &misc[0]);

    // ================= gate/up =================
    // (a) inputs: the activation panel (raw bf16, converted in place below)
    // and the tile partials
    {
      const int cpr = p.KBg * 16;  // 16-byte chunks per token row
      for (int i = tid; i < M * cpr; i += kSMathThreads) {
        const int m = i / cpr, c = i % cpr;
        cp_async16(xp + (size_t)m * p.xstride + c * 8, cur + (size_t)m * a.d + c * 8);
      }
      cp_async_commit();
      // tile partials summed over the RTd tiles: thread (item, split) adds
      // the tiles t = split, split + S, ... (eight loads in flight; adjacent
      // threads read adjacent 16 bytes), then a fixed tree over the S splits
      {
        const int Q4 = Qp / 4, items = M * Q4;
        int S = 1;
        while (S * 2 * items <= kSMathThreads && S * 2 <= p.RTd) S *= 2;
        float4 *tr = reinterpret_cast<float4 *>(red);  // [S][items]
        if (tid < S * items) {
          const int item = tid % items, sp = tid / items, m = item / Q4, j = item % Q4;
          float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
          for (int tb = sp; tb < p.RTd; tb += 8 * S) {
            float4 v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
              v[u] = tb + u * S < p.RTd
                         ? __ldcg(reinterpret_cast<const float4 *>(a.tp + ((size_t)(tb + u * S) * M + m) * Qp) + j)
                         : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              acc.x += v[u].x;
              acc.y += v[u].y;
              acc.z += v[u].z;
              acc.w += v[u].w;
            }
          }
          tr[tid] = acc;
        }
        for (int h = S >> 1; h >= 1; h >>= 1) {
          math_sync();
          if (tid < h * items) {
            const float4 b2 = tr[tid + h * items];
            float4 v = tr[tid];
            v.x += b2.x;
            v.y += b2.y;
            v.z += b2.z;
            v.w += b2.w;
            tr[tid] = v;
          }
        }
        math_sync();
        if (tid < items) reinterpret_cast<float4 *>(rt)[tid] = tr[tid];
      }
      cp_async_wait_all();
      math_sync();
      if (a.prenorm)
        for (int m = tid; m < M; m += kSMathThreads)
          rt[(size_t)m * Qp] = __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(rt[(size_t)m * Qp], (float)a.d), kRmsEps)));
    }
    // (b) activation panel -> binary16 in place, per (block, token): 2^e puts
    // the block's max |x| in [2^14, 2^15), times 4^-c (2-bit) or 16^-c
    // (4-bit) for the code class c the features meet
    {
      const int st = lane >> 2, hi = (lane >> 1) & 1;
      const int shc = BITS_GU == 2 ? 4 * (st & 1) + 2 * hi : 4 * hi;
      const int u0 = 4 * (lane & 1) + hi;
      for (int i = tid; i < p.KBg * (8 - M); i += kSMathThreads) {
        // padding tokens: zero scales and group sums
        const int kb = i / (8 - M), m = M + i % (8 - M);
        xsc[kb * 8 + m] = 0.f;
        for (int g = 0; g < GPBg; ++g) xs[(kb * GPBg + g) * 8 + m] = 0.f;
      }
      for (int it = warp; it < p.KBg * M; it += kSW) {
        const int kb = it / M, m = it % M;
        const uint2 raw = lds64(xp + (size_t)m * p.xstride + kb * 128 + 4 * lane);
        const float f0 = bf16_lo(raw.x), f1 = bf16_hi(raw.x), f2 = bf16_lo(raw.y), f3 = bf16_hi(raw.y);
        const uint32_t v = __float_as_uint(fmaxf(fmaxf(fabsf(f0), fabsf(f1)), fmaxf(fabsf(f2), fabsf(f3))));
        const int e = block_exp(__reduce_max_sync(0xffffffffu, v));
        __syncwarp();
        const float mul = exp2i(e - shc);
        uint32_t *w = reinterpret_cast<uint32_t *>(xp + (size_t)m * p.xstride + kb * 128 + st * 16);
        w[u0] = pack_half2(f0 * mul, f1 * mul);
        w[u0 + 2] = pack_half2(f2 * mul, f3 * mul);
        float gs = (f0 + f1) + (f2 + f3);
#pragma unroll
        for (int o = 1; o < LPG; o <<= 1) gs += __shfl_xor_sync(0xffffffffu, gs, o);
        if ((lane % LPG) == 0) xs[(kb * GPBg + lane / LPG) * 8 + m] = gs;
        if (lane == 0) xsc[kb * 8 + m] = exp2i(24 - e);
      }
    }
    math_sync();
    // (c) the dot products: warp (tile tl, k-slice ksl) takes the stage's
    // k-blocks ksl and ksl + WPT
    {
      const int tl = warp / p.WPT, ksl = warp % p.WPT;
      const bool active = tl < sh.T;
      float ctot[2][4];
#pragma unroll
      for (int pj = 0; pj < 2; ++pj)
#pragma unroll
        for (int u = 0; u < 4; ++u) ctot[pj][u] = 0.f;
      const int col = 2 * (lane & 3);  // tokens of this lane's accumulators
      for (int s = 0; s < nsg; ++s, ++q) {
        const int sl = q % p.NS;
        const bool ok = !misc[0] && mbar_wait(&full[sl], (q / p.NS) & 1);
        if (!ok && lane == 0 && !misc[0]) {
          record_timeout();
          misc[0] = 1;
        }
        const int kb0 = s * p.kps, nk = min(p.kps, p.KBg - kb0);
        const uint8_t *stg = ring + (size_t)sl * p.SB;
        const uint32_t cbytes = (uint32_t)(2 * sh.T * p.kps * BPK);
        // the warp's blocks in this stage: ksl and ksl + WPT, two in flight
        if (active && ok && !misc[0] && ksl < nk) {
          if (ksl + p.WPT < nk) {
            const int kb[2] = {kb0 + ksl, kb0 + ksl + p.WPT}, kbl[2] = {ksl, ksl + p.WPT};
            gu_blocks<BITS_GU, GG, 2>(ctot, kb, kbl, stg, cbytes, sh.T, tl, p.kps, p.gmy, xp, p.xstride, xsc, xs, M, lane);
          } else {
            const int kb[1] = {kb0 + ksl}, kbl[1] = {ksl};
            gu_blocks<BITS_GU, GG, 1>(ctot, kb, kbl, stg, cbytes, sh.T, tl, p.kps, p.gmy, xp, p.xstride, xsc, xs, M, lane);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[sl]);
      }
      // the warp's partial sums -> slot [tl][ksl][pj][16][M]
      if (active) {
        const int r0 = lane >> 2;
#pragma unroll
        for (int pj = 0; pj < 2; ++pj) {
          float *so = slot + ((size_t)(tl * p.WPT + ksl) * 2 + pj) * 16 * M;
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            if (col + c >= M) continue;
            so[r0 * M + col + c] = ctot[pj][c];
            so[(r0 + 8) * M + col + c] = ctot[pj][2 + c];
          }
        }
      }
    }
    math_sync();
    // (d) epilogue: add the k-slices in order, LoRA-B, RMSNorm scale, SiLU(g) * u
    for (int i = tid; i < sh.T * 16 * M; i += kSMathThreads) {
      const int tl = i / (16 * M), rem = i % (16 * M), row = rem / M, m = rem % M;
      float g = 0.f, u = 0.f;
      for (int k = 0; k < p.WPT; ++k) {
        g += slot[(((size_t)(tl * p.WPT + k) * 2 + 0) * 16 + row) * M + m];
        u += slot[(((size_t)(tl * p.WPT + k) * 2 + 1) * 16 + row) * M + m];
      }
      const int rl = tl * 16 + row;
      if (r > 0) {
        const float *tg = rt + (size_t)m * Qp + 1, *tu = tg + r;
        const __nv_bfloat16 *bg = lb + (size_t)rl * r, *bu = lb + ((size_t)p.Tmax * 16 + rl) * r;
        float lg = 0.f, lu = 0.f;
        for (int qq = 0; qq < r; qq += 8) {
          const uint4 vg = lds128(bg + qq), vu = lds128(bu + qq);
          const uint32_t wg[4] = {vg.x, vg.y, vg.z, vg.w}, wu[4] = {vu.x, vu.y, vu.z, vu.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            lg = fmaf(tg[qq + 2 * e], bf16_lo(wg[e]), lg);
            lg = fmaf(tg[qq + 2 * e + 1], bf16_hi(wg[e]), lg);
            lu = fmaf(tu[qq + 2 * e], bf16_lo(wu[e]), lu);
            lu = fmaf(tu[qq + 2 * e + 1], bf16_hi(wu[e]), lu);
          }
        }
        g = fmaf(Ly.lora_scale, lg, g);
        u = fmaf(Ly.lora_scale, lu, u);
      }
      const float rs = a.prenorm ? rt[(size_t)m * Qp] : 1.f;
      g *= rs;
      u *= rs;
      const __nv_bfloat16 hb = __float2bfloat16_rn(g / (1.f + __expf(-g)) * u);
      hs[(size_t)m * p.Tmax * 16 + rl] = __bfloat162float(hb);
      const int n = (sh.g0 + tl) * 16 + row;
      if (p.h_barrier) B16(a.hg)[(size_t)m * a.inter + n] = hb;
      if (a.h_states) B16(a.h_states)[((size_t)l * M + m) * a.inter + n] = hb;
    }
    if (p.h_barrier) {
      math_sync();
      grid_arrive(a.ctr);
      ++gen;
      grid_wait(a.ctr, base + (unsigned long long)p.G * gen, &misc[0]);
    } else {
      math_sync();
    }

    // ================= down (K-slice) =================
    // (a) the next layer's LoRA-A columns of the owned tiles (used by the owner phase)
    const bf16 *A_next = last ? nullptr : B16(a.L[l + 1].lora_a);
    if (!last && r > 0 && A_next) {
      // la [own*16 rows][2r]: element (row, j) = A_next[j][o0*16 + row]
      for (int i = tid; i < 2 * r * sh.no * 2; i += kSMathThreads) {
        const int j = i % (2 * r), c = i / (2 * r);  // c: 8-feature chunk of the owned rows
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(A_next + (size_t)j * a.d + sh.o0 * 16 + c * 8));
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int t = 0; t < 8; ++t)
          la[(size_t)(c * 8 + t) * 2 * r + j] = __ushort_as_bfloat16(static_cast<unsigned short>(w[t >> 1] >> (16 * (t & 1))));
      }
    }
    // (b) B fragments of h per half block: per (half block, token) 2^e puts the
    // largest |h| in [2^14, 2^15); features 8..15 of each k-step times 16^-1
    for (int it = warp; it < sh.nj * 8; it += kSW) {
      const int jl = it >> 3, m = it & 7, j = sh.j0 + jl;
      const int f = 2 * lane;  // features f, f + 1 of the half block
      float v0 = 0.f, v1 = 0.f;
      if (m < M) {
        const int n = j * 64 + f;
        const int tloc = n / 16 - sh.g0;
        if (!p.h_barrier && tloc >= 0 && tloc < sh.T) {
          v0 = hs[(size_t)m * p.Tmax * 16 + (n - sh.g0 * 16)];
          v1 = hs[(size_t)m * p.Tmax * 16 + (n - sh.g0 * 16) + 1];
        } else if (n < a.inter) {
          const uint32_t w = __ldcg(reinterpret_cast<const unsigned int *>(a.hg + (size_t)m * a.inter + n));
          v0 = bf16_lo(w);
          v1 = bf16_hi(w);
        }
      }
      const uint32_t mv = __float_as_uint(fmaxf(fabsf(v0), fabsf(v1)));
      const int e = block_exp(__reduce_max_sync(0xffffffffu, mv));
      const int ks = f >> 4, pp = (f & 15) >> 1;  // k-step, feature pair in it
      const float mul = exp2i(e - 4 * ((f >> 3) & 1));
      uint32_t *w = reinterpret_cast<uint32_t *>(hp + ((size_t)(jl * 4 + ks) * 8 + m) * 4 + (pp & 3));
      w[pp >> 2] = pack_half2(v0 * mul, v1 * mul);
      float s = v0 + v1;
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if ((lane & 15) == 0) hxs[(jl * 2 + (lane >> 4)) * 8 + m] = s;
      if (lane == 0) hsc[jl * 8 + m] = exp2i(24 - e);
    }
    math_sync();
    // (c) the cells: warp w takes cells w, w + 16, ... of each stage; a cell
    // (half block j, row tile t) is 4 MMAs and yields y's partial sums of the
    // tile's 16 rows over the half block's 64 features
    DnWalk dw;
    dw.start(p, sh);
    for (int s = 0; s < nsd; ++s, ++q) {
      const int sl = q % p.NS;
      const bool ok = !misc[0] && mbar_wait(&full[sl], (q / p.NS) & 1);
      if (!ok && lane == 0 && !misc[0]) {
        record_timeout();
        misc[0] = 1;
      }
      int j, rt0, nc;
      dw.next(p, sh, &j, &rt0, &nc);
      const uint8_t *stg = ring + (size_t)sl * p.SB;
      if (ok && !misc[0] && warp < nc) {
        // cells warp, warp + 16, warp + 32, warp + 48 of the stage (same half
        // block): their MMA chains interleaved on the shared B fragments
        constexpr int CW = 4;
        const int jl = j - sh.j0;
        uint32_t wd[CW][4];
#pragma unroll
        for (int c2 = 0; c2 < CW; ++c2) {
          const int cl = warp + c2 * kSW;
          const uint4 wv = cl < nc ? lds128(stg + (size_t)cl * 512 + lane * 16) : make_uint4(0u, 0u, 0u, 0u);
          wd[c2][0] = wv.x; wd[c2][1] = wv.y; wd[c2][2] = wv.z; wd[c2][3] = wv.w;
        }
        float acc[CW][2][4];
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          const uint2 bv = hp[((size_t)(jl * 4 + ks) * 8 + (lane >> 2)) * 4 + (lane & 3)];
          const int ch = GD == 32 ? (ks >> 1) : 0;
#pragma unroll
          for (int c2 = 0; c2 < CW; ++c2) {
            const uint32_t x = wd[c2][ks], x8 = x >> 8;
            const uint32_t af[4] = {x & 0x000F000Fu, x8 & 0x000F000Fu, x & 0x00F000F0u, x8 & 0x00F000F0u};
            if (GD == 32 ? (ks & 1) == 0 : ks == 0)
              mma_f16_16816_zc(acc[c2][ch], af, bv.x, bv.y);
            else
              mma_f16_16816(acc[c2][ch], af, bv.x, bv.y);
          }
        }
        const int col = 2 * (lane & 3);
        const float2 sc = *reinterpret_cast<const float2 *>(hsc + jl * 8 + col);
        float2 gs[GPH];
#pragma unroll
        for (int ch = 0; ch < GPH; ++ch) {
          if (GD == 32) {
            gs[ch] = make_float2(hxs[(jl * 2 + ch) * 8 + col], hxs[(jl * 2 + ch) * 8 + col + 1]);
          } else {
            gs[ch] = make_float2(hxs[(jl * 2) * 8 + col] + hxs[(jl * 2 + 1) * 8 + col],
                                 hxs[(jl * 2) * 8 + col + 1] + hxs[(jl * 2 + 1) * 8 + col + 1]);
          }
        }
#pragma unroll
        for (int c2 = 0; c2 < CW; ++c2) {
          const int cl = warp + c2 * kSW, t = rt0 + cl;
          if (cl >= nc) break;
          float y[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int ch = 0; ch < GPH; ++ch) {
            const uint2 sz = lds64(stg + (size_t)p.RPS * 512 + ((size_t)cl * GPH + ch) * 64 + (lane >> 2) * 8);
            const float s_lo = half_bits(sz.x), s_hi = half_bits(sz.x >> 16);
            const float zs_lo = -s_lo * half_bits(sz.y), zs_hi = -s_hi * half_bits(sz.y >> 16);
            y[0] = fmaf(s_lo * sc.x, acc[c2][ch][0], y[0]);
            y[1] = fmaf(s_lo * sc.y, acc[c2][ch][1], y[1]);
            y[2] = fmaf(s_hi * sc.x, acc[c2][ch][2], y[2]);
            y[3] = fmaf(s_hi * sc.y, acc[c2][ch][3], y[3]);
            y[0] = fmaf(zs_lo, gs[ch].x, y[0]);
            y[1] = fmaf(zs_lo, gs[ch].y, y[1]);
            y[2] = fmaf(zs_hi, gs[ch].x, y[2]);
            y[3] = fmaf(zs_hi, gs[ch].y, y[3]);
          }
          const int r0 = t * 16 + (lane >> 2);
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            if (col + c >= M) continue;
            float *pr = a.part + ((size_t)j * M + col + c) * a.d;
            if (r0 < a.d) pr[r0] = y[c];
            if (r0 + 8 < a.d) pr[r0 + 8] = y[2 + c];
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[sl]);
    }
    math_sync();
    grid_arrive(a.ctr);
    ++gen;
    grid_wait(a.ctr, base + (unsigned long long)p.G * gen, &misc[0]);

    // ================= owner: y tiles =================
    // output (tile, m, row): sum over half blocks j of part[j][m][row]:
    // thread (output, split) adds j = split, split + S, ... (eight loads in
    // flight; adjacent threads read adjacent rows), then a fixed tree over
    // the S splits; plus the residual, kept in shared memory from the
    // previous layer
    {
      const int nout = sh.no * 16 * M;
      int S = 1;
      while (S * 2 * nout <= kSMathThreads && S * 2 <= p.U) S *= 2;
      bf16 *dst = last ? B16(a.y_out) : B16(a.xw);
      for (int base = 0; base < nout; base += kSMathThreads) {  // one round unless nout > 512
        const int nb = min(nout - base, kSMathThreads);
        const int SS = base == 0 ? S : 1;
        if (tid < SS * nb) {
          const int o = base + tid % nb, sp = tid / nb;
          const int tl = o / (16 * M), rem = o % (16 * M), m = rem / 16, row = rem % 16;
          const int n = (sh.o0 + tl) * 16 + row;
          float sum = 0.f;
          for (int jb = sp; jb < p.U; jb += 8 * SS) {
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
              v[u] = jb + u * SS < p.U ? __ldcg(a.part + ((size_t)(jb + u * SS) * M + m) * a.d + n) : 0.f;
#pragma unroll
            for (int u = 0; u < 8; ++u) sum += v[u];
          }
          red[tid] = sum;
        }
        for (int h = SS >> 1; h >= 1; h >>= 1) {
          math_sync();
          if (tid < h * nb) red[tid] += red[tid + h * nb];
        }
        math_sync();
        if (tid < nb) {
          const int o = base + tid;
          const int tl = o / (16 * M), rem = o % (16 * M), m = rem / 16, row = rem % 16;
          const int n = (sh.o0 + tl) * 16 + row;
          const float res = l == 0 ? __bfloat162float(cur[(size_t)m * a.d + n]) : yo[o];
          const __nv_bfloat16 yb = __float2bfloat16_rn(red[tid] + res);
          dst[(size_t)m * a.d + n] = yb;
          if (a.states) B16(a.states)[((size_t)l * M + m) * a.d + n] = yb;
          yo[o] = __bfloat162float(yb);  // the next layer's residual and tile partials
        }
        math_sync();
      }
      math_sync();
      // the next layer's tile partials of the stored y: same fma order as the
      // first layer's (w_c * y_c over the tile's features in order)
      if (!last) {
        const float *yv = yo;  // [tl][m][16]
        for (int i = tid; i < sh.no * M * Qp; i += kSMathThreads) {
          const int tl = i / (M * Qp), rem = i % (M * Qp), m = rem / Qp, qq = rem % Qp;
          const int t = sh.o0 + tl;
          float s = 0.f;
          if (qq < Q) {
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              const float y = yv[((size_t)tl * M + m) * 16 + c];
              const float w = qq == 0 ? y : __bfloat162float(la[(size_t)(tl * 16 + c) * 2 * r + (qq - 1)]);
              s = fmaf(w, y, s);
            }
          }
          a.tp[((size_t)t * M + m) * Qp + qq] = s;
        }
      }
    }
    if (!last) prefetch_lb(l + 1);
    math_sync();
    if (!last) {
      grid_arrive(a.ctr);
      ++gen;
    }
  }
  // drain: every stage the stream warp issued has landed before the CTA exits
  if (tid == 0 && misc[0]) {
    const unsigned long long t0 = global_timer_ns();
    while (misc[1] < 0 && global_timer_ns() - t0 < kWaitLimitNs) {
    }
    for (int qq = q; qq < misc[1]; ++qq)
      if (!mbar_wait(&full[qq % p.NS], (qq / p.NS) & 1)) break;
  }
}

uint32_t up128(uint32_t v) { return (v + 127u) / 128u * 128u; }

}  // namespace

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
size_t stack_buffer_bytes(int M, int d, int inter, int r) {
  const size_t RTd = (size_t)(d + 15) / 16, U = (size_t)(inter + 63) / 64;
  const size_t Qp = WQ_TP_STRIDE(r);
  size_t off = 0;
  off += ((size_t)M * d * 2 + 255) / 256 * 256;       // xw
  off += (RTd * M * Qp * 4 + 255) / 256 * 256;        // tp
  off += ((size_t)M * inter * 2 + 255) / 256 * 256;   // hg
  off += (U * M * d * 4 + 255) / 256 * 256;           // part
  off += ((size_t)M * d * 2 + 255) / 256 * 256;       // output of a launch that is not the last of a stack
  return off;
}

bool stack_plan(int M, int d, int inter, int r, int bits_gu, int g_gu, int g_dn, int num_sms, StackPlan *out) {
  if (M < 1 || M > 8 || num_sms <= 0) return false;
  if (g_gu != g_dn || (g_gu != 32 && g_gu != 64 && g_gu != 128) || (bits_gu != 2 && bits_gu != 4)) return false;
  if (d % 128 != 0 || inter % 64 != 0 || d < 128) return false;
  if (r < 0 || r > kMaxRank || r % 8 != 0) return false;
  StackPlan p{};
  p.RTg = inter / 16;
  p.G = std::min(num_sms, p.RTg);  // every CTA takes at least one gate/up row tile
  p.KBg = d / 128;
  p.RTd = d / 16;
  p.U = inter / 64;
  p.cells = p.U * p.RTd;
  p.Tmax = (p.RTg + p.G - 1) / p.G;
  if (p.Tmax > kSW) return false;  // every CTA takes 1..16 gate/up tiles
  p.WPT = kSW / p.Tmax;
  p.own_max = (p.RTd + p.G - 1) / p.G;
  p.Qp = WQ_TP_STRIDE(r);
  // the largest number of half blocks a CTA's cells touch, and whether every
  // CTA's half blocks lie inside its own gate/up rows
  p.nj_max = 0;
  p.h_barrier = 0;
  for (int c = 0; c < p.G; ++c) {
    const Share s = cta_share(p, c);
    p.nj_max = std::max(p.nj_max, s.nj);
    if (s.ne > 0 && (s.j0 * 4 < s.g0 || (s.j0 + s.nj) * 4 > s.g0 + s.T)) p.h_barrier = 1;
  }
  const int BPK = bits_gu == 2 ? 512 : 1024, GPBg = 128 / g_gu, GPH = g_dn == 32 ? 2 : 1;
  const int MP = 8;  // token columns of the MMA
  const int nout = p.own_max * 16 * M;
  p.nchk = std::max(1, std::min(kSMathThreads / (M * (p.Qp / 4)), p.RTd));
  uint32_t off = 0;
  p.off_full = off;  off = up128(off + 64 * 8);
  p.off_empty = off; off = up128(off + 64 * 8);
  p.off_misc = off;  off = up128(off + 32);
  p.xstride = d + 16;
  p.off_x = off;     off = up128(off + (uint32_t)M * p.xstride * 2);
  p.off_xsc = off;   off = up128(off + (uint32_t)p.KBg * MP * 4);
  p.off_xs = off;    off = up128(off + (uint32_t)p.KBg * GPBg * MP * 4);
  p.off_slot = off;  off = up128(off + (uint32_t)kSW * 2 * 16 * M * 4);
  p.off_h = off;     off = up128(off + (uint32_t)M * p.Tmax * 16 * 4);
  p.off_hp = off;    off = up128(off + (uint32_t)std::max(p.nj_max, 1) * 4 * MP * 4 * 8);
  p.off_hsc = off;   off = up128(off + (uint32_t)std::max(p.nj_max, 1) * MP * 4);
  p.off_hxs = off;   off = up128(off + (uint32_t)std::max(p.nj_max, 1) * 2 * MP * 4);
  p.off_lb = off;    off = up128(off + (uint32_t)2 * p.Tmax * 16 * r * 2);
  p.off_la = off;    off = up128(off + (uint32_t)p.own_max * 16 * 2 * r * 2);
  p.off_rt = off;    off = up128(off + (uint32_t)M * p.Qp * 4);
  p.off_yo = off;    off = up128(off + (uint32_t)nout * 4);
  p.off_red = off;   off = up128(off + (uint32_t)kSMathThreads * 16);
  off = (off + 1023) / 1024 * 1024;
  p.off_ring = off;
  constexpr uint32_t kSmemLimit = 232448;
  // The ring's stages.  A gate/up stage: `depth` k-blocks for each of the
  // WPT k-slice warps of a tile (kps blocks of the CTA's rows; codes and gmy
  // groups of meta per projection and row tile); a down stage: RPS = 32 depth
  // row tiles of a half block (2 depth cells for each of the 16 warps).
  // Depth 2 (two independent MMA chains per warp and projection) unless
  // fewer than four such stages fit.
  const int dn_cell = 512 + GPH * 64;
  auto gmy_of = [&](int k) { return (k * GPBg + 1) / 2 * 2; };
  auto gu_stage = [&](int k) { return 2 * p.Tmax * (k * BPK + gmy_of(k) * 64); };
  for (int depth = 2; depth >= 1; --depth) {
    p.kps = std::min(depth * p.WPT, p.KBg);
    p.RPS = 2 * depth * kSW;
    p.SB = std::max(gu_stage(p.kps), p.RPS * dn_cell);
    p.SB = (p.SB + 127) / 128 * 128;
    if (off + 4u * (uint32_t)p.SB <= kSmemLimit) break;
  }
  p.gmy = gmy_of(p.kps);
  p.cps = p.RPS;
  p.Tbox = p.RTg % p.G == 0 ? p.Tmax : 1;
  if (p.gmy > 256 || p.kps * BPK / 128 > 256) return false;  // TMA box limits
  p.NS = std::min(64, (int)((kSmemLimit - off) / (uint32_t)p.SB));
  if (p.NS < 4) return false;
  p.smem = off + (uint32_t)p.NS * p.SB;
  *out = p;
  return true;
}

namespace {

template <int B, int GG, int GD>
cudaError_t launch_stack_t(const StackArgs &a, const StackPlan &p, const StackMaps &maps, cudaStream_t s) {
  auto kern = stack_kernel<B, GG, GD>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.G);
  cfg.blockDim = dim3(kSThreads);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident at once, or the launch fails
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a, p, maps);
}

template <int B>
cudaError_t launch_stack_b(const StackArgs &a, const StackPlan &p, const StackMaps &maps, cudaStream_t s) {
  if (a.g_gu != a.g_dn) return cudaErrorInvalidValue;
  switch (a.g_gu) {
    case 32: return launch_stack_t<B, 32, 32>(a, p, maps, s);
    case 64: return launch_stack_t<B, 64, 64>(a, p, maps, s);
    case 128: return launch_stack_t<B, 128, 128>(a, p, maps, s);
  }
  return cudaErrorInvalidValue;
}

// cuTensorMapEncodeTiled from the driver (looked up once).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// A 3-D byte view [z][y][x] of a packed buffer (x = inner bytes), boxes of bx x by x bz.
cudaError_t encode3(const void *base, uint64_t x, uint64_t y, uint64_t z, uint32_t by, uint32_t bz, CUtensorMap *out) {
  using Key = std::tuple<const void *, uint64_t, uint64_t, uint64_t, uint32_t, uint32_t>;
  static std::mutex mu;
  static std::map<Key, CUtensorMap> cache;
  const Key key{base, x, y, z, by, bz};
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *out = it->second;
    return cudaSuccess;
  }
  PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[3] = {x, y, z};
  const cuuint64_t strides[2] = {x, x * y};
  const cuuint32_t box[3] = {(cuuint32_t)x, by, bz};
  const cuuint32_t e1[3] = {1, 1, 1};
  if (fn(out, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void *>(base), dims, strides, box, e1,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  if (cache.size() > 65536) cache.clear();
  cache[key] = *out;
  return cudaSuccess;
}

}  // namespace

cudaError_t stack_layer_maps(const void *gate_codes, const void *up_codes, const void *gate_meta, const void *up_meta,
                             const void *down_codes, const void *down_meta, int d, int inter, int bits_gu, int group,
                             const StackPlan &p, CUtensorMap out[6]) {
  const uint64_t BPK = bits_gu == 2 ? 512 : 1024, GPB = 128 / group, GPH = group == 32 ? 2 : 1;
  const uint64_t RTg = (uint64_t)inter / 16, KBg = (uint64_t)d / 128, RTd = (uint64_t)d / 16, KBd = (uint64_t)inter / 128;
  const uint64_t NGd = KBd * 128 / group;
  cudaError_t e;
  if ((e = encode3(gate_codes, 128, KBg * BPK / 128, RTg, (uint32_t)(p.kps * BPK / 128), p.Tbox, &out[0])) != cudaSuccess ||
      (e = encode3(up_codes, 128, KBg * BPK / 128, RTg, (uint32_t)(p.kps * BPK / 128), p.Tbox, &out[1])) != cudaSuccess ||
      (e = encode3(gate_meta, 64, KBg * GPB, RTg, (uint32_t)p.gmy, p.Tbox, &out[2])) != cudaSuccess ||
      (e = encode3(up_meta, 64, KBg * GPB, RTg, (uint32_t)p.gmy, p.Tbox, &out[3])) != cudaSuccess ||
      (e = encode3(down_codes, 128, KBd * 8, RTd, 4, (uint32_t)p.RPS, &out[4])) != cudaSuccess ||
      (e = encode3(down_meta, 64, NGd, RTd, (uint32_t)GPH, (uint32_t)p.RPS, &out[5])) != cudaSuccess)
    return e;
  return cudaSuccess;
}

cudaError_t launch_stack(const StackArgs &a, const StackPlan &p, const StackMaps &maps, cudaStream_t s) {
  return a.bits_gu == 2 ? launch_stack_b<2>(a, p, maps, s) : launch_stack_b<4>(a, p, maps, s);
}

// Self-check of the bounded waits (no GPU fault, no hang): one CTA of the
// stack kernel's shape waits on an mbarrier that nothing arrives on, then at
// a grid barrier whose counter nothing advances; each wait gives up after its
// limit (kWaitLimitNs), records WQ_ERR_TIMEOUT in the status word and lets
// the kernel end, so the context stays usable.
__device__ unsigned long long g_wait_check_ctr = 0;

__global__ void __launch_bounds__(kSThreads) wait_check_kernel() {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
    abort_flag = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0)) record_timeout();  // phase 0 never completes
  __syncthreads();
  if (threadIdx.x < kSMathThreads) grid_wait(&g_wait_check_ctr, ld_acquire_u64(&g_wait_check_ctr) + 1, &abort_flag);
}

cudaError_t launch_wait_check(cudaStream_t s) {
  wait_check_kernel<<<1, kSThreads, 0, s>>>();
  return cudaGetLastError();
}

cudaError_t read_stack_status(int *status) {
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(status, g_stack_status, sizeof(int));
  if (e != cudaSuccess) return e;
  const int zero = 0;
  return cudaMemcpyToSymbol(g_stack_status, &zero, sizeof(int));
}

}  // namespace wq
