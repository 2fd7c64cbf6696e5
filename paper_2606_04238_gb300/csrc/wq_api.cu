// wq_api.cu -- the C ABI of include/wq.h: argument validation, workspace
// layout, launch sequencing.  Every check happens on the host before any
// launch; nothing here allocates device memory or synchronizes (except
// wq_device_status, which is documented to).
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <algorithm>
#include <mutex>
#include <string>

#include "wq.h"
#include "wq_internal.h"
#include "wq_launch.h"
#include "wq_stack.h"

using namespace wq;

namespace {

thread_local std::string g_last_error;

wq_status fail(wq_status st, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

wq_status ok() {
  g_last_error.clear();
  return WQ_OK;
}

wq_status cuda_fail(cudaError_t e, const char *what) {
  return fail(WQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool group_ok(int g) { return g == 32 || g == 64 || g == 128; }

int num_sms() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cached[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cached[dev] = v;
  }
  return cached[dev];
}

wq_status check_qweight(const wq_qweight *q, int bits, const char *name) {
  if (!q) return fail(WQ_ERR_ARG, "%s: null wq_qweight", name);
  if (!q->codes || !q->meta) return fail(WQ_ERR_ARG, "%s: null codes or meta pointer", name);
  if (!aligned16(q->codes) || !aligned16(q->meta)) return fail(WQ_ERR_ALIGN, "%s: codes/meta not 16-byte aligned", name);
  if (q->bits != bits) return fail(WQ_ERR_SHAPE, "%s: bits %d, expected %d", name, q->bits, bits);
  if (q->n <= 0 || q->k <= 0) return fail(WQ_ERR_SHAPE, "%s: bad shape [%d, %d]", name, q->n, q->k);
  if (!group_ok(q->group)) return fail(WQ_ERR_SHAPE, "%s: group %d not in {32, 64, 128}", name, q->group);
  if (q->k % q->group != 0) return fail(WQ_ERR_SHAPE, "%s: k=%d not a multiple of group %d", name, q->k, q->group);
  return WQ_OK;
}

// A stack layer's down matrix: 4-bit packed, or dense bf16 (bits 16: codes
// holds the bf16 [n, k] matrix, k a multiple of 32; meta unused).
wq_status check_down(const wq_qweight *q) {
  if (q && q->bits == 16) {
    if (!q->codes) return fail(WQ_ERR_ARG, "down: null bf16 matrix");
    if (!aligned16(q->codes)) return fail(WQ_ERR_ALIGN, "down: bf16 matrix not 16-byte aligned");
    if (q->n <= 0 || q->k <= 0 || q->k % 32 != 0) return fail(WQ_ERR_SHAPE, "down: bf16 shape [%d, %d] (k a multiple of 32)", q->n, q->k);
    return WQ_OK;
  }
  return check_qweight(q, 4, "down");
}

// Byte layout of the workspace for up to m tokens of a (d, inter) layer.
struct WsLayout {
  // arrival counters: at fixed offsets for every token count (zero once, kept
  // at zero -- or, for the stack kernel's, at a multiple of its grid -- by the calls)
  size_t cnt1, cnt2, sctr, sk_cnt;
  size_t tp, xa, xb, h, hq, hsc, hxs, part1, part2;
  // dequant-GEMM path (m > kMaxTokens, or a shape the GEMV path has no plan for)
  size_t x16, rs, ta, h16, hsx, sk_part;
  bool gemm;  // the GEMM buffers are laid out
  // single-launch stack (1..8 tokens)
  size_t sxw, stp, shg, spart, sxc;
  bool stack;
  size_t total;
};

size_t up256(size_t v) { return (v + 255) / 256 * 256; }

// Token count above which the calls take the dequant-GEMM path: 16, or 8 for
// layers of hidden size 4096 and more (measured on GB300: at 16 tokens the
// launch chain of the d 4096 and d 5120 stacks took 157 and 266 us a layer,
// the GEMM chain at 64 tokens 119 and 147 us; up to 8 tokens the single-launch
// stack kernel serves those shapes).
int gemv_prefer_tokens(int d) { return d >= 4096 ? 8 : kGemvPreferTokens; }

size_t partial_bytes(const GemvPlan &p, int nproj) {
  return p.P > 1 ? (size_t)p.RT * p.P * nproj * 16 * p.M * 4 : 0;
}

// Largest split-K partial buffer any plan of this shape can need (every
// group size and LoRA rank, including the down launch that writes the next
// layer's tile partials).
bool max_partials(int m, int d, int inter, size_t *p1, size_t *p2, bool *all_fit = nullptr) {
  const int sms = num_sms();
  if (sms <= 0) return false;
  *p1 = *p2 = 0;
  bool fit = true;
  const int groups[3] = {32, 64, 128};
  for (int g : groups) {
    for (int r = 0; r <= kMaxRank; r += 8) {
      GemvPlan pl;
      if (d % g == 0) {
        if (plan_gemv(kGateUpW2, inter, d, m, g, r, sms, &pl)) *p1 = std::max(*p1, partial_bytes(pl, 2));
        else fit = false;
        if (plan_gemv(kGateUpW3, inter, d, m, g, r, sms, &pl)) *p1 = std::max(*p1, partial_bytes(pl, 2));
        if (r == 0) {
          if (plan_gemv(kGateUpW4, inter, d, m, g, 0, sms, &pl)) *p1 = std::max(*p1, partial_bytes(pl, 2));
          else fit = false;
        }
      }
      if (inter % g == 0 && (r == 0 || d % 8 == 0)) {
        if (plan_gemv(kDownW4, d, inter, m, g, r, sms, &pl)) *p2 = std::max(*p2, partial_bytes(pl, 1));
        else fit = false;
      }
    }
  }
  if (all_fit) *all_fit = fit;
  return true;
}

// The counter block every layout starts with: the GEMV split-panel counters
// of gate/up and down, the stack kernel's grid-barrier counter and the
// stream-K tile counters of the GEMM path (sized for its largest token count).
size_t counter_block(int d, int inter, WsLayout *L) {
  size_t off = 0;
  L->cnt1 = off;   off = up256(off + (size_t)((inter + 15) / 16) * 4);
  L->cnt2 = off;   off = up256(off + (size_t)((d + 15) / 16) * 4);
  L->sctr = off;   off = up256(off + 8);
  const size_t cnt = std::max(gemm_counters(kMaxGemmTokens, inter), gemm_counters(kMaxGemmTokens, d));
  L->sk_cnt = off; off = up256(off + cnt * 4);
  return off;
}

// The dequant-GEMM buffers from offset `off`: binary16 copies of the GEMM
// inputs, RMSNorm scales, the LoRA-A products and the stream-K scratch.
bool gemm_layout(int m, int d, int inter, size_t off, WsLayout *L) {
  const size_t lda = (size_t)(std::max(d, inter) + 127) / 128 * 128, ldi = (size_t)(inter + 127) / 128 * 128;
  const int sms = num_sms();
  if (sms <= 0) return false;
  const size_t part = std::max(gemm_scratch_floats(m, inter, d, 2, sms), gemm_scratch_floats(m, d, inter, 1, sms));
  L->x16 = off;     off = up256(off + (size_t)m * lda * 2);
  L->rs = off;      off = up256(off + (size_t)m * 4);
  L->ta = off;      off = up256(off + (size_t)m * 2 * kMaxRank * 2);
  L->h16 = off;     off = up256(off + (size_t)m * ldi * 2);
  L->hsx = off;     off = up256(off + (size_t)m * 4);
  L->sk_part = off; off = up256(off + part * 4);
  L->gemm = true;
  L->total = off;
  return true;
}

// The single-launch stack's buffers from offset `off` (1..8 tokens of a
// shape it can take).
void stack_layout(int m, int d, int inter, size_t off, WsLayout *L) {
  if (m < 1 || m > 8 || d % 128 != 0 || inter % 64 != 0) return;
  const size_t Qp = WQ_TP_STRIDE(kMaxRank);
  L->sxw = off;   off = up256(off + (size_t)m * d * 2);
  L->stp = off;   off = up256(off + (size_t)(d / 16) * m * Qp * 4);
  L->shg = off;   off = up256(off + (size_t)m * inter * 2);
  L->spart = off; off = up256(off + (size_t)(inter / 64) * m * d * 4);
  L->sxc = off;   off = up256(off + (size_t)m * d * 2);
  L->stack = true;
  L->total = off;
}

// gemv_only: the decode path's buffers alone (the call without a workspace).
bool ws_layout(int m, int d, int inter, WsLayout *L, bool gemv_only = false) {
  *L = WsLayout{};
  size_t off = counter_block(d, inter, L);
  if (m > kMaxTokens) {
    // dequant-GEMM path: the stack's bf16 intermediates, then the GEMM buffers
    L->xa = off;  off = up256(off + (size_t)m * d * 2);
    L->xb = off;  off = up256(off + (size_t)m * d * 2);
    L->h = off;   off = up256(off + (size_t)m * inter * 2);
    return gemm_layout(m, d, inter, off, L);
  }
  size_t p1, p2;
  bool all_fit = true;
  if (!max_partials(m, d, inter, &p1, &p2, &all_fit)) return false;
  L->tp = off;   off = up256(off + (size_t)((d + 15) / 16) * m * WQ_TP_STRIDE(kMaxRank) * 4);
  L->xa = off;   off = up256(off + (size_t)m * d * 2);
  L->xb = off;   off = up256(off + (size_t)m * d * 2);
  L->h = off;    off = up256(off + (size_t)m * inter * 2);
  L->hq = off;   off = up256(off + (size_t)m * ((inter + 127) / 128) * 128 * 2);
  L->hsc = off;  off = up256(off + (size_t)((inter + 63) / 64) * m * 4);
  L->hxs = off;  off = up256(off + (size_t)((inter + 31) / 32) * m * 4);
  L->part1 = off; off = up256(off + p1);
  L->part2 = off; off = up256(off + p2);
  L->total = off;
  if (gemv_only) return true;
  // above gemv_prefer_tokens, or for a shape that lacks a GEMV plan for some
  // group or rank at this token count, the calls take the dequant-GEMM path
  if (m > gemv_prefer_tokens(d) || !all_fit) {
    if (!gemm_layout(m, d, inter, off, L)) return false;
    off = L->total;
  }
  stack_layout(m, d, inter, off, L);
  return true;
}


// Whether a call takes the dequant-GEMM path: above gemv_prefer_tokens (where
// it is the faster path on every measured layer shape; the GEMV kernels'
// work grows faster than linearly with the token count), or where the GEMV
// path has no launch plan.  The workspace holds the GEMM buffers then.
bool gateup_uses_gemm(GemvKind kind, int m, const wq_qweight *gate, int r) {
  if (kind == kGateUpW3) return false;  // the dequant-GEMM path takes 2- and 4-bit codes only
  if (m > gemv_prefer_tokens(gate->k)) return true;
  GemvPlan pl;
  return !plan_gemv(kind, gate->n, gate->k, m, gate->group, r, num_sms(), &pl);
}
bool down_uses_gemm(int m, const wq_qweight *down, int r_next) {
  if (m > gemv_prefer_tokens(down->n)) return true;
  GemvPlan pl;
  return !plan_gemv(kDownW4, down->n, down->k, m, down->group, r_next, num_sms(), &pl);
}

// gate/up (2-bit with LoRA, or 4-bit) for one layer.  tp_in: tile partials of
// x written by the previous launch (the stack's down kernel), or null to have
// them computed here from x when the RMSNorm or the adapter needs them.
// With make_hq (decode chain, plans checked by chain_panel_ok), h is also
// written as the down launch's ready binary16 panel in the workspace.
wq_status run_gateup(GemvKind kind, const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                     const void *lora_a, const void *lora_bg, const void *lora_bu, int r, float lora_scale,
                     unsigned flags, void *h, const float *tp_in, const WsLayout &L, uint8_t *ws, cudaStream_t s,
                     bool make_hq = false) {
  const int d = gate->k, inter = gate->n;
  const bool prenorm = (flags & WQ_PRENORM) != 0;
  GemvPlan plan;
  if (!plan_gemv(kind, inter, d, m, gate->group, r, num_sms(), &plan))
    return fail(WQ_ERR_UNSUPPORTED, "no launch configuration fits [%d x %d], m=%d, group %d", inter, d, m, gate->group);
  const bool need_tp = prenorm || r > 0;
  float *tp_ws = reinterpret_cast<float *>(ws + L.tp);
  const float *tp = tp_in;
  if (need_tp && !tp) {
    cudaError_t e = launch_tile_prep(x, m, d, lora_a, 2 * r, tp_ws, s, true);
    if (e != cudaSuccess) return cuda_fail(e, "tile-partials launch");
    tp = tp_ws;
  }
  GemvArgs a = {};
  a.act = x;
  a.M = m;
  a.K = d;
  a.N = inter;
  a.group = gate->group;
  a.codes[0] = gate->codes;
  a.codes[1] = up->codes;
  a.meta[0] = gate->meta;
  a.meta[1] = up->meta;
  a.tp = need_tp ? tp : nullptr;
  a.ntp = d / 16;
  a.prenorm = prenorm ? 1 : 0;
  a.lora_b[0] = lora_bg;
  a.lora_b[1] = lora_bu;
  a.r = r;
  a.lora_scale = lora_scale;
  a.out = h;
  if (make_hq) {
    a.hq_out = reinterpret_cast<uint16_t *>(ws + L.hq);
    a.hsc_out = reinterpret_cast<float *>(ws + L.hsc);
    a.hxs_out = reinterpret_cast<float *>(ws + L.hxs);
    a.hq_stride = (inter + 127) / 128 * 128;
    a.nb_hq = L.hsc - L.hq;
    a.nb_hsc = L.hxs - L.hsc;
    a.nb_hxs = (size_t)((inter + 31) / 32) * m * 4;
  }
  a.partials = reinterpret_cast<float *>(ws + L.part1);
  a.counters = reinterpret_cast<unsigned *>(ws + L.cnt1);
  size_t cb = 0, mb = 0;
  wq_packed_sizes(gate->bits, inter, d, gate->group, &cb, &mb);
  a.nb_codes[0] = a.nb_codes[1] = cb;
  a.nb_meta[0] = a.nb_meta[1] = mb;
  a.nb_lora_b[0] = a.nb_lora_b[1] = (size_t)inter * r * 2;
  a.nb_act = (size_t)m * d * 2;
  a.nb_tp = (size_t)(d / 16) * m * WQ_TP_STRIDE(r) * 4;
  a.nb_out = (size_t)m * inter * 2;
  a.nb_part = L.part2 - L.part1;
  a.nb_cnt = (size_t)((inter + 15) / 16) * 4;
  cudaError_t e = launch_gemv(kind, plan, a, s, true);
  if (e != cudaSuccess) return cuda_fail(e, "gate/up launch");
  return WQ_OK;
}

// down for one layer; with tp_out, also the next layer's tile partials of y
// (RMSNorm sums and, for r_next > 0, the products with its LoRA-A).
// With use_hq, the input is the ready binary16 panel the gate/up launch left
// in the workspace instead of h.
wq_status run_down(const void *h, int m, const wq_qweight *down, const void *residual, void *y, int y_f32,
                   const void *lora_a_next, int r_next, float *tp_out, const WsLayout &L, uint8_t *ws,
                   cudaStream_t s, bool use_hq = false) {
  const int rr = tp_out ? r_next : 0;
  GemvPlan plan;
  if (!plan_gemv(kDownW4, down->n, down->k, m, down->group, rr, num_sms(), &plan))
    return fail(WQ_ERR_UNSUPPORTED, "no launch configuration fits [%d x %d], m=%d", down->n, down->k, m);
  GemvArgs a = {};
  a.act = h;
  a.M = m;
  a.K = down->k;
  a.N = down->n;
  a.group = down->group;
  a.codes[0] = down->codes;
  a.meta[0] = down->meta;
  a.r = rr;
  a.residual = residual;
  a.out = y;
  a.out_f32 = y_f32;
  a.lora_a_next = rr > 0 ? lora_a_next : nullptr;
  a.tp_out = tp_out;
  if (use_hq) {
    a.pre_x = reinterpret_cast<const uint16_t *>(ws + L.hq);
    a.pre_sc = reinterpret_cast<const float *>(ws + L.hsc);
    a.pre_xs = reinterpret_cast<const float *>(ws + L.hxs);
    a.pre_stride = (down->k + 127) / 128 * 128;
    a.nb_pre_x = L.hsc - L.hq;
    a.nb_pre_sc = L.hxs - L.hsc;
    a.nb_pre_xs = (size_t)((down->k + 31) / 32) * m * 4;
  }
  a.partials = reinterpret_cast<float *>(ws + L.part2);
  a.counters = reinterpret_cast<unsigned *>(ws + L.cnt2);
  size_t cb = 0, mb = 0;
  wq_packed_sizes(4, down->n, down->k, down->group, &cb, &mb);
  a.nb_codes[0] = cb;
  a.nb_meta[0] = mb;
  a.nb_act = (size_t)m * down->k * 2;
  a.nb_res = residual ? (size_t)m * down->n * 2 : 0;
  a.nb_out = (size_t)m * down->n * (y_f32 ? 4 : 2);
  a.nb_an = (size_t)2 * rr * down->n * 2;
  a.nb_tp_out = tp_out ? (size_t)((down->n + 15) / 16) * m * WQ_TP_STRIDE(rr) * 4 : 0;
  a.nb_part = (L.gemm ? L.x16 : L.stack ? L.sxw : L.total) - L.part2;
  a.nb_cnt = (size_t)((down->n + 15) / 16) * 4;
  cudaError_t e = launch_gemv(kDownW4, plan, a, s, true);
  if (e != cudaSuccess) return cuda_fail(e, "down launch");
  return WQ_OK;
}

// ---- dequant-GEMM path (m > kMaxTokens): tcgen05 tensor cores ----
// gate/up: binary16 copy of x, RMSNorm scales and lora_scale * x A^T first,
// then the GEMM (h in bf16).
wq_status run_gateup_gemm(GemvKind kind, const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                          const void *lora_a, const void *lora_bg, const void *lora_bu, int r, float lora_scale,
                          unsigned flags, void *h, const WsLayout &L, uint8_t *ws, cudaStream_t s) {
  const int d = gate->k, inter = gate->n;
  const int lda = (d + 127) / 128 * 128;
  if (!L.gemm) return fail(WQ_ERR_WORKSPACE, "workspace laid out without the dequant-GEMM buffers");
  uint16_t *x16 = reinterpret_cast<uint16_t *>(ws + L.x16);
  float *rs = reinterpret_cast<float *>(ws + L.rs);
  uint16_t *ta = reinterpret_cast<uint16_t *>(ws + L.ta);
  cudaError_t e = launch_gemm_prep(x, m, d, lda, r > 0 ? lora_a : nullptr, r > 0 ? 2 * r : 0, lora_scale,
                                   (flags & WQ_PRENORM) ? 1 : 0, x16, rs, ta, s);
  if (e != cudaSuccess) return cuda_fail(e, "GEMM input launch");
  GemmArgs a = {};
  a.act = x16;
  a.lda = lda;
  a.M = m;
  a.N = inter;
  a.K = d;
  a.group = gate->group;
  a.codes[0] = gate->codes;
  a.codes[1] = up->codes;
  a.meta[0] = gate->meta;
  a.meta[1] = up->meta;
  a.ta = r > 0 ? ta : nullptr;
  a.r = r;
  a.lora_b[0] = lora_bg;
  a.lora_b[1] = lora_bu;
  a.rs = rs;
  a.out = h;
  a.sk_part = reinterpret_cast<float *>(ws + L.sk_part);
  a.sk_cnt = reinterpret_cast<unsigned *>(ws + L.sk_cnt);
  e = launch_gemm(kind, a, s);
  if (e != cudaSuccess) return cuda_fail(e, "gate/up GEMM launch");
  return WQ_OK;
}

// down: h converted to binary16 first (scaled per token), then the GEMM.
wq_status run_down_gemm(const void *h, int m, const wq_qweight *down, const void *residual,
                        void *y, int y_f32, const WsLayout &L, uint8_t *ws, cudaStream_t s) {
  if (!L.gemm) return fail(WQ_ERR_WORKSPACE, "workspace laid out without the dequant-GEMM buffers");
  const int K = down->k, lda = (K + 127) / 128 * 128;
  uint16_t *h16 = reinterpret_cast<uint16_t *>(ws + L.h16);
  float *hsx = reinterpret_cast<float *>(ws + L.hsx);
  cudaError_t e = launch_to_f16(h, m, K, lda, h16, hsx, s);
  if (e != cudaSuccess) return cuda_fail(e, "GEMM input launch");
  GemmArgs a = {};
  a.act = h16;
  a.lda = lda;
  a.M = m;
  a.N = down->n;
  a.K = K;
  a.group = down->group;
  a.codes[0] = down->codes;
  a.meta[0] = down->meta;
  a.residual = residual;
  a.rs = hsx;
  a.out = y;
  a.out_f32 = y_f32;
  a.sk_part = reinterpret_cast<float *>(ws + L.sk_part);
  a.sk_cnt = reinterpret_cast<unsigned *>(ws + L.sk_cnt);
  e = launch_gemm(kDownW4, a, s);
  if (e != cudaSuccess) return cuda_fail(e, "down GEMM launch");
  return WQ_OK;
}

// The gate/up launch can hand the down launch a ready binary16 panel when it
// holds whole 64-feature halves (one panel, row blocks of a multiple of 4
// tiles) and the down kernel scales its input per half (one row tile a warp).
bool chain_panel_ok(GemvKind kind, int m, const wq_qweight &gate, int r, const wq_qweight &down, int r_next) {
  GemvPlan pg, pd;
  if (!plan_gemv(kind, gate.n, gate.k, m, gate.group, r, num_sms(), &pg)) return false;
  if (!plan_gemv(kDownW4, down.n, down.k, m, down.group, r_next, num_sms(), &pd)) return false;
  return pg.P == 1 && pg.RB % 4 == 0 && pd.TPW == 1;
}

wq_status check_tokens(int m) {
  if (m < 0) return fail(WQ_ERR_ARG, "m=%d is negative", m);
  if (m > kMaxGemmTokens) return fail(WQ_ERR_UNSUPPORTED, "m=%d exceeds the %d-token limit of the library", m, kMaxGemmTokens);
  return WQ_OK;
}

wq_status check_ws(void *ws, size_t ws_bytes, int m, int d, int inter, WsLayout *L) {
  if (!ws_layout(m, d, inter, L)) return fail(WQ_ERR_CUDA, "cannot query the current device");
  if (!ws) return fail(WQ_ERR_WORKSPACE, "null workspace");
  if (!aligned16(ws)) return fail(WQ_ERR_ALIGN, "workspace not 16-byte aligned");
  if (ws_bytes < L->total)
    return fail(WQ_ERR_WORKSPACE, "workspace of %zu bytes, %zu needed (wq_workspace_bytes)", ws_bytes, L->total);
  return WQ_OK;
}

wq_status check_lora(const void *lora_a, const void *bg, const void *bu, int r) {
  if (r == 0) return WQ_OK;
  if (r < 0 || r % 8 != 0 || r > kMaxRank) return fail(WQ_ERR_SHAPE, "LoRA rank %d not a multiple of 8 in [8, 64]", r);
  if (!lora_a || !bg || !bu) return fail(WQ_ERR_ARG, "null LoRA pointer with r=%d", r);
  if (!aligned16(lora_a) || !aligned16(bg) || !aligned16(bu)) return fail(WQ_ERR_ALIGN, "LoRA pointers not 16-byte aligned");
  return WQ_OK;
}

wq_status check_gateup_pair(const wq_qweight *gate, const wq_qweight *up, int bits) {
  wq_status st = check_qweight(gate, bits, "gate");
  if (st != WQ_OK) return st;
  if ((st = check_qweight(up, bits, "up")) != WQ_OK) return st;
  if (gate->n != up->n || gate->k != up->k || gate->group != up->group)
    return fail(WQ_ERR_SHAPE, "gate [%d x %d g%d] and up [%d x %d g%d] differ", gate->n, gate->k, gate->group, up->n,
                up->k, up->group);
  return WQ_OK;
}

wq_status gateup_entry(GemvKind kind, const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                       const void *lora_a, const void *bg, const void *bu, int r, float lora_scale, unsigned flags,
                       void *h, void *ws, size_t ws_bytes, void *stream) {
  wq_status st = check_tokens(m);
  if (st != WQ_OK) return st;
  if ((st = check_gateup_pair(gate, up, kind == kGateUpW2 ? 2 : kind == kGateUpW3 ? 3 : 4)) != WQ_OK) return st;
  if (kind == kGateUpW3 && m > kMaxTokens)
    return fail(WQ_ERR_UNSUPPORTED, "3-bit gate/up above %d tokens (the dequant-GEMM path takes 2- and 4-bit codes)",
                kMaxTokens);
  if ((st = check_lora(lora_a, bg, bu, r)) != WQ_OK) return st;
  if (flags & ~WQ_PRENORM) return fail(WQ_ERR_ARG, "unknown flags 0x%x", flags);
  if (m == 0) return ok();
  if (!x || !h) return fail(WQ_ERR_ARG, "null x or h");
  if (!aligned16(x) || !aligned16(h)) return fail(WQ_ERR_ALIGN, "x or h not 16-byte aligned");
  WsLayout L;
  if ((st = check_ws(ws, ws_bytes, m, gate->k, gate->n, &L)) != WQ_OK) return st;
  if (gateup_uses_gemm(kind, m, gate, r))
    st = run_gateup_gemm(kind, x, m, gate, up, lora_a, bg, bu, r, lora_scale, flags, h, L,
                         static_cast<uint8_t *>(ws), static_cast<cudaStream_t>(stream));
  else
    st = run_gateup(kind, x, m, gate, up, lora_a, bg, bu, r, lora_scale, flags, h, nullptr, L,
                    static_cast<uint8_t *>(ws), static_cast<cudaStream_t>(stream));
  return st == WQ_OK ? ok() : st;
}

}  // namespace

extern "C" {

wq_status wq_packed_sizes(int bits, int n, int k, int group, size_t *code_bytes, size_t *meta_bytes) {
  if (bits < 2 || bits > 4) return fail(WQ_ERR_SHAPE, "bits %d not in {2, 3, 4}", bits);
  if (!group_ok(group)) return fail(WQ_ERR_SHAPE, "group %d not in {32, 64, 128}", group);
  if (n < 0 || k < 0 || k % group != 0) return fail(WQ_ERR_SHAPE, "bad shape [%d, %d] for group %d", n, k, group);
  const size_t RT = (size_t)(n + 15) / 16, KB = (size_t)(k + 127) / 128;
  if (code_bytes) *code_bytes = RT * KB * 256 * bits;
  if (meta_bytes) *meta_bytes = RT * (KB * 128 / group) * 64;
  return ok();
}

wq_status wq_pack(const float *w, int n, int k, int group, int bits, wq_qweight *out, int *nonfinite, void *stream) {
  size_t cb, mb;
  wq_status st = wq_packed_sizes(bits, n, k, group, &cb, &mb);
  if (st != WQ_OK) return st;
  if (!out) return fail(WQ_ERR_ARG, "null output wq_qweight");
  if (n == 0 || k == 0) return fail(WQ_ERR_SHAPE, "empty matrix [%d, %d]", n, k);
  if (!w || !out->codes || !out->meta) return fail(WQ_ERR_ARG, "null weight, codes or meta pointer");
  if (!aligned16(w) || !aligned16(out->codes) || !aligned16(out->meta))
    return fail(WQ_ERR_ALIGN, "weight, codes or meta pointer not 16-byte aligned");
  cudaError_t e = launch_pack(w, n, k, group, bits, out->codes, out->meta, nonfinite, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "pack launch");
  out->n = n;
  out->k = k;
  out->group = group;
  out->bits = bits;
  return ok();
}

wq_status wq_pack_w2(const float *w, int n, int k, int group, wq_qweight *out, int *nonfinite, void *stream) {
  return wq_pack(w, n, k, group, 2, out, nonfinite, stream);
}

wq_status wq_pack_w4(const float *w, int n, int k, int group, wq_qweight *out, int *nonfinite, void *stream) {
  return wq_pack(w, n, k, group, 4, out, nonfinite, stream);
}

wq_status wq_merge_lora(const wq_qweight *src, const void *lora_b, const void *lora_a, int r, float lora_scale,
                        float *w_merged, wq_qweight *out, int *nonfinite, void *stream) {
  if (!src) return fail(WQ_ERR_ARG, "src: null wq_qweight");
  if (src->bits < 2 || src->bits > 4) return fail(WQ_ERR_SHAPE, "src: bits %d not in {2, 3, 4}", src->bits);
  wq_status st = check_qweight(src, src->bits, "src");
  if (st != WQ_OK) return st;
  if (r < 0 || r > kMaxRank) return fail(WQ_ERR_SHAPE, "LoRA rank %d not in [0, %d]", r, kMaxRank);
  if (r > 0 && (!lora_a || !lora_b)) return fail(WQ_ERR_ARG, "null LoRA pointer with r=%d", r);
  if ((reinterpret_cast<uintptr_t>(lora_a) | reinterpret_cast<uintptr_t>(lora_b)) & 1u)
    return fail(WQ_ERR_ALIGN, "LoRA pointers not 2-byte aligned");
  if (!std::isfinite(lora_scale)) return fail(WQ_ERR_ARG, "lora_scale is not finite");
  if (!out) return fail(WQ_ERR_ARG, "null output wq_qweight");
  if (!w_merged || !out->codes || !out->meta) return fail(WQ_ERR_ARG, "null w_merged, codes or meta pointer");
  if (!aligned16(w_merged) || !aligned16(out->codes) || !aligned16(out->meta))
    return fail(WQ_ERR_ALIGN, "w_merged, codes or meta pointer not 16-byte aligned");
  const wq_qweight s = *src;  // out may be src itself
  const cudaStream_t cs = static_cast<cudaStream_t>(stream);
  cudaError_t e = launch_merge_lora(static_cast<const uint32_t *>(s.codes), static_cast<const uint16_t *>(s.meta),
                                    s.n, s.k, s.group, s.bits, lora_b, lora_a, r, lora_scale, w_merged, cs);
  if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  e = launch_pack(w_merged, s.n, s.k, s.group, s.bits, static_cast<uint32_t *>(out->codes),
                  static_cast<uint16_t *>(out->meta), nonfinite, cs);
  if (e != cudaSuccess) return cuda_fail(e, "pack launch");
  out->n = s.n;
  out->k = s.k;
  out->group = s.group;
  out->bits = s.bits;
  return ok();
}

size_t wq_workspace_bytes(int m, int d, int inter, int r) {
  (void)r;  // the LoRA-A product area is sized for the largest supported rank
  if (m <= 0 || d <= 0 || inter <= 0 || m > kMaxGemmTokens) return 0;
  size_t most = 0;  // enough for every token count up to m
  if (m > kMaxTokens) {
    WsLayout L;
    if (!ws_layout(m, d, inter, &L)) return 0;  // grows with m
    most = L.total;
  }
  for (int mm = 1; mm <= std::min(m, kMaxTokens); ++mm) {
    WsLayout L;
    if (!ws_layout(mm, d, inter, &L)) return 0;
    most = std::max(most, L.total);
  }
  return most;
}

wq_status wq_workspace_init(void *ws, size_t ws_bytes, void *stream) {
  if (!ws) return fail(WQ_ERR_WORKSPACE, "null workspace");
  cudaError_t e = cudaMemsetAsync(ws, 0, ws_bytes, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "workspace clear");
  return ok();
}

wq_status wq_gateup_w2_lora(const void *x, int m, const wq_qweight *gate, const wq_qweight *up, const void *lora_a,
                            const void *lora_b_gate, const void *lora_b_up, int r, float lora_scale, unsigned flags,
                            void *h, void *ws, size_t ws_bytes, void *stream) {
  return gateup_entry(kGateUpW2, x, m, gate, up, lora_a, lora_b_gate, lora_b_up, r, lora_scale, flags, h, ws, ws_bytes,
                      stream);
}

wq_status wq_gateup_w3_lora(const void *x, int m, const wq_qweight *gate, const wq_qweight *up, const void *lora_a,
                            const void *lora_b_gate, const void *lora_b_up, int r, float lora_scale, unsigned flags,
                            void *h, void *ws, size_t ws_bytes, void *stream) {
  return gateup_entry(kGateUpW3, x, m, gate, up, lora_a, lora_b_gate, lora_b_up, r, lora_scale, flags, h, ws, ws_bytes,
                      stream);
}

}  // extern "C"

namespace {

// Scratch of wq_gateup_w2_lora_noalloc: a fixed array in the library's device
// code, so the call never allocates.  Its device address is looked up once per
// device (host code only sees a stand-in for the symbol, not the address).
static __device__ __align__(256) uint8_t g_noalloc_scratch[WQ_NOALLOC_SCRATCH_BYTES];
std::mutex g_noalloc_mu;
void *g_noalloc_base[64] = {};

wq_status noalloc_scratch(void **base) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(WQ_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_base[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the built-in scratch");
    g_noalloc_base[dev] = p;
  }
  *base = g_noalloc_base[dev];
  return WQ_OK;
}

}  // namespace

extern "C" {

wq_status wq_gateup_w2_lora_noalloc(const void *x, int m, const wq_qweight *gate, const wq_qweight *up,
                                    const void *lora_a, const void *lora_b_gate, const void *lora_b_up, int r,
                                    float lora_scale, unsigned flags, void *h, void *stream) {
  wq_status st = check_tokens(m);
  if (st != WQ_OK) return st;
  if ((st = check_gateup_pair(gate, up, 2)) != WQ_OK) return st;
  if ((st = check_lora(lora_a, lora_b_gate, lora_b_up, r)) != WQ_OK) return st;
  if (flags & ~WQ_PRENORM) return fail(WQ_ERR_ARG, "unknown flags 0x%x", flags);
  if (m == 0) return ok();
  if (!x || !h) return fail(WQ_ERR_ARG, "null x or h");
  if (!aligned16(x) || !aligned16(h)) return fail(WQ_ERR_ALIGN, "x or h not 16-byte aligned");
  if (m > gemv_prefer_tokens(gate->k))
    return fail(WQ_ERR_UNSUPPORTED, "m=%d: the built-in scratch serves the decode path (m <= %d here; use wq_gateup_w2_lora)",
                m, gemv_prefer_tokens(gate->k));
  GemvPlan plan;
  if (!plan_gemv(kGateUpW2, gate->n, gate->k, m, gate->group, r, num_sms(), &plan))
    return fail(WQ_ERR_UNSUPPORTED,
                "no decode launch configuration fits [%d x %d], m=%d, group %d (use wq_gateup_w2_lora, which can take "
                "the dequant-GEMM path)", gate->n, gate->k, m, gate->group);
  WsLayout L;
  if (!ws_layout(m, gate->k, gate->n, &L, true)) return fail(WQ_ERR_CUDA, "cannot query the current device");
  if (L.total > (size_t)WQ_NOALLOC_SCRATCH_BYTES)
    return fail(WQ_ERR_UNSUPPORTED, "this layer needs %zu bytes of scratch; the built-in scratch holds %u (use wq_gateup_w2_lora)",
                L.total, (unsigned)WQ_NOALLOC_SCRATCH_BYTES);
  void *base = nullptr;
  if ((st = noalloc_scratch(&base)) != WQ_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the arrival counters must start at zero
  cudaError_t e = cudaMemsetAsync(static_cast<uint8_t *>(base) + L.cnt1, 0, L.tp - L.cnt1, s);
  if (e != cudaSuccess) return cuda_fail(e, "clearing the built-in scratch counters");
  st = run_gateup(kGateUpW2, x, m, gate, up, lora_a, lora_b_gate, lora_b_up, r, lora_scale, flags, h, nullptr, L,
                  static_cast<uint8_t *>(base), s);
  return st == WQ_OK ? ok() : st;
}

wq_status wq_gateup_w4(const void *x, int m, const wq_qweight *gate, const wq_qweight *up, unsigned flags, void *h,
                       void *ws, size_t ws_bytes, void *stream) {
  return gateup_entry(kGateUpW4, x, m, gate, up, nullptr, nullptr, nullptr, 0, 0.f, flags, h, ws, ws_bytes, stream);
}

wq_status wq_down_w4(const void *h, int m, const wq_qweight *down, const void *residual, void *y, int y_dtype, void *ws,
                     size_t ws_bytes, void *stream) {
  wq_status st = check_tokens(m);
  if (st != WQ_OK) return st;
  if ((st = check_qweight(down, 4, "down")) != WQ_OK) return st;
  if (y_dtype != WQ_BF16 && y_dtype != WQ_F32) return fail(WQ_ERR_ARG, "y_dtype %d not WQ_BF16 or WQ_F32", y_dtype);
  if (m == 0) return ok();
  if (!h || !y) return fail(WQ_ERR_ARG, "null h or y");
  if (!aligned16(h) || !aligned16(y) || (residual && !aligned16(residual)))
    return fail(WQ_ERR_ALIGN, "h, y or residual not 16-byte aligned");
  WsLayout L;
  if ((st = check_ws(ws, ws_bytes, m, down->n, down->k, &L)) != WQ_OK) return st;
  if (down_uses_gemm(m, down, 0))
    st = run_down_gemm(h, m, down, residual, y, y_dtype == WQ_F32, L, static_cast<uint8_t *>(ws),
                       static_cast<cudaStream_t>(stream));
  else
    st = run_down(h, m, down, residual, y, y_dtype == WQ_F32, nullptr, 0, nullptr, L, static_cast<uint8_t *>(ws),
                  static_cast<cudaStream_t>(stream));
  return st == WQ_OK ? ok() : st;
}

wq_status wq_down_bf16(const void *h, int m, const void *wd, int d, int inter, const void *residual, void *y,
                       int y_dtype, void *stream) {
  wq_status st = check_tokens(m);
  if (st != WQ_OK) return st;
  if (d <= 0 || inter <= 0 || inter % 32 != 0)
    return fail(WQ_ERR_SHAPE, "bad shape d=%d, inter=%d (inter a positive multiple of 32)", d, inter);
  if (y_dtype != WQ_BF16 && y_dtype != WQ_F32) return fail(WQ_ERR_ARG, "y_dtype %d not WQ_BF16 or WQ_F32", y_dtype);
  if (m == 0) return ok();
  if (!h || !wd || !y) return fail(WQ_ERR_ARG, "null h, wd or y");
  if (!aligned16(h) || !aligned16(wd) || !aligned16(y) || (residual && !aligned16(residual)))
    return fail(WQ_ERR_ALIGN, "h, wd, y or residual not 16-byte aligned");
  cudaError_t e = launch_down_bf16(h, m, wd, d, inter, residual, y, y_dtype == WQ_F32,
                                   static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "bf16 down launch");
  return ok();
}

}  // extern "C"

namespace {

// Validates a stack and fills in its shape (d, inter).
wq_status check_stack(int m, const wq_mlp_layer *layers, int n_layers, unsigned flags, int *d_out, int *inter_out) {
  wq_status st = check_tokens(m);
  if (st != WQ_OK) return st;
  if (n_layers < 0) return fail(WQ_ERR_ARG, "n_layers=%d is negative", n_layers);
  if (n_layers > 0 && !layers) return fail(WQ_ERR_ARG, "null layer array");
  if (flags & ~(WQ_PRENORM | WQ_LAUNCH_CHAIN | WQ_LAUNCH_STACK)) return fail(WQ_ERR_ARG, "unknown flags 0x%x", flags);
  if ((flags & WQ_LAUNCH_CHAIN) && (flags & WQ_LAUNCH_STACK))
    return fail(WQ_ERR_ARG, "WQ_LAUNCH_CHAIN and WQ_LAUNCH_STACK together");
  int d = 0, inter = 0;
  for (int l = 0; l < n_layers; ++l) {
    const wq_mlp_layer &Ly = layers[l];
    const int bits = Ly.gate.bits;
    if (bits < 2 || bits > 4) return fail(WQ_ERR_SHAPE, "layer %d: gate bits %d not in {2, 3, 4}", l, bits);
    if (bits == 3 && m > kMaxTokens)
      return fail(WQ_ERR_UNSUPPORTED, "layer %d: 3-bit gate/up above %d tokens (the dequant-GEMM path takes 2- and "
                  "4-bit codes)", l, kMaxTokens);
    if ((st = check_gateup_pair(&Ly.gate, &Ly.up, bits)) != WQ_OK) return fail(st, "layer %d: %s", l, g_last_error.c_str());
    if ((st = check_down(&Ly.down)) != WQ_OK) return fail(st, "layer %d: %s", l, g_last_error.c_str());
    if (bits == 4 && Ly.r != 0) return fail(WQ_ERR_UNSUPPORTED, "layer %d: LoRA on 4-bit gate/up is not supported", l);
    if ((st = check_lora(Ly.lora_a, Ly.lora_b_gate, Ly.lora_b_up, Ly.r)) != WQ_OK)
      return fail(st, "layer %d: %s", l, g_last_error.c_str());
    if (Ly.down.n != Ly.gate.k || Ly.down.k != Ly.gate.n)
      return fail(WQ_ERR_SHAPE, "layer %d: down [%d x %d] does not match gate/up [%d x %d]", l, Ly.down.n, Ly.down.k,
                  Ly.gate.n, Ly.gate.k);
    if (l == 0) {
      d = Ly.gate.k;
      inter = Ly.gate.n;
    } else if (Ly.gate.k != d || Ly.gate.n != inter) {
      return fail(WQ_ERR_SHAPE, "layer %d: shape [%d x %d] differs from layer 0 [%d x %d]", l, Ly.gate.n, Ly.gate.k,
                  inter, d);
    }
  }
  *d_out = d;
  *inter_out = inter;
  return WQ_OK;
}

// How a stack runs: the per-layer dequant-GEMV launch chain, the
// dequant-GEMM launch chain (every layer's launches need a GEMV plan for the
// first; above gemv_prefer_tokens tokens the second), or the single-launch
// stack kernel (1..8 tokens, every layer with the same bits, groups and rank,
// unless the caller asks for the chain).
enum StackRoute { kRouteGemvChain = 0, kRouteGemmChain = 1, kRouteStack = 2 };

bool cooperative_ok() {
  static int cached[64] = {0};  // 0 unknown, 1 yes, -1 no
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (cached[dev] == 0) {
    int v = 0;
    cached[dev] = cudaDeviceGetAttribute(&v, cudaDevAttrCooperativeLaunch, dev) == cudaSuccess && v ? 1 : -1;
  }
  return cached[dev] > 0;
}

bool stack_kernel_plan(int m, const wq_mlp_layer *layers, int n_layers, unsigned flags, StackPlan *plan) {
  if ((flags & WQ_LAUNCH_CHAIN) || m < 1 || m > 8 || n_layers < 1) return false;
  const wq_mlp_layer &L0 = layers[0];
  for (int l = 0; l < n_layers; ++l) {
    const wq_mlp_layer &Ly = layers[l];
    if (Ly.gate.bits != L0.gate.bits || Ly.gate.group != L0.gate.group || Ly.down.group != L0.down.group ||
        Ly.r != L0.r || Ly.down.bits != 4)
      return false;
  }
  if (!cooperative_ok()) return false;
  return stack_plan(m, L0.gate.k, L0.gate.n, L0.r, L0.gate.bits, L0.gate.group, L0.down.group, num_sms(), plan);
}

// Where the stack kernel is the measured-faster route (GB300, CUDA-graph
// replays of whole stacks, us per layer, stack kernel vs launch chain):
//   2-bit gate/up, d 2560 / inter 9728: m=1 18.5 vs 16.7, m=2 20.1 vs 23.1,
//     m=4 22.9 vs 24.2, m=8 29.2 vs 29.5;
//   d 4096 / inter 14336: m=1 33.0 vs 41.6, m=4 44.1 vs 61.5, m=8 68.8 vs 87.2;
//   d 5120 / inter 17408: m=1 48.7 vs 52.6, m=4 80.1 vs 76.8, m=8 104.1 vs 132.9;
//   4-bit gate/up, d 2560: m=1 20.9 vs 18.0, m=4 23.6 vs 22.5, m=8 28.0 vs 25.9.
bool stack_preferred(int m, const wq_mlp_layer &L0) { return L0.gate.bits == 2 && (m >= 2 || L0.gate.k >= 4096); }

StackRoute stack_route(int m, const wq_mlp_layer *layers, int n_layers, unsigned flags) {
  StackPlan sp;
  if (((flags & WQ_LAUNCH_STACK) || stack_preferred(m, layers[0])) && stack_kernel_plan(m, layers, n_layers, flags, &sp))
    return kRouteStack;
  for (int l = 0; l < n_layers; ++l)
    if (layers[l].gate.bits == 3) return kRouteGemvChain;  // 3-bit codes run on the GEMV kernels only
  if (m > gemv_prefer_tokens(layers[0].gate.k)) return kRouteGemmChain;
  for (int l = 0; l < n_layers; ++l) {
    const wq_mlp_layer &Ly = layers[l];
    const bool next_tp = l + 1 < n_layers && ((flags & WQ_PRENORM) || layers[l + 1].r > 0);
    if (gateup_uses_gemm(gateup_kind(Ly.gate.bits), m, &Ly.gate, Ly.r) ||
        (Ly.down.bits == 4 && down_uses_gemm(m, &Ly.down, next_tp ? layers[l + 1].r : 0)))
      return kRouteGemmChain;
  }
  return kRouteGemvChain;
}

// wq_mlp_forward, with every layer's output also stored in `states`
// (bf16 [n_layers][m][d]) when it is not null.
wq_status mlp_forward_impl(const void *x, int m, const wq_mlp_layer *layers, int n_layers, unsigned flags, void *y,
                           void *states, void *h_states, void *ws, size_t ws_bytes, void *stream) {
  int d = 0, inter = 0;
  wq_status st = check_stack(m, layers, n_layers, flags, &d, &inter);
  if (st != WQ_OK) return st;
  if (m == 0 || n_layers == 0) {
    if (n_layers == 0 && m > 0 && x != y) return fail(WQ_ERR_ARG, "n_layers=0 needs y == x");
    return ok();
  }
  if (!x || !y) return fail(WQ_ERR_ARG, "null x or y");
  if (!aligned16(x) || !aligned16(y) || (states && !aligned16(states)) || (h_states && !aligned16(h_states)))
    return fail(WQ_ERR_ALIGN, "x, y, states or h_states not 16-byte aligned");
  WsLayout L;
  if ((st = check_ws(ws, ws_bytes, m, d, inter, &L)) != WQ_OK) return st;
  uint8_t *w8 = static_cast<uint8_t *>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t state_bytes = (size_t)m * d * 2;
  // output of layer l: the caller's state slot, y for the last layer, else a ping-pong buffer
  auto layer_out = [&](int l) -> void * {
    if (states) return static_cast<uint8_t *>(states) + (size_t)l * state_bytes;
    return (l == n_layers - 1) ? y : (void *)(w8 + ((l & 1) ? L.xb : L.xa));
  };
  // h of layer l: the caller's slot, else the workspace buffer
  auto layer_h = [&](int l) -> void * {
    return h_states ? static_cast<uint8_t *>(h_states) + (size_t)l * m * inter * 2 : (void *)(w8 + L.h);
  };
  auto finish = [&]() -> wq_status {
    if (states) {
      cudaError_t e = cudaMemcpyAsync(y, static_cast<uint8_t *>(states) + (size_t)(n_layers - 1) * state_bytes,
                                      state_bytes, cudaMemcpyDeviceToDevice, s);
      if (e != cudaSuccess) return cuda_fail(e, "copy of the last state to y");
    }
    return ok();
  };
  const StackRoute route = stack_route(m, layers, n_layers, flags);
  if (route == kRouteStack) {
    StackPlan sp;
    if (!stack_kernel_plan(m, layers, n_layers, flags, &sp) || !L.stack)
      return fail(WQ_ERR_UNSUPPORTED, "single-launch stack: no plan or workspace layout");
    // launches of up to kStackMaxLayers layers; each takes x_in and gives y_out
    const void *cur = x;
    for (int l0 = 0; l0 < n_layers; l0 += kStackMaxLayers) {
      const int nl = std::min(kStackMaxLayers, n_layers - l0);
      const bool last_launch = l0 + nl == n_layers;
      StackArgs a = {};
      a.M = m;
      a.d = d;
      a.inter = inter;
      a.r = layers[0].r;
      a.g_gu = layers[0].gate.group;
      a.g_dn = layers[0].down.group;
      a.bits_gu = layers[0].gate.bits;
      a.n_layers = nl;
      a.prenorm = (flags & WQ_PRENORM) ? 1 : 0;
      a.x_in = static_cast<const uint16_t *>(cur);
      a.y_out = reinterpret_cast<uint16_t *>(last_launch ? static_cast<uint8_t *>(y) : w8 + L.sxc);
      a.states = states ? reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(states) + (size_t)l0 * state_bytes) : nullptr;
      a.h_states = h_states ? reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(h_states) + (size_t)l0 * m * inter * 2)
                            : nullptr;
      a.xw = reinterpret_cast<uint16_t *>(w8 + L.sxw);
      a.tp = reinterpret_cast<float *>(w8 + L.stp);
      a.hg = reinterpret_cast<uint16_t *>(w8 + L.shg);
      a.part = reinterpret_cast<float *>(w8 + L.spart);
      a.ctr = reinterpret_cast<unsigned long long *>(w8 + L.sctr);
      static thread_local StackMaps maps;  // 24 KB: kept off the stack
      for (int l = 0; l < nl; ++l) {
        const wq_mlp_layer &Ly = layers[l0 + l];
        StackLayerDev &D = a.L[l];
        D.lora_a = static_cast<const uint16_t *>(Ly.lora_a);
        D.lora_b[0] = static_cast<const uint16_t *>(Ly.lora_b_gate);
        D.lora_b[1] = static_cast<const uint16_t *>(Ly.lora_b_up);
        D.lora_scale = Ly.lora_scale;
        cudaError_t e = stack_layer_maps(Ly.gate.codes, Ly.up.codes, Ly.gate.meta, Ly.up.meta, Ly.down.codes,
                                         Ly.down.meta, d, inter, Ly.gate.bits, Ly.gate.group, sp, maps.m[l]);
        if (e != cudaSuccess) return cuda_fail(e, "tensor maps of the stack's weights");
      }
      cudaError_t e = launch_stack(a, sp, maps, s);
      if (e != cudaSuccess) return cuda_fail(e, "single-launch stack");
      cur = a.y_out;
    }
    return ok();
  }
  if (route == kRouteGemmChain) {
    // dequant-GEMM chain: per layer the GEMM inputs of x, gate/up, the
    // binary16 copy of h (scaled per token), down with the residual
    const void *cur = x;
    for (int l = 0; l < n_layers; ++l) {
      const wq_mlp_layer &Ly = layers[l];
      void *out = layer_out(l);
      const GemvKind kind = gateup_kind(Ly.gate.bits);
      st = run_gateup_gemm(kind, cur, m, &Ly.gate, &Ly.up, Ly.lora_a, Ly.lora_b_gate, Ly.lora_b_up, Ly.r, Ly.lora_scale,
                           flags, layer_h(l), L, w8, s);
      if (st != WQ_OK) return fail(st, "layer %d: %s", l, g_last_error.c_str());
      if (Ly.down.bits == 16) {
        cudaError_t e = launch_down_bf16(layer_h(l), m, Ly.down.codes, d, inter, cur, out, false, s);
        if (e != cudaSuccess) return cuda_fail(e, "bf16 down launch");
      } else {
        st = run_down_gemm(layer_h(l), m, &Ly.down, cur, out, 0, L, w8, s);
        if (st != WQ_OK) return fail(st, "layer %d: %s", l, g_last_error.c_str());
      }
      cur = out;
    }
    return finish();
  }
  const bool prenorm = (flags & WQ_PRENORM) != 0;
  float *tp = reinterpret_cast<float *>(w8 + L.tp);
  // Launch chain (programmatic dependent launch throughout): the first
  // layer's tile partials from x, then per layer gate/up -> down, each down
  // also writing the next layer's tile partials of its output.
  if (prenorm || layers[0].r > 0) {
    cudaError_t e = launch_tile_prep(x, m, d, layers[0].lora_a, 2 * layers[0].r, tp, s, true);
    if (e != cudaSuccess) return cuda_fail(e, "tile-partials launch");
  }
  const void *cur = x;
  bool tp_ready = true;  // the tile partials of cur are in tp (from tile_prep or the previous down launch)
  for (int l = 0; l < n_layers; ++l) {
    const wq_mlp_layer &Ly = layers[l];
    void *out = layer_out(l);
    void *hbuf = layer_h(l);
    const GemvKind kind = gateup_kind(Ly.gate.bits);
    const bool need_tp = prenorm || Ly.r > 0;
    const wq_mlp_layer *nx = l + 1 < n_layers ? &layers[l + 1] : nullptr;
    const bool dense_down = Ly.down.bits == 16;
    const bool next_tp = nx && (prenorm || nx->r > 0) && !dense_down;
    const int r_next = next_tp ? nx->r : 0;
    const bool panel = !dense_down && chain_panel_ok(kind, m, Ly.gate, Ly.r, Ly.down, r_next);
    // after a bf16 down (which writes no tile partials) the gate/up launch
    // computes its input's partials itself
    st = run_gateup(kind, cur, m, &Ly.gate, &Ly.up, Ly.lora_a, Ly.lora_b_gate, Ly.lora_b_up, Ly.r, Ly.lora_scale, flags,
                    hbuf, need_tp && tp_ready ? tp : nullptr, L, w8, s, panel);
    if (st != WQ_OK) return fail(st, "layer %d: %s", l, g_last_error.c_str());
    if (dense_down) {
      cudaError_t e = launch_down_bf16(hbuf, m, Ly.down.codes, d, inter, cur, out, false, s);
      if (e != cudaSuccess) return cuda_fail(e, "bf16 down launch");
    } else {
      st = run_down(hbuf, m, &Ly.down, cur, out, 0, next_tp ? nx->lora_a : nullptr, r_next, next_tp ? tp : nullptr, L,
                    w8, s, panel);
      if (st != WQ_OK) return fail(st, "layer %d: %s", l, g_last_error.c_str());
    }
    tp_ready = next_tp;
    cur = out;
  }
  return finish();
}

}  // namespace

extern "C" {

wq_status wq_mlp_forward(const void *x, int m, const wq_mlp_layer *layers, int n_layers, unsigned flags, void *y,
                         void *ws, size_t ws_bytes, void *stream) {
  return mlp_forward_impl(x, m, layers, n_layers, flags, y, nullptr, nullptr, ws, ws_bytes, stream);
}

wq_status wq_mlp_forward_states(const void *x, int m, const wq_mlp_layer *layers, int n_layers, unsigned flags,
                                void *y, void *states, void *h_states, void *ws, size_t ws_bytes, void *stream) {
  if (!states && n_layers > 0 && m > 0) return fail(WQ_ERR_ARG, "null states");
  return mlp_forward_impl(x, m, layers, n_layers, flags, y, states, h_states, ws, ws_bytes, stream);
}

wq_status wq_mlp_forward_info(int m, const wq_mlp_layer *layers, int n_layers, unsigned flags, int64_t info[16]) {
  if (!info) return fail(WQ_ERR_ARG, "null info array");
  int d = 0, inter = 0;
  wq_status st = check_stack(m, layers, n_layers, flags, &d, &inter);
  if (st != WQ_OK) return st;
  if (m <= 0 || n_layers <= 0) return fail(WQ_ERR_ARG, "m=%d, n_layers=%d: nothing runs", m, n_layers);
  const int sms = num_sms();
  if (sms <= 0) return fail(WQ_ERR_CUDA, "cannot query the current device");
  for (int i = 0; i < 16; ++i) info[i] = -1;
  const StackRoute route = stack_route(m, layers, n_layers, flags);
  info[0] = route;
  if (route == kRouteStack) {
    StackPlan sp;
    if (!stack_kernel_plan(m, layers, n_layers, flags, &sp)) return fail(WQ_ERR_UNSUPPORTED, "no stack plan");
    const int64_t v[7] = {sp.G, sp.NS, sp.SB, sp.h_barrier, sp.WPT, sp.Tmax, (int64_t)sp.smem};
    for (int i = 0; i < 7; ++i) info[1 + i] = v[i];
  }
  if (route == kRouteGemvChain) {
    const wq_mlp_layer &L0 = layers[0];
    const GemvKind kind = gateup_kind(L0.gate.bits);
    const bool next_tp = n_layers > 1 && ((flags & WQ_PRENORM) || layers[1].r > 0);
    const int r_next = next_tp ? layers[1].r : 0;
    GemvPlan pg, pd{};
    if (!plan_gemv(kind, L0.gate.n, L0.gate.k, m, L0.gate.group, L0.r, sms, &pg) ||
        (L0.down.bits == 4 && !plan_gemv(kDownW4, L0.down.n, L0.down.k, m, L0.down.group, r_next, sms, &pd)))
      return fail(WQ_ERR_UNSUPPORTED, "no launch configuration fits");
    if (L0.down.bits == 16) pd.RB = pd.KP = pd.WK = pd.TPW = pd.P = pd.units = -1;  // the bf16 down kernel
    const int64_t v[13] = {pg.RB, pg.KP, pg.WK, pg.TPW, pg.P, pg.units, pd.RB, pd.KP, pd.WK, pd.TPW, pd.P, pd.units,
                           L0.down.bits == 4 && chain_panel_ok(kind, m, L0.gate, L0.r, L0.down, r_next) ? 1 : 0};
    for (int i = 0; i < 13; ++i) info[1 + i] = v[i];
  }
  return ok();
}

size_t wq_attn_workspace_bytes(int batch, int n_heads, int n_kv, int head_dim, int max_len) {
  const int sms = num_sms();
  if (batch <= 0 || n_heads <= 0 || n_kv <= 0 || head_dim <= 0 || max_len <= 0 || sms <= 0) return 0;
  const int S = attn_splits(batch, n_kv, max_len, sms);
  return up256((size_t)batch * n_heads * S * (head_dim + 2) * 4);
}

wq_status wq_attn_decode(const float *qkv, const void *x, const int32_t *lens, int batch, int d, int n_heads, int n_kv,
                         int head_dim, float theta, void *k_cache, void *v_cache, int max_len, void *o, void *ws,
                         size_t ws_bytes, void *stream) {
  if (batch < 0 || d <= 0 || d % 8 != 0) return fail(WQ_ERR_SHAPE, "batch %d, d %d (a positive multiple of 8)", batch, d);
  if (head_dim != 64 && head_dim != 128) return fail(WQ_ERR_UNSUPPORTED, "head_dim %d not 64 or 128", head_dim);
  if (n_kv <= 0 || n_heads <= 0 || n_heads % n_kv != 0 || n_heads / n_kv > 8)
    return fail(WQ_ERR_UNSUPPORTED, "n_heads %d / n_kv %d: a multiple, at most 8 query heads a kv head", n_heads, n_kv);
  if (max_len <= 0) return fail(WQ_ERR_SHAPE, "max_len %d", max_len);
  if (!(theta > 0.f)) return fail(WQ_ERR_ARG, "rope theta must be positive");
  if (batch == 0) return ok();
  if (!qkv || !x || !lens || !k_cache || !v_cache || !o || !ws) return fail(WQ_ERR_ARG, "null pointer");
  if (!aligned16(qkv) || !aligned16(x) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(o) ||
      !aligned16(ws))
    return fail(WQ_ERR_ALIGN, "qkv, x, caches, o or workspace not 16-byte aligned");
  if (ws_bytes < wq_attn_workspace_bytes(batch, n_heads, n_kv, head_dim, max_len))
    return fail(WQ_ERR_WORKSPACE, "attention workspace of %zu bytes, %zu needed", ws_bytes,
                wq_attn_workspace_bytes(batch, n_heads, n_kv, head_dim, max_len));
  const int S = attn_splits(batch, n_kv, max_len, num_sms());
  cudaError_t e = launch_attn_decode(qkv, x, reinterpret_cast<const int *>(lens), batch, d, n_heads, n_kv, head_dim,
                                     (double)theta, k_cache, v_cache, max_len, static_cast<float *>(ws), S, o,
                                     static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "attention launch");
  return ok();
}

}  // extern "C"

namespace {

// Regions of a decoder layer's workspace: the MLP's, the two projections'
// (each with its own arrival counters), the attention partials, then the
// intermediates qkv (fp32), o, x1 and h (bf16).
struct DecoderWs {
  size_t mlp, proj_qkv, proj_o, attn, qkv, o, x1, h, total;
  size_t n_mlp, n_qkv, n_o, n_attn;
};

bool decoder_ws(int batch, const wq_decoder_layer &Ly, int max_len, DecoderWs *W) {
  const int d = Ly.mlp.gate.k, inter = Ly.mlp.gate.n;
  const int H = Ly.n_heads, Hkv = Ly.n_kv, hd = Ly.head_dim;
  const int nqkv = (H + 2 * Hkv) * hd;
  W->n_mlp = wq_workspace_bytes(batch, d, inter, Ly.mlp.r);
  W->n_qkv = wq_workspace_bytes(batch, nqkv, d, 0);
  W->n_o = wq_workspace_bytes(batch, d, H * hd, 0);
  W->n_attn = wq_attn_workspace_bytes(batch, H, Hkv, hd, max_len);
  if (!W->n_mlp || !W->n_qkv || !W->n_o || !W->n_attn) return false;
  size_t off = 0;
  W->mlp = off;      off = up256(off + W->n_mlp);
  W->proj_qkv = off; off = up256(off + W->n_qkv);
  W->proj_o = off;   off = up256(off + W->n_o);
  W->attn = off;     off = up256(off + W->n_attn);
  W->qkv = off;      off = up256(off + (size_t)batch * nqkv * 4);
  W->o = off;        off = up256(off + (size_t)batch * H * hd * 2);
  W->x1 = off;       off = up256(off + (size_t)batch * d * 2);
  W->h = off;        off = up256(off + (size_t)batch * inter * 2);
  W->total = off;
  return true;
}

}  // namespace

extern "C" {

size_t wq_decoder_workspace_bytes(int batch, const wq_decoder_layer *layer, int max_len) {
  if (!layer || batch <= 0 || max_len <= 0) return 0;
  DecoderWs W;
  return decoder_ws(batch, *layer, max_len, &W) ? W.total : 0;
}

wq_status wq_decoder_layer_forward(const void *x, int batch, const int32_t *lens, const wq_decoder_layer *layer,
                                   void *k_cache, void *v_cache, int max_len, unsigned flags, void *y, void *ws,
                                   size_t ws_bytes, void *stream) {
  if (!layer) return fail(WQ_ERR_ARG, "null layer");
  const wq_decoder_layer &Ly = *layer;
  const int d = Ly.mlp.gate.k, inter = Ly.mlp.gate.n;
  const int H = Ly.n_heads, Hkv = Ly.n_kv, hd = Ly.head_dim;
  wq_status st;
  if ((st = check_qweight(&Ly.qkv, 4, "qkv")) != WQ_OK || (st = check_qweight(&Ly.o, 4, "o")) != WQ_OK) return st;
  if (H <= 0 || Hkv <= 0 || hd <= 0 || Ly.qkv.n != (H + 2 * Hkv) * hd || Ly.qkv.k != d || Ly.o.n != d ||
      Ly.o.k != H * hd || Ly.mlp.down.n != d || Ly.mlp.down.k != inter)
    return fail(WQ_ERR_SHAPE, "decoder layer shapes disagree (qkv [%d x %d], o [%d x %d], d %d, heads %d/%d x %d)",
                Ly.qkv.n, Ly.qkv.k, Ly.o.n, Ly.o.k, d, H, Hkv, hd);
  if (flags & ~WQ_PRENORM) return fail(WQ_ERR_ARG, "unknown flags 0x%x", flags);
  if (batch < 0) return fail(WQ_ERR_ARG, "batch %d", batch);
  if (batch == 0) return ok();
  DecoderWs W;
  if (!decoder_ws(batch, Ly, max_len, &W)) return fail(WQ_ERR_SHAPE, "no workspace layout for this layer");
  if (!ws || ws_bytes < W.total)
    return fail(WQ_ERR_WORKSPACE, "decoder workspace of %zu bytes, %zu needed", ws_bytes, W.total);
  uint8_t *w8 = static_cast<uint8_t *>(ws);
  if ((st = wq_down_w4(x, batch, &Ly.qkv, nullptr, w8 + W.qkv, WQ_F32, w8 + W.proj_qkv, W.n_qkv, stream)) != WQ_OK)
    return fail(st, "qkv projection: %s", g_last_error.c_str());
  if ((st = wq_attn_decode(reinterpret_cast<const float *>(w8 + W.qkv), x, lens, batch, d, H, Hkv, hd, Ly.rope_theta,
                           k_cache, v_cache, max_len, w8 + W.o, w8 + W.attn, W.n_attn, stream)) != WQ_OK)
    return fail(st, "attention: %s", g_last_error.c_str());
  const wq_mlp_layer &M = Ly.mlp;
  // Decode sizes: the output projection's epilogue also writes the MLP
  // input's tile partials (RMSNorm sums and LoRA-A products of x1, as the
  // stack's down launches do for the next layer), so the gate/up launch needs
  // no partials kernel, and gate/up hands down the ready binary16 panel of h.
  {
    const int bits = M.gate.bits;
    const bool gu_ok = bits >= 2 && bits <= 4 && check_gateup_pair(&M.gate, &M.up, bits) == WQ_OK &&
                       check_lora(M.lora_a, M.lora_b_gate, M.lora_b_up, M.r) == WQ_OK && !(bits == 4 && M.r != 0) &&
                       M.down.bits == 4 && check_down(&M.down) == WQ_OK;
    const GemvKind kind = gateup_kind(bits);
    const bool need_tp = (flags & WQ_PRENORM) || M.r > 0;
    const int r_o = need_tp ? M.r : 0;
    if (gu_ok && !gateup_uses_gemm(kind, batch, &M.gate, M.r) && !down_uses_gemm(batch, &M.down, 0) &&
        !down_uses_gemm(batch, &Ly.o, r_o) && (r_o == 0 || d % 8 == 0)) {
      if (!y) return fail(WQ_ERR_ARG, "null y");
      if (!aligned16(y)) return fail(WQ_ERR_ALIGN, "y not 16-byte aligned");
      WsLayout Lm, Lo;
      if ((st = check_ws(w8 + W.mlp, W.n_mlp, batch, d, inter, &Lm)) != WQ_OK ||
          (st = check_ws(w8 + W.proj_o, W.n_o, batch, d, H * hd, &Lo)) != WQ_OK)
        return st;
      cudaStream_t s = static_cast<cudaStream_t>(stream);
      float *tp = need_tp ? reinterpret_cast<float *>(w8 + W.mlp + Lm.tp) : nullptr;
      if ((st = run_down(w8 + W.o, batch, &Ly.o, x, w8 + W.x1, 0, need_tp ? M.lora_a : nullptr, r_o, tp, Lo,
                         w8 + W.proj_o, s)) != WQ_OK)
        return fail(st, "output projection: %s", g_last_error.c_str());
      const bool panel = chain_panel_ok(kind, batch, M.gate, M.r, M.down, 0);
      if ((st = run_gateup(kind, w8 + W.x1, batch, &M.gate, &M.up, M.lora_a, M.lora_b_gate, M.lora_b_up, M.r,
                           M.lora_scale, flags, w8 + W.h, tp, Lm, w8 + W.mlp, s, panel)) != WQ_OK)
        return fail(st, "gate/up: %s", g_last_error.c_str());
      if ((st = run_down(w8 + W.h, batch, &M.down, w8 + W.x1, y, 0, nullptr, 0, nullptr, Lm, w8 + W.mlp, s,
                         panel)) != WQ_OK)
        return fail(st, "down: %s", g_last_error.c_str());
      return ok();
    }
  }
  if ((st = wq_down_w4(w8 + W.o, batch, &Ly.o, x, w8 + W.x1, WQ_BF16, w8 + W.proj_o, W.n_o, stream)) != WQ_OK)
    return fail(st, "output projection: %s", g_last_error.c_str());
  if (M.gate.bits == 3)
    st = wq_gateup_w3_lora(w8 + W.x1, batch, &M.gate, &M.up, M.lora_a, M.lora_b_gate, M.lora_b_up, M.r, M.lora_scale,
                           flags, w8 + W.h, w8 + W.mlp, W.n_mlp, stream);
  else if (M.gate.bits == 2)
    st = wq_gateup_w2_lora(w8 + W.x1, batch, &M.gate, &M.up, M.lora_a, M.lora_b_gate, M.lora_b_up, M.r, M.lora_scale,
                           flags, w8 + W.h, w8 + W.mlp, W.n_mlp, stream);
  else
    st = wq_gateup_w4(w8 + W.x1, batch, &M.gate, &M.up, flags, w8 + W.h, w8 + W.mlp, W.n_mlp, stream);
  if (st != WQ_OK) return fail(st, "gate/up: %s", g_last_error.c_str());
  if ((st = wq_down_w4(w8 + W.h, batch, &M.down, w8 + W.x1, y, WQ_BF16, w8 + W.mlp, W.n_mlp, stream)) != WQ_OK)
    return fail(st, "down: %s", g_last_error.c_str());
  return ok();
}

}  // extern "C"

namespace {

// Plans and workspace regions of a mixture-of-experts block for m tokens:
// the slots' arrival counters first (zero between calls), then the routing
// outputs, tile partials, h and the experts' fp32 outputs of every slot, then
// the split-K partials.  Each slot's launches are planned as one token on
// its share of the SMs (all slots of a launch run side by side).
struct MoeWs {
  GemvPlan gu, dn;
  size_t cnt_gu, cnt_dn, idx, w, tp, h, ys, part_gu, part_dn, total;
};

bool moe_plan(GemvKind kind, int N, int K, int group, int r, int slots, GemvPlan *p) {
  const int sms = num_sms();
  if (sms <= 0) return false;
  for (int share = std::max(1, sms / slots);; share = std::min(sms, share * 2)) {
    if (plan_gemv(kind, N, K, 1, group, r, share, p)) return true;
    if (share == sms) return false;
  }
}

wq_status moe_check(int m, const wq_moe_layer *layer) {
  if (!layer) return fail(WQ_ERR_ARG, "null MoE layer");
  const wq_mlp_layer &X = layer->experts;
  const int E = layer->n_experts, k = layer->top_k;
  if (E < 1 || E > moe_max_experts()) return fail(WQ_ERR_SHAPE, "n_experts %d not in [1, %d]", E, moe_max_experts());
  if (k < 1 || k > std::min(E, moe_max_top_k()))
    return fail(WQ_ERR_SHAPE, "top_k %d not in [1, min(n_experts, %d)]", k, moe_max_top_k());
  const int bits = X.gate.bits == 4 ? 4 : 2;
  wq_status st;
  if ((st = check_qweight(&X.gate, bits, "gate")) != WQ_OK || (st = check_qweight(&X.up, bits, "up")) != WQ_OK ||
      (st = check_qweight(&X.down, 4, "down")) != WQ_OK)
    return st;
  const int d = X.gate.k;
  if (X.gate.n % E != 0) return fail(WQ_ERR_SHAPE, "gate rows %d not a multiple of n_experts %d", X.gate.n, E);
  const int inter = X.gate.n / E;
  if (X.up.n != X.gate.n || X.up.k != d || X.up.group != X.gate.group || X.down.n != E * d || X.down.k != inter)
    return fail(WQ_ERR_SHAPE, "expert shapes disagree (gate [%d x %d], up [%d x %d], down [%d x %d], %d experts)",
                X.gate.n, X.gate.k, X.up.n, X.up.k, X.down.n, X.down.k, E);
  if (d % 16 != 0 || inter % 16 != 0)
    return fail(WQ_ERR_SHAPE, "d %d and the expert width %d must be multiples of 16", d, inter);
  if (X.r < 0 || X.r > kMaxRank || X.r % 8 != 0) return fail(WQ_ERR_SHAPE, "LoRA rank %d", X.r);
  if (X.r > 0) {
    if (bits != 2) return fail(WQ_ERR_UNSUPPORTED, "adapters on 4-bit experts");
    if (!X.lora_a || !X.lora_b_gate || !X.lora_b_up) return fail(WQ_ERR_ARG, "null LoRA factor");
    if (!aligned16(X.lora_a) || !aligned16(X.lora_b_gate) || !aligned16(X.lora_b_up))
      return fail(WQ_ERR_ALIGN, "LoRA factors not 16-byte aligned");
  }
  if (m < 0 || m > kMaxTokens) return fail(WQ_ERR_SHAPE, "m = %d tokens not in [0, %d]", m, kMaxTokens);
  return WQ_OK;
}

bool moe_ws(int m, const wq_moe_layer &L, unsigned flags, MoeWs *W) {
  const wq_mlp_layer &X = L.experts;
  const int E = L.n_experts, S = m * L.top_k, d = X.gate.k, inter = X.gate.n / E, r = X.r;
  const GemvKind kgu = X.gate.bits == 4 ? kGateUpW4 : kGateUpW2;
  if (!moe_plan(kgu, inter, d, X.gate.group, r, S, &W->gu) || !moe_plan(kDownW4, d, inter, X.down.group, 0, S, &W->dn))
    return false;
  const bool need_tp = (flags & WQ_PRENORM) || r > 0;
  size_t off = 0;
  W->cnt_gu = off;  off = up256(off + (size_t)S * W->gu.RT * 4);
  W->cnt_dn = off;  off = up256(off + (size_t)S * W->dn.RT * 4);
  W->idx = off;     off = up256(off + (size_t)S * 4);
  W->w = off;       off = up256(off + (size_t)S * 4);
  W->tp = off;      off = up256(off + (need_tp ? (size_t)S * (d / 16) * WQ_TP_STRIDE(r) * 4 : 0));
  W->h = off;       off = up256(off + (size_t)S * inter * 2);
  W->ys = off;      off = up256(off + (size_t)S * d * 4);
  W->part_gu = off; off = up256(off + (size_t)S * partial_bytes(W->gu, 2));
  W->part_dn = off; off = up256(off + (size_t)S * partial_bytes(W->dn, 1));
  W->total = off;
  return true;
}

}  // namespace

extern "C" {

size_t wq_moe_workspace_bytes(int m, const wq_moe_layer *layer, unsigned flags) {
  if (m <= 0 || moe_check(m, layer) != WQ_OK) return 0;
  MoeWs W;
  return moe_ws(m, *layer, flags, &W) ? W.total : 0;
}

wq_status wq_moe_forward(const void *x, int m, const float *logits, const wq_moe_layer *layer, unsigned flags,
                         void *y, int32_t *expert_idx, float *expert_w, void *h_slots, float *y_slots, void *ws,
                         size_t ws_bytes, void *stream) {
  wq_status st = moe_check(m, layer);
  if (st != WQ_OK) return st;
  if (flags & ~WQ_PRENORM) return fail(WQ_ERR_ARG, "unknown flags 0x%x", flags);
  if (m == 0) return ok();
  if (!x || !logits || !y) return fail(WQ_ERR_ARG, "null x, logits or y");
  if (!aligned16(x) || !aligned16(logits) || !aligned16(y) || !aligned16(expert_idx) || !aligned16(expert_w) ||
      !aligned16(h_slots) || !aligned16(y_slots))
    return fail(WQ_ERR_ALIGN, "a device pointer is not 16-byte aligned");
  const wq_moe_layer &L = *layer;
  const wq_mlp_layer &X = L.experts;
  MoeWs W;
  if (!moe_ws(m, L, flags, &W)) return fail(WQ_ERR_UNSUPPORTED, "no launch configuration fits the experts");
  if (!ws || ws_bytes < W.total) return fail(WQ_ERR_WORKSPACE, "MoE workspace of %zu bytes, %zu needed", ws_bytes, W.total);
  uint8_t *w8 = static_cast<uint8_t *>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int E = L.n_experts, k = L.top_k, S = m * k, d = X.gate.k, inter = X.gate.n / E, r = X.r;
  const bool need_tp = (flags & WQ_PRENORM) || r > 0;
  int *idx = expert_idx ? expert_idx : reinterpret_cast<int *>(w8 + W.idx);
  float *wt = expert_w ? expert_w : reinterpret_cast<float *>(w8 + W.w);
  void *h = h_slots ? h_slots : static_cast<void *>(w8 + W.h);
  float *ys = y_slots ? y_slots : reinterpret_cast<float *>(w8 + W.ys);
  float *tp = need_tp ? reinterpret_cast<float *>(w8 + W.tp) : nullptr;

  cudaError_t e = launch_moe_prep(x, m, d, logits, E, k, r > 0 ? X.lora_a : nullptr, 2 * r, tp, idx, wt, s);
  if (e != cudaSuccess) return cuda_fail(e, "MoE routing launch");

  GemvArgs a = {};
  a.act = x;
  a.M = 1;
  a.K = d;
  a.N = inter;
  a.group = X.gate.group;
  a.codes[0] = X.gate.codes;
  a.codes[1] = X.up.codes;
  a.meta[0] = X.gate.meta;
  a.meta[1] = X.up.meta;
  a.tp = tp;
  a.ntp = d / 16;
  a.prenorm = (flags & WQ_PRENORM) ? 1 : 0;
  a.lora_b[0] = r > 0 ? X.lora_b_gate : nullptr;
  a.lora_b[1] = r > 0 ? X.lora_b_up : nullptr;
  a.r = r;
  a.lora_scale = X.lora_scale;
  a.out = h;
  a.partials = reinterpret_cast<float *>(w8 + W.part_gu);
  a.counters = reinterpret_cast<unsigned *>(w8 + W.cnt_gu);
  a.slot_expert = idx;
  a.n_experts = E;
  a.slot_div = k;
  e = launch_gemv_slots(X.gate.bits == 4 ? kGateUpW4 : kGateUpW2, W.gu, a, S, s, true);
  if (e != cudaSuccess) return cuda_fail(e, "MoE gate/up launch");

  GemvArgs b = {};
  b.act = h;
  b.M = 1;
  b.K = inter;
  b.N = d;
  b.group = X.down.group;
  b.codes[0] = X.down.codes;
  b.meta[0] = X.down.meta;
  b.out = ys;
  b.out_f32 = 1;
  b.partials = reinterpret_cast<float *>(w8 + W.part_dn);
  b.counters = reinterpret_cast<unsigned *>(w8 + W.cnt_dn);
  b.slot_expert = idx;
  b.n_experts = E;
  b.slot_div = 1;
  b.slot_expert_ready = 1;  // the routing launch is two launches back: the down weights stream before the wait
  e = launch_gemv_slots(kDownW4, W.dn, b, S, s, true);
  if (e != cudaSuccess) return cuda_fail(e, "MoE down launch");

  e = launch_moe_combine(x, m, d, k, wt, ys, y, s);
  if (e != cudaSuccess) return cuda_fail(e, "MoE combine launch");
  return ok();
}

wq_status wq_plan_info(int kind, int n, int k, int m, int group, int r, int64_t info[10]) {
  if (!info) return fail(WQ_ERR_ARG, "null info array");
  if (kind < 0 || kind > 3) return fail(WQ_ERR_ARG, "kind %d not in {0, 1, 2, 3}", kind);
  if (!group_ok(group) || k % group != 0) return fail(WQ_ERR_SHAPE, "group %d / k %d unsupported", group, k);
  const int sms = num_sms();
  if (sms <= 0) return fail(WQ_ERR_CUDA, "cannot query the current device");
  GemvPlan p;
  if (!plan_gemv(static_cast<GemvKind>(kind), n, k, m, group, r, sms, &p))
    return fail(WQ_ERR_UNSUPPORTED, "no launch configuration fits");
  const int64_t v[10] = {p.RT, p.KB, p.RB, p.KP, p.WK, p.P, p.units, p.threads, p.smem, 8 * p.NT};
  for (int i = 0; i < 10; ++i) info[i] = v[i];
  return ok();
}

wq_status wq_wait_check(void *stream) {
  cudaError_t e = launch_wait_check(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "wait self-check launch");
  return ok();
}

const char *wq_last_error(void) { return g_last_error.c_str(); }

// Debug builds: first failed in-kernel bounds / alignment check.
wq_status wq_debug_record(long long rec[4]) {
  if (!rec) return fail(WQ_ERR_ARG, "null record");
  cudaError_t e = read_debug_record(rec);
  if (e != cudaSuccess) return cuda_fail(e, "debug record read");
  return ok();
}

wq_status wq_device_status(int *status) {
  if (!status) return fail(WQ_ERR_ARG, "null status pointer");
  cudaError_t e = read_device_status(status);
  if (e != cudaSuccess) return cuda_fail(e, "device status read");
  int g = 0;
  e = read_gemm_status(&g);
  if (e != cudaSuccess) return cuda_fail(e, "device status read");
  if (*status == 0) *status = g;
  e = read_stack_status(&g);
  if (e != cudaSuccess) return cuda_fail(e, "device status read");
  if (*status == 0) *status = g;
  e = read_attn_status(&g);
  if (e != cudaSuccess) return cuda_fail(e, "device status read");
  if (*status == 0) *status = g;
  return ok();
}

const char *wq_version(void) { return "wq 0.1 (sm_103a)"; }

}  // extern "C"
