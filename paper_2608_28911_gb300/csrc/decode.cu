// decode.cu — single-query decode attention over the packed mixed-precision cache
// ("use Ĉ_KV for decoding", Algorithm 1; the fp16 tail of Algorithm 2 takes part).
//
// out[b][qh] = sum_i softmax_i(scale * q . k^_i) v^_i over every token i of the
// high pool, the low pool and the staged fp16 tail of sequence b, KV head
// h = qh / G (G = q_heads / kv_heads <= 8).  Affine rows dequantize as z + s*c.
//
// Work split.  The tokens of each (b, h) are cut into 16-token tiles, per source
// (high pool, low pool, fp16 stage).  A CTA of 8 warps handles a contiguous range of
// tiles of ONE source (so its level count L is uniform), the warps taking tiles
// round-robin; a final kernel merges the per-CTA partials (m, l, o) per (b, qh).
//
// Per warp and tile (affine, level L):
//  - a 4-deep ring of cp.async.bulk copies (one 16-record tile each) completes on
//    per-stage mbarriers; waits are bounded and report a timeout in the error word;
//  - QK^T as S^T = Kc * Q^T on mma.sync m16n8k16 (M = 16 tokens, N = 8 query heads
//    of the group, K = 128 dims): the A fragments are built straight from the packed
//    symbols.  Each lane decodes a quarter row of two tokens; two symbols ride in the
//    16-bit halves of a register and each digit is peeled with one multiply
//    (y = x*L, digit = y >> W), landing as the fp16 value 8 + c.  q is permuted to
//    match the decode order once per CTA;
//  - logits = scale*log2e * (s*(acc - 8*sum q) + z*sum q); online softmax in base 2;
//  - P V as O^T = Vc^T * P'^T (M = 128 dims, N = 8 heads, K = 16 tokens) with
//    P' = p * s_v in fp16; the offset 8 and the zero point are added back per head
//    from the same rounded P' (sum p' * 8) and from sum p * z_v.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace semkv {

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kStages = 4;
constexpr int kTile = 16;
constexpr int kMaxRec = 104;
constexpr int kStageBytes = kTile * kMaxRec + 16;  // +16: window loads may run 12 B past a tile
constexpr int kRingBytes = kWarps * kStages * kStageBytes;
constexpr int kMaxSplits = 64;                     // pool splits per (b, h)
constexpr uint32_t kSpinLimit = 1u << 22;

static_assert(kStageBytes % 16 == 0, "bulk copies need 16-byte aligned stages");
static_assert(kRingBytes >= kWarps * (8 * 128 + 16) * 4, "merge area reuses the ring");

// ------------------------------------------------------------------ PTX -------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait: false after kSpinLimit polls
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  for (uint32_t i = 0; i < kSpinLimit; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

__device__ __forceinline__ void mma16816(float c[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi) {
  return (uint32_t)__half_as_ushort(__float2half_rn(lo)) |
         ((uint32_t)__half_as_ushort(__float2half_rn(hi)) << 16);
}

// ------------------------------------------------------------ decoding --------

// 96 bits starting at bit `pos` of a 4-byte-aligned record (q0 = lowest 32 bits)
struct Window {
  uint32_t q0, q1, q2;
};
__device__ __forceinline__ Window load_window(const uint8_t* rec, int pos) {
  const uint32_t* w = reinterpret_cast<const uint32_t*>(rec) + (pos >> 5);
  const int sh = pos & 31;
  const uint32_t w0 = w[0], w1 = w[1], w2 = w[2], w3 = w[3];
  Window r;
  r.q0 = __funnelshift_r(w0, w1, sh);
  r.q1 = __funnelshift_r(w1, w2, sh);
  r.q2 = __funnelshift_r(w2, w3, sh);
  return r;
}
// bits [p, p+n) of a window, n <= 16 (p, n compile-time after unrolling)
__device__ __forceinline__ uint32_t wbits(const Window& w, int p, int n) {
  const uint32_t mask = (1u << n) - 1u;
  uint32_t v;
  if (p + n <= 32) v = w.q0 >> p;
  else if (p >= 32 && p + n <= 64) v = w.q1 >> (p - 32);
  else if (p >= 64) v = w.q2 >> (p - 64);
  else if (p < 32) v = __funnelshift_r(w.q0, w.q1, p);
  else v = __funnelshift_r(w.q1, w.q2, p - 32);
  return v & mask;
}
// same with a run-time position
__device__ __forceinline__ uint32_t wbits_rt(const Window& w, int p, int n) {
  const uint32_t lo = p < 32 ? w.q0 : (p < 64 ? w.q1 : w.q2);
  const uint32_t hi = p < 32 ? w.q1 : w.q2;
  return __funnelshift_r(lo, hi, p & 31) & ((1u << n) - 1u);
}

// fp16 (8 + digit) in both halves: digit sits at bits [Wd, Wd+3) of each 16-bit lane
template <int Wd>
__device__ __forceinline__ uint32_t digit_half2(uint32_t y) {
  uint32_t t;
  if constexpr (Wd >= 7) t = y >> (Wd - 7);
  else t = y << (7 - Wd);
  return (t & 0x03800380u) | 0x48004800u;
}

// Peel the G digits of two symbols held in the 16-bit halves of x (most
// significant first) into out[0..G).
template <int L, int G, int Wd>
__device__ __forceinline__ void peel(uint32_t x, uint32_t* out) {
  constexpr uint32_t kMask = ((1u << Wd) - 1u) * 0x00010001u;
#pragma unroll
  for (int k = 0; k < G; ++k) {
    const uint32_t y = x * (uint32_t)L;
    out[k] = digit_half2<Wd>(y);
    x = y & kMask;
  }
}

// The 16 half2 of one quarter row of one token (K side: both halves of a register
// are codes of the same token).  Order p: symbol pairs (s, s + NG/2) digit by digit,
// then the tail symbol's two codes.
template <int L>
__device__ __forceinline__ void decode_quarter(const Window& w, uint32_t h[16]) {
  using F = Fmt<L>;
  constexpr int kHalf = F::NG / 2;
#pragma unroll
  for (int s = 0; s < kHalf; ++s) {
    const uint32_t x = wbits(w, s * F::W, F::W) | (wbits(w, (s + kHalf) * F::W, F::W) << 16);
    peel<L, F::G, F::W>(x, h + s * F::G);
  }
  if constexpr (F::R > 0) {
    static_assert(F::R == 2 && kHalf * F::G == 15, "tail layout");
    // the two tail digits: peel the tail symbol twice in one lane
    const uint32_t t = wbits(w, F::NG * F::W, F::WT);
    const uint32_t y0 = t * (uint32_t)L;
    const uint32_t d0 = y0 >> F::WT;
    const uint32_t y1 = (y0 & ((1u << F::WT) - 1u)) * (uint32_t)L;
    const uint32_t d1 = y1 >> F::WT;
    h[15] = ((d0 << 7) | (d1 << 23)) | 0x48004800u;
  } else {
    static_assert(kHalf * F::G == 16, "layout");
  }
}

// dims (lo half, hi half) of K-side half2 p of quarter t
template <int L>
__device__ __forceinline__ void k_dims(int t, int p, int& dlo, int& dhi) {
  using F = Fmt<L>;
  constexpr int kHalf = F::NG / 2;
  if (F::R > 0 && p == 15) {
    dlo = 32 * t + 30;
    dhi = 32 * t + 31;
  } else {
    const int s = p / F::G, k = p % F::G;
    dlo = 32 * t + s * F::G + k;
    dhi = 32 * t + (s + kHalf) * F::G + k;
  }
}

// V side: lane group g decodes half `hh` of quarter qv for two tokens at once (the
// halves of each register are the two tokens).  Output u = 0..15: symbol s' digit k
// at u = s'*G + k, then (when present) tail digit hh at u = 15.
template <int L>
__device__ __forceinline__ void decode_half_quarter_pair(const Window& wa, const Window& wb,
                                                         const Window& ta, const Window& tb,
                                                         int hh, uint32_t h[16]) {
  using F = Fmt<L>;
  constexpr int kHalf = F::NG / 2;
#pragma unroll
  for (int s = 0; s < kHalf; ++s) {
    const uint32_t x = wbits(wa, s * F::W, F::W) | (wbits(wb, s * F::W, F::W) << 16);
    peel<L, F::G, F::W>(x, h + s * F::G);
  }
  if constexpr (F::R > 0) {
    const uint32_t x = wbits(ta, F::NG * F::W, F::WT) | (wbits(tb, F::NG * F::W, F::WT) << 16);
    const uint32_t y0 = x * (uint32_t)L;
    const uint32_t y1 = (y0 & (((1u << F::WT) - 1u) * 0x00010001u)) * (uint32_t)L;
    h[15] = digit_half2<F::WT>(hh ? y1 : y0);
  }
}

template <int L>
__device__ __forceinline__ int v_dim(int g, int u) {
  using F = Fmt<L>;
  constexpr int kHalf = F::NG / 2;
  const int qv = g >> 1, hh = g & 1;
  if (F::R > 0 && u == 15) return 32 * qv + 30 + hh;
  const int s = u / F::G, k = u % F::G;
  return 32 * qv + (hh * kHalf + s) * F::G + k;
}

// ------------------------------------------------------- per-warp state -------

struct WarpState {
  float O[8][4];     // O^T accumulators: rows (dims) x columns (heads 2t, 2t+1)
  float m[2];        // running max (base-2 logits) of heads 2t, 2t+1
  float l[2];        // partial sum of p over this lane's tokens
  float poff[2];     // partial sum of the rounded p*s_v (offset correction)
  float zs[2];       // partial sum of p*z_v
};

__device__ __forceinline__ void state_init(WarpState& st) {
#pragma unroll
  for (int m = 0; m < 8; ++m)
#pragma unroll
    for (int e = 0; e < 4; ++e) st.O[m][e] = 0.0f;
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    st.m[e] = -INFINITY;
    st.l[e] = 0.0f;
    st.poff[e] = 0.0f;
    st.zs[e] = 0.0f;
  }
}

struct Shared {
  uint16_t q[8][128];       // the group's query heads (rows >= G are zero)
  uint64_t bar[kWarps][kStages];
};

// ------------------------------------------------------------ pool tiles ------

template <int L>
__device__ void run_pool(const DecodeArgs& a, const Shared& sh, uint8_t* ring,
                         uint64_t* bars, const uint8_t* pool_bh, int64_t count, int t_begin,
                         int t_end, int G, WarpState& st) {
  using F = Fmt<L>;
  constexpr int kRec = 2 * F::RB + 8;
  constexpr uint32_t kTileBytes = kTile * kRec;
  static_assert(kTileBytes % 16 == 0, "tile size must be a multiple of 16 bytes");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  uint8_t* my_ring = ring + warp * kStages * kStageBytes;
  uint64_t* my_bar = bars + warp * kStages;

  // q fragments (B of S^T = Kc Q^T): column n = g, rows = this quarter's decode order
  uint32_t bq[16];
#pragma unroll
  for (int p = 0; p < 16; ++p) {
    int dlo, dhi;
    k_dims<L>(t, p, dlo, dhi);
    bq[p] = (uint32_t)sh.q[g][dlo] | ((uint32_t)sh.q[g][dhi] << 16);
  }
  float sumq[2];
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    float s = 0.0f;
    for (int d = 0; d < 128; ++d) s += f16_to_f32(sh.q[2 * t + e][d]);
    sumq[e] = s;
  }
  const int qv = g >> 1, hh = g & 1;
  const int vpos = 8 * F::RB + qv * F::QB + hh * (F::NG / 2) * F::W;  // V half-quarter
  const int vtail = 8 * F::RB + qv * F::QB;                           // V quarter (tail)

  const int nmine = t_end - t_begin <= warp ? 0 : (t_end - t_begin - warp + kWarps - 1) / kWarps;
  // prologue: fill the ring
  if (lane == 0) {
    for (int i = 0; i < kStages && i < nmine; ++i) {
      const int tile = t_begin + warp + i * kWarps;
      mbar_expect_tx(&my_bar[i], kTileBytes);
      bulk_g2s(my_ring + i * kStageBytes, pool_bh + (int64_t)tile * kTileBytes, kTileBytes,
               &my_bar[i]);
    }
  }
  __syncwarp();
  bool ok = true;
  int it = 0;
  for (; it < nmine; ++it) {
    const int stage = it % kStages;
    if (!mbar_wait(&my_bar[stage], (uint32_t)((it / kStages) & 1))) {
      ok = false;
      break;
    }
    const int tile = t_begin + warp + it * kWarps;
    const uint8_t* tb = my_ring + stage * kStageBytes;
    const int nvalid = (int)min((int64_t)kTile, count - (int64_t)tile * kTile);

    // ---- S^T = Kc Q^T
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    {
      uint32_t h0[16], h1[16];
      decode_quarter<L>(load_window(tb + g * kRec, t * F::QB), h0);
      decode_quarter<L>(load_window(tb + (g + 8) * kRec, t * F::QB), h1);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        mma16816(acc, h0[2 * j], h1[2 * j], h0[2 * j + 1], h1[2 * j + 1], bq[2 * j], bq[2 * j + 1]);
    }
    // ---- logits and online softmax (base 2)
    float p[2][2], ph_sum[2] = {0.f, 0.f}, zadd[2] = {0.f, 0.f};
    uint32_t X[2];
    {
      float lg[2][2];
      float sv[2], zv[2];
      bool valid[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int tok = g + 8 * e;
        const uint32_t* prm = reinterpret_cast<const uint32_t*>(tb + tok * kRec + 2 * F::RB);
        const uint32_t kp = prm[0], vp = prm[1];
        const float sk = f16_to_f32((uint16_t)(kp & 0xFFFF)), zk = f16_to_f32((uint16_t)(kp >> 16));
        sv[e] = f16_to_f32((uint16_t)(vp & 0xFFFF));
        zv[e] = f16_to_f32((uint16_t)(vp >> 16));
        valid[e] = tok < nvalid;
        const float A = a.scale_log2 * sk;
        const float Bz = a.scale_log2 * (zk - 8.0f * sk);
#pragma unroll
        for (int c = 0; c < 2; ++c)
          lg[e][c] = valid[e] ? fmaf(A, acc[2 * e + c], Bz * sumq[c]) : -INFINITY;
      }
      float mnew[2];
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        float mx = fmaxf(lg[0][c], lg[1][c]);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        mnew[c] = fmaxf(st.m[c], mx);
      }
      const bool grow = (mnew[0] > st.m[0]) || (mnew[1] > st.m[1]);
      if (__any_sync(0xffffffffu, grow)) {
        float al[2];
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          al[c] = (st.m[c] == -INFINITY) ? 0.0f : exp2f(st.m[c] - mnew[c]);
          st.m[c] = mnew[c];
          st.l[c] *= al[c];
          st.poff[c] *= al[c];
          st.zs[c] *= al[c];
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
          st.O[m][0] *= al[0];
          st.O[m][1] *= al[1];
          st.O[m][2] *= al[0];
          st.O[m][3] *= al[1];
        }
      }
#pragma unroll
      for (int c = 0; c < 2; ++c) {
#pragma unroll
        for (int e = 0; e < 2; ++e) p[e][c] = valid[e] ? exp2f(lg[e][c] - st.m[c]) : 0.0f;
      }
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const __half a0 = __float2half_rn(p[0][c] * sv[0]);
        const __half a1 = __float2half_rn(p[1][c] * sv[1]);
        X[c] = (uint32_t)__half_as_ushort(a0) | ((uint32_t)__half_as_ushort(a1) << 16);
        ph_sum[c] = __half2float(a0) + __half2float(a1);
        zadd[c] = p[0][c] * zv[0] + p[1][c] * zv[1];
        st.l[c] += p[0][c] + p[1][c];
        st.poff[c] += ph_sum[c];
        st.zs[c] += zadd[c];
      }
    }
    // ---- P'^T into the B fragment: column g (head g), rows = tokens 2t, 2t+1, 2t+8, 2t+9
    uint32_t b0, b1;
    {
      const int src0 = (2 * t) * 4 + (g >> 1), src1 = (2 * t + 1) * 4 + (g >> 1);
      const uint32_t v0 = __shfl_sync(0xffffffffu, X[0], src0);
      const uint32_t v1 = __shfl_sync(0xffffffffu, X[1], src0);
      const uint32_t w0 = __shfl_sync(0xffffffffu, X[0], src1);
      const uint32_t w1 = __shfl_sync(0xffffffffu, X[1], src1);
      const uint32_t A = (g & 1) ? v1 : v0;  // tokens 2t (lo), 2t+8 (hi)
      const uint32_t B = (g & 1) ? w1 : w0;  // tokens 2t+1 (lo), 2t+9 (hi)
      b0 = g < G ? __byte_perm(A, B, 0x5410) : 0u;
      b1 = g < G ? __byte_perm(A, B, 0x7632) : 0u;
    }
    // ---- O^T += Vc^T P'^T
    {
      uint32_t ha[16], hb[16];
      const Window wa0 = load_window(tb + (2 * t) * kRec, vpos);
      const Window wa1 = load_window(tb + (2 * t + 1) * kRec, vpos);
      const Window ta0 = load_window(tb + (2 * t) * kRec, vtail);
      const Window ta1 = load_window(tb + (2 * t + 1) * kRec, vtail);
      decode_half_quarter_pair<L>(wa0, wa1, ta0, ta1, hh, ha);
      const Window wb0 = load_window(tb + (2 * t + 8) * kRec, vpos);
      const Window wb1 = load_window(tb + (2 * t + 9) * kRec, vpos);
      const Window tb0 = load_window(tb + (2 * t + 8) * kRec, vtail);
      const Window tb1 = load_window(tb + (2 * t + 9) * kRec, vtail);
      decode_half_quarter_pair<L>(wb0, wb1, tb0, tb1, hh, hb);
#pragma unroll
      for (int m = 0; m < 8; ++m)
        mma16816(st.O[m], ha[2 * m], ha[2 * m + 1], hb[2 * m], hb[2 * m + 1], b0, b1);
    }
    __syncwarp();
    // refill this stage with the tile kStages ahead
    if (lane == 0 && it + kStages < nmine) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      const int nt = t_begin + warp + (it + kStages) * kWarps;
      mbar_expect_tx(&my_bar[stage], kTileBytes);
      bulk_g2s(my_ring + stage * kStageBytes, pool_bh + (int64_t)nt * kTileBytes, kTileBytes,
               &my_bar[stage]);
    }
  }
  if (!ok) {
    // a copy never completed: record it, give the copies still in flight a bounded
    // chance to land, and drop this warp's contribution
    if (lane == 0) raise_error(a.err, kDevWaitTimeout);
    for (int j = it; j < nmine && j < it + kStages; ++j)
      mbar_wait(&my_bar[j % kStages], (uint32_t)((j / kStages) & 1));
    state_init(st);
  }
}

// ------------------------------------------------------- fp16 stage tokens ----

// Staged tokens are few (< block): one warp per token, lane = 4 dims, CUDA cores.
__device__ void run_stage(const DecodeArgs& a, const Shared& sh, int b, int h, int G,
                          float* m_out, float* l_out, float* o_out /* [8][128] */) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float qf[8][4];
#pragma unroll
  for (int c = 0; c < 8; ++c)
#pragma unroll
    for (int j = 0; j < 4; ++j) qf[c][j] = c < G ? f16_to_f32(sh.q[c][4 * lane + j]) : 0.0f;
  float m[8], l[8], o[8][4];
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    m[c] = -INFINITY;
    l[c] = 0.0f;
#pragma unroll
    for (int j = 0; j < 4; ++j) o[c][j] = 0.0f;
  }
  const int64_t base = (((int64_t)b * a.NL + a.layer) * a.H + h) * a.block;
  for (int i = warp; i < a.stage_n; i += kWarps) {
    const uint2 ku = *reinterpret_cast<const uint2*>(a.stage_k + (base + i) * 128 + 4 * lane);
    const uint2 vu = *reinterpret_cast<const uint2*>(a.stage_v + (base + i) * 128 + 4 * lane);
    const float kx[4] = {f16_to_f32(ku.x & 0xFFFF), f16_to_f32(ku.x >> 16),
                         f16_to_f32(ku.y & 0xFFFF), f16_to_f32(ku.y >> 16)};
    const float vx[4] = {f16_to_f32(vu.x & 0xFFFF), f16_to_f32(vu.x >> 16),
                         f16_to_f32(vu.y & 0xFFFF), f16_to_f32(vu.y >> 16)};
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      if (c >= G) break;
      float d = qf[c][0] * kx[0] + qf[c][1] * kx[1] + qf[c][2] * kx[2] + qf[c][3] * kx[3];
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off);
      const float lg = d * a.scale_log2;
      const float mn = fmaxf(m[c], lg);
      const float al = m[c] == -INFINITY ? 0.0f : exp2f(m[c] - mn);
      const float pp = exp2f(lg - mn);
      m[c] = mn;
      l[c] = l[c] * al + pp;
#pragma unroll
      for (int j = 0; j < 4; ++j) o[c][j] = o[c][j] * al + pp * vx[j];
    }
  }
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    if (c >= G) break;
    if (lane == 0) {
      m_out[warp * 8 + c] = m[c];
      l_out[warp * 8 + c] = l[c];
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) o_out[(warp * 8 + c) * 128 + 4 * lane + j] = o[c][j];
  }
}

// -------------------------------------------------------------- kernel --------

__global__ void __launch_bounds__(kThreads, 2) decode_kernel(DecodeArgs a) {
  extern __shared__ __align__(128) uint8_t dyn[];
  __shared__ Shared sh;
  __shared__ float merge_m[kWarps * 8], merge_l[kWarps * 8];
  uint8_t* ring = dyn;
  float* merge_o = reinterpret_cast<float*>(dyn);  // [kWarps][8][128], after the loop

  const int b = blockIdx.z, h = blockIdx.y, split = blockIdx.x;
  const int G = a.Hq / a.H;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const DecodePlan& P = a.plan;

  for (int i = threadIdx.x; i < 8 * 128; i += kThreads) {
    const int c = i >> 7, d = i & 127;
    sh.q[c][d] = c < G ? a.q[((int64_t)b * a.Hq + h * G + c) * 128 + d] : (uint16_t)0;
  }
  if (threadIdx.x < kWarps * kStages) {
    mbar_init(&sh.bar[0][0] + threadIdx.x);
  }
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncthreads();

  // which source and which tiles
  int src, s_idx, nsrc, ntiles;
  if (split < P.splits_hi) {
    src = 0; s_idx = split; nsrc = P.splits_hi; ntiles = P.tiles_hi;
  } else if (split < P.splits_hi + P.splits_lo) {
    src = 1; s_idx = split - P.splits_hi; nsrc = P.splits_lo; ntiles = P.tiles_lo;
  } else {
    src = 2; s_idx = 0; nsrc = 1; ntiles = P.tiles_st;
  }
  const int per = (ntiles + nsrc - 1) / nsrc;
  const int t_begin = min(ntiles, s_idx * per), t_end = min(ntiles, t_begin + per);

  if (src == 2) {
    __syncthreads();
    run_stage(a, sh, b, h, G, merge_m, merge_l, merge_o);
  } else {
    WarpState st;
    state_init(st);
    const int L = src == 0 ? a.L_hi : a.L_lo;
    const int64_t cap = src == 0 ? a.hi_cap : a.lo_cap;
    const int64_t count = src == 0 ? a.hi_count : a.lo_count;
    const uint8_t* pool = src == 0 ? a.hi_pool : a.lo_pool;
    const int rec = record_bytes_rt(SEMKV_BASE_AFFINE, L);
    const uint8_t* pool_bh = pool + (((int64_t)b * a.NL + a.layer) * a.H + h) * cap * rec;
    switch (L) {
      case 2: run_pool<2>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      case 3: run_pool<3>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      case 4: run_pool<4>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      case 5: run_pool<5>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      case 6: run_pool<6>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      case 7: run_pool<7>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      case 8: run_pool<8>(a, sh, ring, &sh.bar[0][0], pool_bh, count, t_begin, t_end, G, st); break;
      default: break;
    }
    // reduce the per-lane partial sums over the 8 token rows (lanes with equal t)
#pragma unroll
    for (int c = 0; c < 2; ++c) {
#pragma unroll
      for (int off = 4; off <= 16; off <<= 1) {
        st.l[c] += __shfl_xor_sync(0xffffffffu, st.l[c], off);
        st.poff[c] += __shfl_xor_sync(0xffffffffu, st.poff[c], off);
        st.zs[c] += __shfl_xor_sync(0xffffffffu, st.zs[c], off);
      }
    }
    __syncthreads();  // every warp is done with the ring: reuse it as the merge area
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const int qh = 2 * t + c;
      if (qh < G) {
        const float corr = st.zs[c] - 8.0f * st.poff[c];
        if (g == 0) {
          merge_m[warp * 8 + qh] = st.m[c];
          merge_l[warp * 8 + qh] = st.l[c];
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            int dim;
            switch (L) {
              case 2: dim = v_dim<2>(g, 2 * m + r); break;
              case 3: dim = v_dim<3>(g, 2 * m + r); break;
              case 4: dim = v_dim<4>(g, 2 * m + r); break;
              case 5: dim = v_dim<5>(g, 2 * m + r); break;
              case 6: dim = v_dim<6>(g, 2 * m + r); break;
              case 7: dim = v_dim<7>(g, 2 * m + r); break;
              default: dim = v_dim<8>(g, 2 * m + r); break;
            }
            merge_o[(warp * 8 + qh) * 128 + dim] = st.O[m][2 * r + c] + corr;
          }
        }
      }
    }
  }
  __syncthreads();

  // merge the warps into this CTA's partial (unnormalised o, base-2 max m, sum l)
  float* part = a.partials + (((int64_t)b * a.H + h) * P.splits + split) * kPartialFloats;
  for (int i = threadIdx.x; i < G * 128; i += kThreads) {
    const int qh = i >> 7, d = i & 127;
    float M = -INFINITY;
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, merge_m[w * 8 + qh]);
    float o = 0.0f, lsum = 0.0f;
    if (M != -INFINITY) {
      for (int w = 0; w < kWarps; ++w) {
        const float mw = merge_m[w * 8 + qh];
        if (mw == -INFINITY) continue;
        const float sc = exp2f(mw - M);
        o += sc * merge_o[(w * 8 + qh) * 128 + d];
        lsum += sc * merge_l[w * 8 + qh];
      }
    }
    part[16 + qh * 128 + d] = o;
    if (d == 0) {
      part[qh] = M;
      part[8 + qh] = lsum;
    }
  }
}

// merge the splits of each (b, qh): one warp per head, 4 dims per lane
__global__ void combine_kernel(DecodeArgs a) {
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (gw >= a.B * a.Hq) return;
  const int b = gw / a.Hq, qh = gw % a.Hq;
  const int G = a.Hq / a.H, h = qh / G, c = qh % G;
  const int S = a.plan.splits;
  const float* base = a.partials + ((int64_t)b * a.H + h) * S * kPartialFloats;
  float M = -INFINITY;
  for (int s = 0; s < S; ++s) M = fmaxf(M, base[s * kPartialFloats + c]);
  float o[4] = {0.f, 0.f, 0.f, 0.f}, lsum = 0.0f;
  if (M != -INFINITY) {
    for (int s = 0; s < S; ++s) {
      const float* p = base + s * kPartialFloats;
      const float ms = p[c];
      if (ms == -INFINITY) continue;
      const float sc = exp2f(ms - M);
      lsum += sc * p[8 + c];
      const float4 v = *reinterpret_cast<const float4*>(p + 16 + c * 128 + 4 * lane);
      o[0] += sc * v.x;
      o[1] += sc * v.y;
      o[2] += sc * v.z;
      o[3] += sc * v.w;
    }
  }
  const float inv = 1.0f / lsum;
  float4 r = make_float4(o[0] * inv, o[1] * inv, o[2] * inv, o[3] * inv);
  *reinterpret_cast<float4*>(a.out + ((int64_t)b * a.Hq + qh) * 128 + 4 * lane) = r;
}

}  // namespace

DecodePlan make_decode_plan(int B, int H, int64_t hi_count, int64_t lo_count, int stage_n,
                            int num_sms) {
  DecodePlan p;
  p.tiles_hi = (int)((hi_count + kTile - 1) / kTile);
  p.tiles_lo = (int)((lo_count + kTile - 1) / kTile);
  p.tiles_st = (stage_n + kTile - 1) / kTile;
  const int st = stage_n > 0 ? 1 : 0;
  const int64_t pairs = (int64_t)B * H;
  const int64_t slots = (int64_t)num_sms * 2;  // two 8-warp CTAs per SM
  const int nt = p.tiles_hi + p.tiles_lo;
  int best_s = 1;
  double best_cost = 1e300;
  for (int S = 1; S <= kMaxSplits; ++S) {
    int shi = 0, slo = 0;
    if (p.tiles_hi > 0 && p.tiles_lo > 0) {
      if (S < 2) continue;
      shi = (int)((double)S * p.tiles_hi / nt + 0.5);
      shi = shi < 1 ? 1 : (shi > S - 1 ? S - 1 : shi);
      slo = S - shi;
    } else if (p.tiles_hi > 0) {
      shi = S;
    } else if (p.tiles_lo > 0) {
      slo = S;
    } else {
      break;
    }
    const int per_hi = shi ? (p.tiles_hi + shi - 1) / shi : 0;
    const int per_lo = slo ? (p.tiles_lo + slo - 1) / slo : 0;
    const int per = per_hi > per_lo ? per_hi : per_lo;
    const int64_t ctas = pairs * (S + st);
    const double waves = (double)((ctas + slots - 1) / slots);
    // time ~ waves x per-CTA work (8 warps share a CTA's tiles), plus a small charge
    // for each partial written and merged
    const double cost = waves * (double)((per + kWarps - 1) / kWarps) * (1.0 + 0.002 * S);
    if (cost < best_cost) {
      best_cost = cost;
      best_s = S;
    }
  }
  if (nt == 0) {
    p.splits_hi = p.splits_lo = 0;
  } else if (p.tiles_hi > 0 && p.tiles_lo > 0) {
    int shi = (int)((double)best_s * p.tiles_hi / nt + 0.5);
    shi = shi < 1 ? 1 : (shi > best_s - 1 ? best_s - 1 : shi);
    p.splits_hi = shi;
    p.splits_lo = best_s - shi;
  } else {
    p.splits_hi = p.tiles_hi > 0 ? best_s : 0;
    p.splits_lo = p.tiles_lo > 0 ? best_s : 0;
  }
  p.splits_st = st;
  p.splits = p.splits_hi + p.splits_lo + p.splits_st;
  return p;
}

size_t decode_workspace_floats(int B, int H, int Hq) {
  return (size_t)B * H * (kMaxSplits + 1) * kPartialFloats + (size_t)B * Hq * 128;
}

cudaError_t launch_decode_attention(const DecodeArgs& a, cudaStream_t stream) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kRingBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  if (a.plan.splits == 0) return cudaErrorInvalidValue;
  dim3 grid(a.plan.splits, a.H, a.B);
  decode_kernel<<<grid, kThreads, kRingBytes, stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int heads = a.B * a.Hq;
  combine_kernel<<<(heads + 7) / 8, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace semkv
