// decode.cu — single-query decode attention over the packed mixed-precision cache
// ("use Ĉ_KV for decoding", Algorithm 1; the fp16 tail of Algorithm 2 takes part).
//
// out[b][qh] = sum_i softmax_i(scale * q . k^_i) v^_i over every token i of the
// high pool, the low pool and the staged fp16 tail of sequence b, KV head
// h = qh / G (G = q_heads / kv_heads <= 8).  Affine rows dequantize as z + s*c.
//
// Work split.  The tokens of each (b, h) are cut into 16-token tiles, per source
// (high pool, low pool, fp16 stage).  A CTA runs each (b, h, pool) segment of its range
// of tiles in turn (so the level count L is uniform within a segment), its warps taking
// the segment's tiles round-robin (two at a time on the fast path), and writes one
// partial (m, l, o) per segment; a final kernel merges the partials per (b, qh).  The
// affine pools take a balanced plan (equal weighted ranges over all pairs, or ranges
// aligned to the segments when the sequences are few), the TQ pools a split plan.
//
// Decoding on the FMA pipe.  A group symbol is stored as the W-bit integer
// beta = ceil(t 2^W / L^G), so F_k = floor(beta L^(k+1) / 2^W) is the number formed by
// the first k+1 digits and c_k = F_k - L F_{k-1}.  Read as an fp32 bit pattern, beta
// is the denormal beta * 2^-149; one multiply rounded toward zero by the exact
// constant L^(k+1)/2^W yields a float whose bit pattern is F_k; the packed binary32
// forms (mul/fma.rz.f32x2) take two symbols, or two constants, per instruction.  For
// five-level groups two symbols also share one lane of a multiply (beta_a + 65536 beta_b
// is still a denormal) and a mask separates the halves.  Integers (all < 256) become fp16 values with a
// byte placed over them (1024 + v) and one f16x2 subtract.
//  - QK^T as S = Q' F^T on mma.sync m16n8k16 (M = heads, N = 8 tokens, K = 128 F
//    slots): the q coefficient of F_k is q'_k = q_{d_k} - L q_{d_{k+1}} when F_k
//    carries a share of digit k+1, scaled by a power of two and split into fp16 hi
//    and lo rows; logit = scale log2e (s acc + z sum q).  The output fragment is
//    the B operand of the PV product as it stands (at most one exchange of halves).
//  - softmax in base 2 against a per-head reference exponent e that keeps
//    P' = p * s_v below 2^14 (the largest near 2^12) and p below 2^52; e moves, and
//    the running sums are rescaled, only when a tile
//    would exceed that bound.
//  - P V as O^T = C^T P'^T (M = 128 dims, N = 8 columns, K = 16 tokens) on the digits
//    c_k (formed lane-wise as F_k - L F_{k-1} in f16x2), with P' = p * s_v as fp16
//    hi + lo (lo in columns 4..7 when G <= 4, else a second pass), plus sum p * z_v
//    per head.  (Feeding F values to PV and undoing the mixing after accumulation was
//    tried and rejected: the subtraction cancels ~30x and amplified the tensor
//    cores' truncating fp32 accumulation past the attention tolerance.)
// Six-level groups (F_4 up to 7775 would not fit) restart the chain after two
// digits from the remainder x = beta * 36 mod 2^13.
//
// Per warp: a 4-deep ring of cp.async.bulk tile copies completing on per-stage
// mbarriers (bounded waits that report a timeout in the error word).
//
// The description above is that of decode_affine_kernel, which serves every level
// count and GQA group size.  Five- and six-level affine pools with groups of up to
// four heads (the workloads' shape) run decode_affine_fast_kernel instead: the same
// plan, ring and merge, with S^T = F Q'^T (eight MMAs per tile, the coefficients in
// B fragments), five-level digits on the f16x2 FMA pipe, and the softmax in packed
// binary32 (see "affine pools: fast path" below).
#include <float.h>

#include <cstring>

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
constexpr int kAqBytes = 8 * 32 * 16;   // q-coefficient A fragments: 8 k-steps x 32 lanes x uint4
constexpr int kQbBytes = 8 * 32 * 8;    // fast path: coefficient B fragments, 8 steps x 32 lanes x uint2
constexpr int kCtasAffine = 2;          // resident CTAs per SM: affine pools / other sources
constexpr int kCtasOther = 2;
constexpr int kCtasFast = 2;           // resident CTAs per SM: the fast affine path with 8 warps
constexpr int kMaxSplits = 64;                     // pool splits per (b, h)
constexpr float kPMax = 0x1p52f;                   // bound on p = 2^(logit - e)

static_assert(kStageBytes % 16 == 0, "bulk copies need 16-byte aligned stages");
// merge area rows: kMoStride floats per (warp, column) row, dim d at d + d / 32 (each
// quarter one bank further on), so that the lanes writing one dim of each quarter, or
// four consecutive dims each, reach distinct banks
constexpr int kMoStride = 132;
__host__ __device__ constexpr int mo_at(int row, int d) { return row * kMoStride + d + (d >> 5); }
// The fast path copies two tiles (32 consecutive slots) per bulk copy into a ring of
// kFastStages stages per warp: one wait, one refill and one round of ring bookkeeping
// serve 32 tokens.
constexpr int kChunk = 2;                  // tiles per copy on the fast path
constexpr int kFastStages = 3;
constexpr int kFastRec = 92;               // largest fast-path record (six levels)
constexpr int kFastStageBytes = kChunk * kTile * kFastRec + 16;  // +16: window over-read
// The fast path has two CTA shapes.  Over long straddled ranges (many sequences) it runs
// one CTA of 16 warps per SM: the warp schedulers favour the warps of the CTA that
// reached an SM first, so of two 8-warp CTAs with equal ranges one finishes long before
// the other, which then runs alone at half occupancy, while the warps of one CTA advance
// evenly.  With segment-aligned ranges (few sequences), two CTAs of 8 warps per SM, whose
// set-up and merge overlap each other's tiles.
constexpr int kFastWarps = 16;
constexpr int kMaxWarps = 16;                // warps of the largest CTA (barriers, merge area)
template <int NW>
constexpr int fast_ring_bytes() { return NW * kFastStages * kFastStageBytes; }
static_assert(kFastStageBytes % 16 == 0, "bulk copies need 16-byte aligned stages");
static_assert(kFastStages <= kStages, "the fast path uses the first barriers of each warp");
static_assert(fast_ring_bytes<kWarps>() >= (kWarps * 8 * kMoStride + 8 * 128) * 4 &&
                  fast_ring_bytes<kFastWarps>() >= (kFastWarps * 8 * kMoStride + 8 * 128) * 4,
              "merge area reuses the ring");
static_assert(kRingBytes >= (kWarps * 8 * kMoStride + 8 * 128) * 4, "merge area reuses the ring");

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
// expect_tx + bulk copy issued by the lanes where `pred` holds (no branch)
__device__ __forceinline__ void bulk_refill(bool pred, void* dst, const void* src, uint32_t bytes,
                                            uint64_t* bar) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %0, 0;\n"
      " @p mbarrier.arrive.expect_tx.shared::cta.b64 _, [%1], %2;\n"
      " @p cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%3], [%4], %2, [%1];\n}" ::"r"(
          (uint32_t)pred),
      "r"(smem_u32(bar)), "r"(bytes), "r"(smem_u32(dst)), "l"(src)
      : "memory");
}
// bounded wait: false after kWaitPolls polls
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  return mbar_wait_bounded(bar, parity);
}

__device__ __forceinline__ void mma16816(float c[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ---------------------------------------------------------- digit helpers -----

// F = floor(beta * c) for the exact constant c: beta read as a denormal float,
// multiplied with rounding toward zero; the result's bit pattern is the integer F.
__device__ __forceinline__ uint32_t fdig(uint32_t beta, float c) {
  return __float_as_uint(__fmul_rz(__uint_as_float(beta), c));
}
// fdig of two symbols (or one symbol and two constants) in one packed binary32
// instruction, lane 0 taking (a, ca) and lane 1 (b, cb); fdig1024_x2 adds 0x6400 in the
// denormal grid, so the low 16 bits are the fp16 value 1024 + F (F < 1024)
__device__ __forceinline__ unsigned long long u2_pack(uint32_t lo, uint32_t hi) {
  return (unsigned long long)lo | ((unsigned long long)hi << 32);
}
__device__ __forceinline__ void fdig_x2(uint32_t a, uint32_t b, float ca, float cb,
                                        uint32_t& ra, uint32_t& rb) {
  unsigned long long y;
  asm("mul.rz.f32x2 %0, %1, %2;"
      : "=l"(y)
      : "l"(u2_pack(a, b)), "l"(u2_pack(__float_as_uint(ca), __float_as_uint(cb))));
  ra = (uint32_t)y;
  rb = (uint32_t)(y >> 32);
}
__device__ __forceinline__ void fdig1024_x2(uint32_t a, uint32_t b, float ca, float cb,
                                            uint32_t& ra, uint32_t& rb) {
  unsigned long long y;
  asm("fma.rz.f32x2 %0, %1, %2, %3;"
      : "=l"(y)
      : "l"(u2_pack(a, b)), "l"(u2_pack(__float_as_uint(ca), __float_as_uint(cb))),
        "l"(0x0000640000006400ull));
  ra = (uint32_t)y;
  rb = (uint32_t)(y >> 32);
}
// the low halves of a and b side by side
__device__ __forceinline__ uint32_t fpair(uint32_t a, uint32_t b) {
  return __byte_perm(a, b, 0x5410);
}
// subtract 1024 from both fp16 halves: 1024 + v -> v exactly (v < 1024).  Integers
// reach the tensor cores as normal fp16 values: read directly as the subnormals
// v * 2^-24 they multiply exactly in isolation, but a chained accumulation over
// subnormal operands loses about 10 bits (measured: ~1e-3 relative attention error).
__device__ __forceinline__ uint32_t hsub1024(uint32_t x) {
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(x), "r"(0x64006400u));
  return r;
}
// integers in bytes 0 and 2 (< 256; bytes 1 and 3 ignored) -> fp16 values: one byte
// permute lays 0x64 over each (1024 + v) and one f16x2 subtract removes the 1024
__device__ __forceinline__ uint32_t bytes_to_h2(uint32_t P) {
  return hsub1024(__byte_perm(P, 0x64646464u, 0x7250));
}
// fp16 bit pattern of -L
__host__ __device__ constexpr uint32_t neg_half_bits(int L) {
  return L == 2 ? 0xC000u : L == 3 ? 0xC200u : L == 4 ? 0xC400u : L == 5 ? 0xC500u
       : L == 6 ? 0xC600u : L == 7 ? 0xC700u : 0xC800u;
}
// digit pair cur - L prev on fp16 integers (exact: all values are small integers)
template <int L>
__device__ __forceinline__ uint32_t hdigit(uint32_t prev, uint32_t cur) {
  constexpr uint32_t kNegL = neg_half_bits(L) * 0x00010001u;
  uint32_t r;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(prev), "r"(kNegL), "r"(cur));
  return r;
}
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}
// x0, x1 as fp16 hi + lo parts, packed pairwise (exact to ~2^-22 relative)
__device__ __forceinline__ void split_h2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x0, x1);
  const float2 f = __half22float2(h);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = pack_h2(x0 - f.x, x1 - f.y);
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// the largest power of two <= x (x positive and normal)
__device__ __forceinline__ float pow2_floor(float x) {
  return __uint_as_float(__float_as_uint(x) & 0x7F800000u);
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
// bits [p, p+n) of a window (p, n compile-time after unrolling)
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

template <int L>
struct Dec {
  using F = Fmt<L>;
  static constexpr int G = F::G;
  static constexpr int kHalf = F::NG / 2;                     // symbols per half quarter
  static constexpr int kRestart = (L == 6) ? 2 : G;           // F chain restarts here
  // 1024 + F values of two full symbols (fa, fb: the low 16 bits of each word, F < 256),
  // two per packed instruction
  __device__ __forceinline__ static void sym2(uint32_t ba, uint32_t bb, uint32_t* fa,
                                              uint32_t* fb) {
    if constexpr (G == 1) {
      if constexpr (L == 7) {
        fdig1024_x2(ba, bb, 7.0f / 8.0f, 7.0f / 8.0f, fa[0], fb[0]);
      } else {
        fa[0] = ba | 0x6400u;
        fb[0] = bb | 0x6400u;
      }
    } else if constexpr (L == 6) {
      constexpr float c1 = 6.0f / 8192.0f, c2 = 36.0f / 8192.0f, c3 = 216.0f / 8192.0f;
      fdig1024_x2(ba, bb, c1, c1, fa[0], fb[0]);
      fdig1024_x2(ba, bb, c2, c2, fa[1], fb[1]);
      const uint32_t xa = (ba * 36u) & 8191u, xb = (bb * 36u) & 8191u;
      fdig1024_x2(xa, xb, c1, c1, fa[2], fb[2]);
      fdig1024_x2(xa, xb, c2, c2, fa[3], fb[3]);
      fdig1024_x2(xa, xb, c3, c3, fa[4], fb[4]);
    } else {
      float c = (float)L / (float)(1u << F::W);
#pragma unroll
      for (int k = 0; k < G; ++k) {
        fdig1024_x2(ba, bb, c, c, fa[k], fb[k]);
        c *= (float)L;
      }
    }
  }
  // 1024 + F values of the two-code tail symbol
  __device__ __forceinline__ static void tail(uint32_t beta, uint32_t* f) {
    constexpr float c = (float)L / (float)(1u << F::WT);
    fdig1024_x2(beta, beta, c, c * (float)L, f[0], f[1]);
  }
  // the tails of two symbols: fa, fb as in tail
  __device__ __forceinline__ static void tail2(uint32_t ba, uint32_t bb, uint32_t* fa,
                                               uint32_t* fb) {
    constexpr float c = (float)L / (float)(1u << F::WT);
    fdig1024_x2(ba, bb, c, c, fa[0], fb[0]);
    fdig1024_x2(ba, bb, c * (float)L, c * (float)L, fa[1], fb[1]);
  }
  // does F slot k of a group carry a share of digit k+1?
  __host__ __device__ static constexpr bool chained(int k) { return k + 1 < G && k + 1 != kRestart; }
};

// ---- five-level fast path: two 7-bit symbols per register ---------------------
// u = beta_a + 65536 beta_b is still a denormal (beta < 128), and
// floor(u * 5^(k+1)/128) = F_k(a) + 65536 F_k(b) + 512 * (fraction of b's product):
// one multiply gives both halves' F_k (bytes 0 and 2; the fraction lands in byte 1).
constexpr uint32_t kM7 = 0x007F007Fu;
__device__ __forceinline__ void l5_fpairs(uint32_t u, uint32_t* X) {
  uint32_t P0, P1;
  fdig_x2(u, u, 5.0f / 128.0f, 25.0f / 128.0f, P0, P1);
  X[0] = bytes_to_h2(P0);
  X[1] = bytes_to_h2(P1);
  X[2] = bytes_to_h2(fdig(u, 125.0f / 128.0f));
}
// l5_fpairs of two registers at once
__device__ __forceinline__ void l5_fpairs2(uint32_t u, uint32_t v, uint32_t* X, uint32_t* Y) {
  uint32_t P, Q;
  fdig_x2(u, v, 5.0f / 128.0f, 5.0f / 128.0f, P, Q);
  X[0] = bytes_to_h2(P);
  Y[0] = bytes_to_h2(Q);
  fdig_x2(u, v, 25.0f / 128.0f, 25.0f / 128.0f, P, Q);
  X[1] = bytes_to_h2(P);
  Y[1] = bytes_to_h2(Q);
  fdig_x2(u, v, 125.0f / 128.0f, 125.0f / 128.0f, P, Q);
  X[2] = bytes_to_h2(P);
  Y[2] = bytes_to_h2(Q);
}
// symbol pairs from two windows: symbol j of window a in the low half and of window b
// in the high half, j = 0..4 (bits 7j)
__device__ __forceinline__ void l5_pairs(uint32_t a0, uint32_t a1, uint32_t b0, uint32_t b1,
                                         uint32_t u[5]) {
  uint32_t C = fpair(a0, b0);
  u[0] = C & kM7;
  u[1] = (C >> 7) & kM7;
  C = fpair(a0 >> 14, b0 >> 14);
  u[2] = C & kM7;
  u[3] = (C >> 7) & kM7;
  C = fpair(__funnelshift_r(a0, a1, 28), __funnelshift_r(b0, b1, 28));
  u[4] = C & kM7;
}
// the two-code five-level tail of two windows at once (5-bit symbols, u < 2^21):
// F_0 and F_1 pairs (bytes 0 and 2); the fraction of the high symbol lands in bits 11..15
__device__ __forceinline__ void l5_tail_pairs(uint32_t ut, uint32_t& X0, uint32_t& X1) {
  uint32_t P0, P1;
  fdig_x2(ut, ut, 5.0f / 32.0f, 25.0f / 32.0f, P0, P1);
  X0 = bytes_to_h2(P0);
  X1 = bytes_to_h2(P1);
}

// F side of S = Q' F^T: the fp16 F-value pairs of one quarter row of one token (both
// halves are the same token), as the B fragments of the 8 k-steps: slot p = 2j + i
// goes to f[j][i].  Slot p < kHalf*G holds F_k of symbols s and s + kHalf (s = p / G,
// k = p % G); slot 15 holds the tail's F_0 and F_1.
template <int L>
__device__ __forceinline__ void k_quarter(const Window& w, uint32_t (&f)[8][2]) {
  using D = Dec<L>;
  using F = typename D::F;
  uint32_t h[16];
  if constexpr (L == 5) {
    uint32_t u[5];
    // symbol s + 5 sits 35 bits after symbol s
    l5_pairs(w.q0, w.q1, __funnelshift_r(w.q1, w.q2, 3), w.q2 >> 3, u);
    l5_fpairs2(u[0], u[1], h, h + 3);
    l5_fpairs2(u[2], u[3], h + 6, h + 9);
    l5_fpairs(u[4], h + 12);
    uint32_t ft[2];
    D::tail(wbits(w, 70, 5), ft);
    h[15] = hsub1024(fpair(ft[0], ft[1]));
  } else {
#pragma unroll
    for (int s = 0; s < D::kHalf; ++s) {
      uint32_t fa[D::G], fb[D::G];
      D::sym2(wbits(w, s * F::W, F::W), wbits(w, (s + D::kHalf) * F::W, F::W), fa, fb);
#pragma unroll
      for (int k = 0; k < D::G; ++k) h[s * D::G + k] = hsub1024(fpair(fa[k], fb[k]));
    }
    if constexpr (F::R > 0) {
      static_assert(F::R == 2 && D::kHalf * D::G == 15, "tail layout");
      uint32_t ft[2];
      D::tail(wbits(w, F::NG * F::W, F::WT), ft);
      h[15] = hsub1024(fpair(ft[0], ft[1]));
    } else {
      static_assert(D::kHalf * D::G == 16, "layout");
    }
  }
#pragma unroll
  for (int p = 0; p < 16; ++p) f[p >> 1][p & 1] = h[p];
}

// q coefficient of F slot p (lo or hi half) of quarter t for one head: the digit k
// weight minus the share of digit k+1 that F_k carries
__device__ __forceinline__ float qval(const uint16_t* qrow, int d) { return f16_to_f32(qrow[d]); }
__device__ __forceinline__ float qval(const float* qrow, int d) { return qrow[d]; }
template <int L, typename QT>
__device__ __forceinline__ float k_coef(const QT* qrow, int t, int p, int half) {
  using D = Dec<L>;
  using F = typename D::F;
  const int base = 32 * t;
  if (F::R > 0 && p == 15)
    return half == 0 ? qval(qrow, base + 30) - (float)L * qval(qrow, base + 31)
                     : qval(qrow, base + 31);
  const int s = p / D::G + (half ? D::kHalf : 0), k = p % D::G;
  const int d = base + s * D::G + k;
  return D::chained(k) ? qval(qrow, d) - (float)L * qval(qrow, d + 1) : qval(qrow, d);
}
// (2c - 3)^3 of both fp16 halves (c a code of four levels)
__device__ __forceinline__ uint32_t cube_phi(uint32_t c) {
  uint32_t f, f2, f3;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(f) : "r"(c), "r"(0x40004000u), "r"(0xC200C200u));
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(f2) : "r"(f), "r"(f));
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(f3) : "r"(f2), "r"(f));
  return f3;
}

// V side: lane group g holds half hh of quarter qv for two tokens at once (the two
// halves of each register are the two tokens).  Row u = j*G + k is digit k of
// symbol hh*kHalf + j; row 15 is the tail's digit hh.  Digits as fp16 values.
// The 16 rows land in the A fragments of the 8 m-blocks: row u = 2m + i goes to
// A[m][C + i] (C = 0 for tokens 2t, 2t+1 and 2 for tokens 2t+8, 2t+9).
template <int L, int C>
__device__ __forceinline__ void v_half_pair(const Window& wa, const Window& wb, int tpos, int hh,
                                            uint32_t (&A)[8][4]) {
  using D = Dec<L>;
  using F = typename D::F;
  uint32_t h[16];
  if constexpr (L == 5) {
    uint32_t u[5];
    l5_pairs(wa.q0, wa.q1, wb.q0, wb.q1, u);
    uint32_t X[5][3];
    l5_fpairs2(u[0], u[1], X[0], X[1]);
    l5_fpairs2(u[2], u[3], X[2], X[3]);
    l5_fpairs(u[4], X[4]);
#pragma unroll
    for (int j = 0; j < 5; ++j) {
      h[3 * j] = X[j][0];
      h[3 * j + 1] = hdigit<5>(X[j][0], X[j][1]);
      h[3 * j + 2] = hdigit<5>(X[j][1], X[j][2]);
    }
    uint32_t X0, X1;
    l5_tail_pairs(fpair(wbits_rt(wa, tpos, 5), wbits_rt(wb, tpos, 5)), X0, X1);
    h[15] = hh ? hdigit<5>(X0, X1) : X0;
  } else {
#pragma unroll
    for (int j = 0; j < D::kHalf; ++j) {
      uint32_t fa[D::G], fb[D::G], X[D::G];
      D::sym2(wbits(wa, j * F::W, F::W), wbits(wb, j * F::W, F::W), fa, fb);
#pragma unroll
      for (int k = 0; k < D::G; ++k) X[k] = hsub1024(fpair(fa[k], fb[k]));
#pragma unroll
      for (int k = 0; k < D::G; ++k)
        h[j * D::G + k] = (k == 0 || k == D::kRestart) ? X[k] : hdigit<L>(X[k - 1], X[k]);
    }
    if constexpr (F::R > 0) {
      uint32_t fa[2], fb[2];
      D::tail2(wbits_rt(wa, tpos, F::WT), wbits_rt(wb, tpos, F::WT), fa, fb);
      const uint32_t X0 = hsub1024(fpair(fa[0], fb[0]));
      const uint32_t X1 = hsub1024(fpair(fa[1], fb[1]));
      h[15] = hh ? hdigit<L>(X0, X1) : X0;
    }
  }
#pragma unroll
  for (int u = 0; u < 16; ++u) A[u >> 1][C + (u & 1)] = h[u];
}

// output dim of V row u of lane group g
template <int L>
__device__ __forceinline__ int v_dim(int g, int u) {
  using D = Dec<L>;
  using F = typename D::F;
  const int qv = g >> 1, hh = g & 1;
  if (F::R > 0 && u == 15) return 32 * qv + 30 + hh;
  const int s = u / D::G, k = u % D::G;
  return 32 * qv + (hh * D::kHalf + s) * D::G + k;
}

// ------------------------------------------------------- per-warp state -------

struct WarpState {
  float O[8][4];     // O^T accumulators: V rows x columns 2t, 2t+1
  float e;           // reference exponent of head g (base 2)
  float l;           // partial sum of p over this lane's tokens
  float zs;          // partial sum of p*z_v
};

__device__ __forceinline__ void state_init(WarpState& st) {
#pragma unroll
  for (int m = 0; m < 8; ++m)
#pragma unroll
    for (int e = 0; e < 4; ++e) st.O[m][e] = 0.0f;
  st.e = -INFINITY;
  st.l = 0.0f;
  st.zs = 0.0f;
}

struct Shared {
  uint16_t q[8][128];       // the group's query heads (rows >= G are zero)
  float qr[8][128];         // TQ base: rotated queries q' = H S q
  float cb[2][8];           // TQ base: centroids of the high / low level count
  float sumq[8];            // sum over dims of each head's q (q' for TQ records)
  float qmax[8];            // max |q_d| of each head (q' for TQ records)
  float cdec[2][3];         // TQ tensor path, per pool: centroids as cz + cs c (+ c3 phi^3)
  uint64_t bar[kMaxWarps][kStages];
};

// ------------------------------------------------------------ pool tiles ------

// One warp streams its tiles.  Per 16-token tile:
//  S = Q' F^T on m16n8k16 in two 8-token halves (N = tokens g, g+8 of lane group g):
//   A rows g and g+8 are head g's q' coefficients, scaled by a power of two so the
//   largest is near 2^13 and split into fp16 hi (row g) and lo (row g+8) parts.  The
//   output fragment (rows = heads, columns = tokens 2t, 2t+1) is, after adding hi and
//   lo, already laid out as the B fragment the PV product needs: no transposition.
//  p = 2^(logit - e) with a per-head reference e chosen so p*s_v stays <= 2^14 and p <= 2^52:
//   e moves (and the sums are rescaled) only when a tile would exceed that.
//  O^T += C^T P'^T (M = 128 V rows, K = 16 tokens) with P' = p*s_v as fp16 hi + lo
//   (PACKED: columns 0..3 hi and 4..7 lo of heads 0..3; else two passes).
// Codes enter as exact fp16 integers; the partners' power-of-two scales keep every
// operand within the fp16 range.
// CODEC 0: affine records [K][V][Ks Kz Vs Vz], rows z + s c against q.
// CODEC 1: TQ records [K][V][Kn Vn] whose centroids are linear in the code (two or
//   three levels, the codebook symmetric): cb[c] = cz + cs c, so the rows (n/128) cb[c]
//   are affine rows with s = cs n/128, z = cz n/128, taken against q' = H S q.
// CODEC 2: TQ, four levels: cb[c] = alpha phi + beta phi^3 with phi = 2c - 3; the phi
//   part as CODEC 1 (cs = 2 alpha, cz = -3 alpha) plus a second pass on phi^3 (beta).
// ring_it: tiles this warp has already taken through its ring (kept across calls so
// the stage and barrier phase of each tile continue from the previous call)
template <int L, bool PACKED, int CODEC = 0>
__device__ void run_pool(const DecodeArgs& a, const Shared& sh, uint8_t* ring, uint4* aq_all,
                         uint64_t* bars, const uint8_t* pool_bh, int64_t count, int t_begin,
                         int t_end, int G, WarpState& st, int& ring_it, int which = 0,
                         bool prefilled = false) {
  using D = Dec<L>;
  using F = typename D::F;
  static_assert(CODEC != 2 || L == 4, "the cubic decomposition is for four levels");
  constexpr int kRec = 2 * F::RB + (CODEC == 0 ? 8 : 4);
  constexpr uint32_t kTileBytes = kTile * kRec;
  static_assert(kTileBytes % 16 == 0, "tile size must be a multiple of 16 bytes");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  uint8_t* my_ring = ring + warp * kStages * kStageBytes;
  uint64_t* my_bar = bars + warp * kStages;

  // head hd: A rows g (hi) and g + 8 (lo) belong to head g; for G <= 4 lanes g and g + 4
  // share the softmax of head g & 3
  const int hd = PACKED ? (g & 3) : g;
  const bool live = hd < G;
  const bool upper = PACKED && g >= 4;
  const float qmax = sh.qmax[hd];
  const float qscale =
      qmax > 0.0f ? pow2_floor(fminf(8192.0f / ((float)(L + 1) * qmax), 1e30f)) : 1.0f;
  // A fragments of the 8 k-steps, {hi 2j, lo 2j, hi 2j+1, lo 2j+1} per lane, the same
  // for every warp of the CTA: warp 0 stores them in shared memory, every warp loads
  // its lane's fragment (one conflict-free 16-byte load per k-step)
  uint4* aq = aq_all + lane;
  __syncthreads();  // the previous pool's fragments and the merge area are no longer read
#pragma unroll
  for (int j = 0; j < 8 && warp == 0; ++j) {
    uint32_t r[4];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int p = 2 * j + i;
      float c0 = 0.0f, c1 = 0.0f;
      if (live && !upper) {
        if (CODEC == 0 && a.base != SEMKV_BASE_AFFINE_HAD) {
          c0 = k_coef<L>(sh.q[g], t, p, 0) * qscale;
          c1 = k_coef<L>(sh.q[g], t, p, 1) * qscale;
        } else {
          c0 = k_coef<L>(sh.qr[g], t, p, 0) * qscale;
          c1 = k_coef<L>(sh.qr[g], t, p, 1) * qscale;
        }
      }
      split_h2(c0, c1, r[2 * i], r[2 * i + 1]);
    }
    aq[32 * j] = make_uint4(r[0], r[1], r[2], r[3]);
  }
  __syncthreads();  // every warp of the CTA runs this pool with the same level count
  const float cS = a.scale_log2 / qscale;   // logit weight of s_k * S
  const float cZ = a.scale_log2 * sh.sumq[hd];  // logit weight of z_k
  // TQ: row parameters per unit norm (the record holds n as fp16; rows are n/128 cb[c])
  const float tq_s = CODEC ? sh.cdec[which][0] * (1.0f / 128.0f) : 0.0f;
  const float tq_z = CODEC ? sh.cdec[which][1] * (1.0f / 128.0f) : 0.0f;
  const float tq_3 = CODEC == 2 ? sh.cdec[which][2] * (1.0f / 128.0f) : 0.0f;
  // O columns 2t, 2t+1 belong to these heads (their e lives in lane 4*head)
  const int oh0 = PACKED ? ((2 * t) & 3) : 2 * t, oh1 = oh0 + 1;

  const int qv = g >> 1, hh = g & 1;
  const int vpos = 8 * F::RB + qv * F::QB + hh * D::kHalf * F::W;  // V half quarter
  const int tpos = F::NG * F::W - hh * D::kHalf * F::W;           // tail, relative

  const int nmine = t_end - t_begin <= warp ? 0 : (t_end - t_begin - warp + kWarps - 1) / kWarps;
  const int count32 = (int)count;  // a pool holds fewer than 2^31 slots
  if (lane == 0 && !prefilled) {
    // the ring may have been the merge area: order those writes before the copies
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    for (int i = 0; i < kStages && i < nmine; ++i) {
      const int tile = t_begin + warp + i * kWarps;
      const int sl = (ring_it + i) % kStages;
      mbar_expect_tx(&my_bar[sl], kTileBytes);
      bulk_g2s(my_ring + sl * kStageBytes, pool_bh + (int64_t)tile * kTileBytes, kTileBytes,
               &my_bar[sl]);
    }
  }
  __syncwarp();
  bool ok = true;
  int it = 0;
  for (; it < nmine; ++it) {
    const int gi = ring_it + it;
    const int stage = gi % kStages;
    if (!mbar_wait(&my_bar[stage], (uint32_t)((gi / kStages) & 1))) {
      ok = false;
      break;
    }
    const int tile = t_begin + warp + it * kWarps;
    const uint8_t* tb = my_ring + stage * kStageBytes;
    const int nvalid = min(kTile, count32 - tile * kTile);

    // ---- S = Q' F^T, tokens 0..7 and 8..15 (and the phi^3 pass for CODEC 2)
    float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
    float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
    {
      uint32_t f0[8][2], f1[8][2];
      k_quarter<L>(load_window(tb + g * kRec, t * F::QB), f0);
      k_quarter<L>(load_window(tb + (g + 8) * kRec, t * F::QB), f1);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint4 A = aq[32 * j];
        mma16816(s0, A.x, A.y, A.z, A.w, f0[j][0], f0[j][1]);
        mma16816(s1, A.x, A.y, A.z, A.w, f1[j][0], f1[j][1]);
        if constexpr (CODEC == 2) {
          mma16816(c0, A.x, A.y, A.z, A.w, cube_phi(f0[j][0]), cube_phi(f0[j][1]));
          mma16816(c1, A.x, A.y, A.z, A.w, cube_phi(f1[j][0]), cube_phi(f1[j][1]));
        }
      }
    }
    // ---- logits of head hd (hi + lo rows).  G > 4: lane (g, t) takes tokens 2t, 2t+1,
    // 2t+8, 2t+9 of head g.  G <= 4 (rows 4..7 empty): lane g < 4 keeps tokens 2t, 2t+1
    // and hands 2t+8, 2t+9 to lane g + 4, which works for the same head.
    constexpr int NT = PACKED ? 2 : 4;
    float S[NT], S3[NT];
    int tk[NT];
    if constexpr (PACKED) {
      const float r0 = __shfl_xor_sync(0xffffffffu, s1[0] + s1[2], 16);
      const float r1 = __shfl_xor_sync(0xffffffffu, s1[1] + s1[3], 16);
      S[0] = upper ? r0 : s0[0] + s0[2];
      S[1] = upper ? r1 : s0[1] + s0[3];
      if constexpr (CODEC == 2) {
        const float u0 = __shfl_xor_sync(0xffffffffu, c1[0] + c1[2], 16);
        const float u1 = __shfl_xor_sync(0xffffffffu, c1[1] + c1[3], 16);
        S3[0] = upper ? u0 : c0[0] + c0[2];
        S3[1] = upper ? u1 : c0[1] + c0[3];
      }
      tk[0] = 2 * t + (upper ? 8 : 0);
      tk[1] = tk[0] + 1;
    } else {
      S[0] = s0[0] + s0[2];
      S[1] = s0[1] + s0[3];
      S[2] = s1[0] + s1[2];
      S[3] = s1[1] + s1[3];
      if constexpr (CODEC == 2) {
        S3[0] = c0[0] + c0[2];
        S3[1] = c0[1] + c0[3];
        S3[2] = c1[0] + c1[2];
        S3[3] = c1[1] + c1[3];
      }
      tk[0] = 2 * t;
      tk[1] = 2 * t + 1;
      tk[2] = 2 * t + 8;
      tk[3] = 2 * t + 9;
    }
    float lg[NT], sv[NT], zv[NT], s3v[NT], p[NT], P[NT];
    bool valid[NT];
    bool bad = false;
#pragma unroll
    for (int i = 0; i < NT; ++i) {
      const uint32_t* prm = reinterpret_cast<const uint32_t*>(tb + tk[i] * kRec + 2 * F::RB);
      valid[i] = live && tk[i] < nvalid;
      float sk, zk;
      if constexpr (CODEC == 0) {
        const uint32_t kp = prm[0], vp = prm[1];
        sk = f16_to_f32((uint16_t)(kp & 0xFFFF));
        zk = f16_to_f32((uint16_t)(kp >> 16));
        // rows past the pool's count are not data: keep whatever they hold out of the sums
        sv[i] = valid[i] ? f16_to_f32((uint16_t)(vp & 0xFFFF)) : 0.0f;
        zv[i] = valid[i] ? f16_to_f32((uint16_t)(vp >> 16)) : 0.0f;
        lg[i] = fmaf(sk * cS, S[i], zk * cZ);
      } else {
        const uint32_t nn = prm[0];
        const float nk = f16_to_f32((uint16_t)(nn & 0xFFFF));
        const float nv = valid[i] ? f16_to_f32((uint16_t)(nn >> 16)) : 0.0f;
        sk = tq_s * nk;
        zk = tq_z * nk;
        sv[i] = tq_s * nv;
        zv[i] = tq_z * nv;
        lg[i] = fmaf(sk * cS, S[i], zk * cZ);
        if constexpr (CODEC == 2) {
          lg[i] = fmaf(tq_3 * nk * cS, S3[i], lg[i]);
          s3v[i] = tq_3 * nv;
        }
      }
      p[i] = valid[i] ? ex2(lg[i] - st.e) : 0.0f;
      P[i] = p[i] * sv[i];
      bad |= !(p[i] <= kPMax) || !(fabsf(P[i]) <= 16384.0f);
    }
    if (__any_sync(0xffffffffu, bad)) {
      // move e up to (max over the head's tokens of logit + log2 max(s_v, 2^-40)) - 12:
      // the largest P' lands near 2^12, well inside fp16's normal range even when the
      // value rows' steps are tiny, and p stays below 2^52 so the fp32 sums of p and
      // p z_v cannot overflow
      float mx = -INFINITY;
#pragma unroll
      for (int i = 0; i < NT; ++i)
        if (valid[i]) mx = fmaxf(mx, lg[i] + fmaxf(-40.0f, __log2f(fabsf(sv[i]))));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      if (PACKED) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
      const float e_new = fmaxf(st.e, mx - 12.0f);
      const float al = st.e == -INFINITY ? 0.0f : ex2(st.e - e_new);
      st.e = e_new;
      st.l *= al;
      st.zs *= al;
      const float a0 = __shfl_sync(0xffffffffu, al, 4 * oh0);
      const float a1 = __shfl_sync(0xffffffffu, al, 4 * oh1);
#pragma unroll
      for (int m = 0; m < 8; ++m) {
        st.O[m][0] *= a0;
        st.O[m][1] *= a1;
        st.O[m][2] *= a0;
        st.O[m][3] *= a1;
      }
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        p[i] = valid[i] ? ex2(lg[i] - st.e) : 0.0f;
        P[i] = p[i] * sv[i];
      }
    }
#pragma unroll
    for (int i = 0; i < NT; ++i) {
      st.l += p[i];
      st.zs = fmaf(p[i], zv[i], st.zs);
    }
    // ---- P'^T as the B fragment: rows = tokens (2t, 2t+1 | 2t+8, 2t+9), column g
    uint32_t b0, b1, b0l = 0u, b1l = 0u;
    if constexpr (PACKED) {
      // column g < 4: hi parts of head g; column g + 4: lo parts of head g
      uint32_t hi, lo;
      split_h2(P[0], P[1], hi, lo);
      const uint32_t recv = __shfl_xor_sync(0xffffffffu, upper ? hi : lo, 16);
      b0 = upper ? recv : hi;
      b1 = upper ? lo : recv;
    } else {
      split_h2(P[0], P[1], b0, b0l);
      split_h2(P[2], P[3], b1, b1l);
    }
    // ---- O^T += C^T P'^T
    {
      uint32_t VA[8][4];
      v_half_pair<L, 0>(load_window(tb + (2 * t) * kRec, vpos),
                        load_window(tb + (2 * t + 1) * kRec, vpos), tpos, hh, VA);
      v_half_pair<L, 2>(load_window(tb + (2 * t + 8) * kRec, vpos),
                        load_window(tb + (2 * t + 9) * kRec, vpos), tpos, hh, VA);
#pragma unroll
      for (int m = 0; m < 8; ++m) {
        mma16816(st.O[m], VA[m][0], VA[m][1], VA[m][2], VA[m][3], b0, b1);
        if constexpr (!PACKED)
          mma16816(st.O[m], VA[m][0], VA[m][1], VA[m][2], VA[m][3], b0l, b1l);
      }
      if constexpr (CODEC == 2) {
        // the phi^3 pass: the same digits cubed, weighted by P3 = p * beta n / 128
        uint32_t e0, e1, e0l = 0u, e1l = 0u;
        float P3[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) P3[i] = p[i] * s3v[i];
        if constexpr (PACKED) {
          uint32_t hi, lo;
          split_h2(P3[0], P3[1], hi, lo);
          const uint32_t recv = __shfl_xor_sync(0xffffffffu, upper ? hi : lo, 16);
          e0 = upper ? recv : hi;
          e1 = upper ? lo : recv;
        } else {
          split_h2(P3[0], P3[1], e0, e0l);
          split_h2(P3[2], P3[3], e1, e1l);
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
          const uint32_t x0 = cube_phi(VA[m][0]), x1 = cube_phi(VA[m][1]);
          const uint32_t x2 = cube_phi(VA[m][2]), x3 = cube_phi(VA[m][3]);
          mma16816(st.O[m], x0, x1, x2, x3, e0, e1);
          if constexpr (!PACKED) mma16816(st.O[m], x0, x1, x2, x3, e0l, e1l);
        }
      }
    }
    __syncwarp();
    {
      // the stage is free again: lane 0 starts the copy of the tile kStages ahead
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      const int nt = t_begin + warp + (it + kStages) * kWarps;
      bulk_refill(lane == 0 && it + kStages < nmine, my_ring + stage * kStageBytes,
                  pool_bh + (int64_t)nt * kTileBytes, kTileBytes, &my_bar[stage]);
    }
  }
  if (!ok) {
    // a copy never completed: record it, give the copies still in flight a bounded
    // chance to land, and drop this warp's contribution
    if (lane == 0) raise_error(a.err, kDevWaitTimeout);
    for (int j = it; j < nmine && j < it + kStages; ++j)
      mbar_wait(&my_bar[(ring_it + j) % kStages], (uint32_t)(((ring_it + j) / kStages) & 1));
    state_init(st);
  }
  ring_it += nmine;
}

// ==================================================== affine pools: fast path =====
// Five- and six-level affine pools with GQA groups of up to four heads (the shape of
// the paper's models and of every workload here), in a kernel of its own so that it
// gets its own register budget (decode_affine_fast_kernel).
//
// S^T = F Q'^T on m16n8k16: M = the tile's 16 tokens, N = 8 columns (column 2h holds
// the hi part of head h's coefficients, 2h + 1 the lo part), K = 16 F slots per step,
// 8 steps: eight MMAs per tile.  Lane (g, t) supplies the F values of quarter t of
// tokens g and g + 8 (A fragment) and the coefficients of head g>>1, part g&1, for the
// same slots (B fragment: 16 registers built once per segment, no per-tile loads); its
// output holds the logits of tokens g and g + 8 for head t.  The softmax runs on those
// two logits per lane; four shuffles and two byte permutes hand P' = p s_v to the
// lanes that hold it in the PV product's B fragment.
//
// Five-level symbols are decoded on the f16x2 FMA pipe.  The mask that extracts a
// pair of symbols also lays the fp16 exponent of 1024 over them, giving the halves
// B = 1024 + beta.  fma(B, 5^(k+1)/128, 1025.5 - 1024 * 5^(k+1)/128) is then
// 1026 + F_k + (f - 1/2) before rounding, f the fraction of beta 5^(k+1)/128: a
// multiple of 1/128, nonzero unless beta = 0 (5 is prime to 128).  So it rounds to
// 1026 + F_k: for f > 0 the offset f - 1/2 lies strictly inside (-1/2, 1/2), and for
// beta = 0 the tie 1025.5 goes to the even 1026.  Subtracting 1026 leaves F_k.  (Every
// constant is exact in fp16; the values stay in [1024, 2048), where fp16's step is 1.)
// Six-level symbols keep the binary32 multiplies of Dec<6> (their 13-bit symbols do
// not fit fp16's 11 bits).

__device__ __forceinline__ uint32_t hfma2u(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t r;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(c));
  return r;
}
// x - 1026 on both halves
__device__ __forceinline__ uint32_t hsub1026(uint32_t x) {
  uint32_t r;
  asm("add.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(x), "r"(0xE402E402u));
  return r;
}
// (x & m) | ov in one LOP3: ov (the fp16 exponent of 1024 in both halves) comes from a
// register the caller made once, so the two constants never both need an immediate
__device__ __forceinline__ uint32_t and_or(uint32_t x, uint32_t m, uint32_t ov) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(x), "r"(m), "r"(ov));
  return r;
}
__device__ __forceinline__ uint32_t overlay1024() {
  uint32_t ov;
  asm volatile("mov.b32 %0, 0x64006400;" : "=r"(ov));
  return ov;
}

// fp16 constants of the five-level digit fmas: 5^(k+1)/128 and 1025.5 - 1024 5^(k+1)/128
__host__ __device__ constexpr uint32_t l5_mul(int k) {
  return k == 0 ? 0x29002900u : k == 1 ? 0x32403240u : 0x3BD03BD0u;
}
__host__ __device__ constexpr uint32_t l5_add(int k) {
  return k == 0 ? 0x63B363B3u : k == 1 ? 0x62736273u : 0x4E604E60u;
}
// the two-code tail (5 bits): F_0 = floor(beta 5/32), F_1 = floor(beta 25/32)
constexpr uint32_t kL5TMul0 = 0x31003100u, kL5TAdd0 = 0x62C362C3u;
constexpr uint32_t kL5TMul1 = 0x3A403A40u, kL5TAdd1 = 0x5B0C5B0Cu;
constexpr uint32_t kL5TMulK = 0x3A403100u, kL5TAddK = 0x5B0C62C3u;  // F_0 low, F_1 high

// B = 1024 + beta pairs of five symbols: symbol j (bits 7j) of the window (a0, a1)
// in the low half and of the window (b0, b1) in the high half
__device__ __forceinline__ void l5_pairsB(uint32_t a0, uint32_t a1, uint32_t b0, uint32_t b1,
                                          uint32_t ov, uint32_t (&B)[5]) {
  const uint32_t C = fpair(a0, b0);                                 // bits 0..15 of each
  B[0] = and_or(C, kM7, ov);
  B[1] = and_or(C >> 7, kM7, ov);
  B[2] = and_or(__byte_perm(a0, b0, 0x6521) >> 6, kM7, ov);         // bits 8..23, >> 6
  B[3] = and_or(__byte_perm(a0, b0, 0x7632) >> 5, kM7, ov);         // bits 16..31, >> 5
  B[4] = and_or(fpair(__funnelshift_r(a0, a1, 28), __funnelshift_r(b0, b1, 28)), kM7, ov);
}

// K side: the B pairs of one quarter (symbols s and s + 5, 35 bits apart) and its tail
// (in both halves).  Register p of the quarter's A-fragment halves: p < 15: F_(p%3)
// of symbols p/3 (low half) and p/3 + 5 (high half); p = 15: the tail's F_0, F_1.
__device__ __forceinline__ void k5_B(const Window& w, uint32_t ov, uint32_t (&B)[5], uint32_t& Bt) {
  l5_pairsB(w.q0, w.q1, __funnelshift_r(w.q1, w.q2, 3), w.q2 >> 3, ov, B);
  Bt = ((w.q2 >> 6) & 0x1Fu) * 0x00010001u + 0x64006400u;          // quarter bits 70..74
}
__device__ __forceinline__ uint32_t k5_reg(const uint32_t (&B)[5], uint32_t Bt, int p) {
  return p < 15 ? hsub1026(hfma2u(B[p / 3], l5_mul(p % 3), l5_add(p % 3)))
                : hsub1026(hfma2u(Bt, kL5TMulK, kL5TAddK));
}
// V side: the B pairs (tokens of wa low, wb high) of lane group g's half quarter and
// the pair of its tail symbols (70 bits on for half 0, 35 for half 1); the digits of
// one symbol; the tail's digit hh (F_hh - 5 hh F_0)
__device__ __forceinline__ void v5_B(const Window& wa, const Window& wb, int hh, uint32_t ov,
                                     uint32_t (&B)[5], uint32_t& Bt) {
  l5_pairsB(wa.q0, wa.q1, wb.q0, wb.q1, ov, B);
  const uint32_t ta = hh ? (wa.q1 >> 3) : (wa.q2 >> 6);
  const uint32_t tb = hh ? (wb.q1 >> 3) : (wb.q2 >> 6);
  Bt = and_or(fpair(ta, tb), 0x001F001Fu, ov);
}
__device__ __forceinline__ void v5_digits(uint32_t B, uint32_t& d0, uint32_t& d1, uint32_t& d2) {
  const uint32_t F0 = hsub1026(hfma2u(B, l5_mul(0), l5_add(0)));
  const uint32_t F1 = hsub1026(hfma2u(B, l5_mul(1), l5_add(1)));
  const uint32_t F2 = hsub1026(hfma2u(B, l5_mul(2), l5_add(2)));
  d0 = F0;
  d1 = hdigit<5>(F0, F1);
  d2 = hdigit<5>(F1, F2);
}
__device__ __forceinline__ uint32_t v5_tail(uint32_t Bt, uint32_t tmul, uint32_t tadd, uint32_t tneg) {
  const uint32_t T0 = hsub1026(hfma2u(Bt, kL5TMul0, kL5TAdd0));
  const uint32_t Th = hsub1026(hfma2u(Bt, tmul, tadd));
  return hfma2u(T0, tneg, Th);
}

// packed binary32 pairs (Blackwell's f32x2 arithmetic: one instruction for two lanes)
__device__ __forceinline__ unsigned long long f2_bits(float2 v) {
  return (unsigned long long)__float_as_uint(v.x) | ((unsigned long long)__float_as_uint(v.y) << 32);
}
__device__ __forceinline__ float2 f2_of(unsigned long long r) {
  return make_float2(__uint_as_float((uint32_t)r), __uint_as_float((uint32_t)(r >> 32)));
}
__device__ __forceinline__ float2 f2_fma(float2 a, float2 b, float2 c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(f2_bits(a)), "l"(f2_bits(b)), "l"(f2_bits(c)));
  return f2_of(r);
}
__device__ __forceinline__ float2 f2_mul(float2 a, float2 b) {
  unsigned long long r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(f2_bits(a)), "l"(f2_bits(b)));
  return f2_of(r);
}
__device__ __forceinline__ float2 f2_add(float2 a, float2 b) {
  unsigned long long r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(f2_bits(a)), "l"(f2_bits(b)));
  return f2_of(r);
}
__device__ __forceinline__ float2 neg_f2(float2 a) { return make_float2(-a.x, -a.y); }
// fp16 pair (low half = x) <-> two binary32
__device__ __forceinline__ float2 h2_to_f2(uint32_t h) {
  return make_float2(f16_to_f32((uint16_t)(h & 0xFFFFu)), f16_to_f32((uint16_t)(h >> 16)));
}
__device__ __forceinline__ uint32_t f2_to_h2(float2 v) { return pack_h2(v.x, v.y); }

// A 96-bit window read with 32-bit shared-memory addressing: addr is the shared address
// of the word holding the window's first bit, sh the bit offset in it.  (volatile keeps
// the loads after the tile's mbarrier wait.)
__device__ __forceinline__ Window load_window_s(uint32_t addr, uint32_t sh) {
  uint32_t w0, w1, w2, w3;
  asm volatile(
      "ld.shared.u32 %0, [%4];\n\t"
      "ld.shared.u32 %1, [%4+4];\n\t"
      "ld.shared.u32 %2, [%4+8];\n\t"
      "ld.shared.u32 %3, [%4+12];"
      : "=r"(w0), "=r"(w1), "=r"(w2), "=r"(w3)
      : "r"(addr));
  Window r;
  r.q0 = __funnelshift_r(w0, w1, sh);
  r.q1 = __funnelshift_r(w1, w2, sh);
  r.q2 = __funnelshift_r(w2, w3, sh);
  return r;
}
__device__ __forceinline__ uint2 ld_shared_u2(uint32_t addr) {
  uint32_t x, y;
  asm volatile("ld.shared.u32 %0, [%2];\n\tld.shared.u32 %1, [%2+4];" : "=r"(x), "=r"(y) : "r"(addr));
  return make_uint2(x, y);
}

struct FastState {
  float O[8][4];  // O^T accumulators: V rows x columns 2t, 2t+1
  float e;        // reference exponent of head t (base 2)
  float l, l2;    // partial sums of p over this lane's tokens g and g + 8 of head t
  float zs, zs2;  // partial sums of p z_v
};

__device__ __forceinline__ void fast_init(FastState& st) {
#pragma unroll
  for (int m = 0; m < 8; ++m)
#pragma unroll
    for (int i = 0; i < 4; ++i) st.O[m][i] = 0.0f;
  st.e = -INFINITY;
  st.l = st.l2 = 0.0f;
  st.zs = st.zs2 = 0.0f;
}

// the power-of-two scale that brings head coefficients near 2^13
__device__ __forceinline__ float coef_scale(float qmax, int L) {
  return qmax > 0.0f ? pow2_floor(fminf(8192.0f / ((float)(L + 1) * qmax), 1e30f)) : 1.0f;
}

// One warp streams its tiles of one (pair, pool) segment (see the section comment),
// two consecutive tiles per copy: the segment's tiles [t_begin, t_end) form chunks of
// kChunk tiles (the last may hold one) and warp w of NW takes chunks w, w + NW, ...
// ring_it: chunks this warp has taken through its ring so far (barrier phases).
template <int L, int NW>
__device__ void run_pool_fast(const DecodeArgs& a, const Shared& sh, uint8_t* ring, uint2* qbs,
                              uint64_t* bars, const uint8_t* pool_bh, int64_t count,
                              int t_begin, int t_end, int G, FastState& st, int& ring_it) {
  using D = Dec<L>;
  using F = typename D::F;
  constexpr int kRec = 2 * F::RB + 8;
  constexpr uint32_t kTileBytes = kTile * kRec;
  static_assert(kTileBytes % 16 == 0, "tile size must be a multiple of 16 bytes");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  uint8_t* my_ring = ring + warp * kFastStages * kFastStageBytes;
  uint64_t* my_bar = bars + warp * kStages;
  const bool rot = a.base == SEMKV_BASE_AFFINE_HAD;

  // B fragments: coefficients of head g>>1 (hi part for even g, lo part for odd g) for
  // the slots of lane (g, t), the same for every warp: warp w builds step w for every
  // lane into shared memory, then every warp loads its lane's pair per step (one
  // conflict-free 8-byte load)
  static_assert(kWarps >= 8, "one warp per coefficient step");
  __syncthreads();  // the previous segment's fragments and the merge area are no longer read
  if (warp < 8) {
    const int hb = g >> 1, j = warp;
    const float sc = coef_scale(sh.qmax[hb], L);
    uint32_t r[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int p = 2 * j + i;
      float c0 = 0.0f, c1 = 0.0f;
      if (hb < G) {
        if (rot) {
          c0 = k_coef<L>(sh.qr[hb], t, p, 0) * sc;
          c1 = k_coef<L>(sh.qr[hb], t, p, 1) * sc;
        } else {
          c0 = k_coef<L>(sh.q[hb], t, p, 0) * sc;
          c1 = k_coef<L>(sh.q[hb], t, p, 1) * sc;
        }
      }
      uint32_t hi, lo;
      split_h2(c0, c1, hi, lo);
      r[i] = (g & 1) ? lo : hi;
    }
    qbs[32 * j + lane] = make_uint2(r[0], r[1]);
  }
  __syncthreads();
  const uint2* qb = qbs + lane;
  // logits of head t
  const bool live = t < G;
  const float cS = a.scale_log2 / coef_scale(sh.qmax[t], L);
  const float cZ = a.scale_log2 * sh.sumq[t];
  // O columns 2t, 2t+1 belong to heads (2t)&3, (2t+1)&3, whose e lives in lanes 0..3
  const int oh0 = (2 * t) & 3, oh1 = oh0 + 1;
  // P' hand-over: this lane's PV column g is head g&3, part g>>2; its rows are tokens
  // 2t, 2t+1 (lanes 8t + (g&3), + 4) and 2t+8, 2t+9
  const int srcX = 8 * t + (g & 3), srcY = srcX + 4;
  const uint32_t psel = (g >> 2) ? 0x7632u : 0x5410u;
  // V half quarter of lane group g, and its tail digit's constants
  const int qv = g >> 1, hh = g & 1;
  const int vpos = 8 * F::RB + qv * F::QB + hh * D::kHalf * F::W;
  const int tpos = F::NG * F::W - hh * D::kHalf * F::W;
  const uint32_t tmul = hh ? kL5TMul1 : kL5TMul0, tadd = hh ? kL5TAdd1 : kL5TAdd0;
  const uint32_t tneg = hh ? 0xC500C500u : 0u;
  const uint32_t ov = overlay1024();
  const int kpos = t * F::QB;
  // 32-bit shared addresses: the ring, and per lane the word offsets of its windows in a
  // tile and their bit shifts
  const uint32_t ring_s = smem_u32(my_ring);
  const uint32_t kw0 = g * kRec + 4 * (kpos >> 5), kw1 = kw0 + 8 * kRec, ksh = kpos & 31;
  const uint32_t vw0 = 2 * t * kRec + 4 * (vpos >> 5), vsh = vpos & 31;
  const uint32_t pw0 = g * kRec + 2 * F::RB, pw1 = pw0 + 8 * kRec;

  // one 16-token tile at shared address ts whose first nvalid rows are tokens of the pool
  auto run_tile = [&](const uint32_t ts, const int nvalid) {
    // ---- S^T = F Q'^T: tokens g (rows g) and g + 8, heads in column pairs
    float s[4] = {0.f, 0.f, 0.f, 0.f};
    {
      if constexpr (L == 5) {
        uint32_t Ba[5], Bb[5], Ta, Tb;
        k5_B(load_window_s(ts + kw0, ksh), ov, Ba, Ta);
        k5_B(load_window_s(ts + kw1, ksh), ov, Bb, Tb);
#pragma unroll
        for (int j = 0; j < 8; ++j)
        {
          const uint2 c = qb[32 * j];
          mma16816(s, k5_reg(Ba, Ta, 2 * j), k5_reg(Bb, Tb, 2 * j), k5_reg(Ba, Ta, 2 * j + 1),
                   k5_reg(Bb, Tb, 2 * j + 1), c.x, c.y);
        }
      } else {
        uint32_t fa[8][2], fb[8][2];
        k_quarter<L>(load_window_s(ts + kw0, ksh), fa);
        k_quarter<L>(load_window_s(ts + kw1, ksh), fb);
#pragma unroll
        for (int j = 0; j < 8; ++j)
        {
          const uint2 c = qb[32 * j];
          mma16816(s, fa[j][0], fb[j][0], fa[j][1], fb[j][1], c.x, c.y);
        }
      }
    }
    // ---- softmax of head t over tokens g and g + 8
    const bool v0 = live && g < nvalid, v1 = live && g + 8 < nvalid;
    const uint2 pr0 = ld_shared_u2(ts + pw0), pr1 = ld_shared_u2(ts + pw1);
    const uint32_t kp0 = pr0.x, kp1 = pr1.x;
    // rows past the pool's count are not data: keep whatever they hold out of the sums
    const uint32_t vp0 = v0 ? pr0.y : 0u, vp1 = v1 ? pr1.y : 0u;
    // both tokens at once in packed binary32 (x: token g, y: token g + 8)
    const float2 k0 = h2_to_f2(kp0), k1 = h2_to_f2(kp1), vv0 = h2_to_f2(vp0), vv1 = h2_to_f2(vp1);
    const float2 lg = f2_fma(f2_mul(make_float2(k0.x, k1.x), make_float2(cS, cS)),
                             make_float2(s[0] + s[1], s[2] + s[3]),
                             f2_mul(make_float2(k0.y, k1.y), make_float2(cZ, cZ)));
    const float2 sv = make_float2(vv0.x, vv1.x), zv = make_float2(vv0.y, vv1.y);
    float2 dl = f2_add(lg, make_float2(-st.e, -st.e));
    float2 p = make_float2(v0 ? ex2(dl.x) : 0.0f, v1 ? ex2(dl.y) : 0.0f);
    float2 P = f2_mul(p, sv);
    const bool bad = !(fmaxf(p.x, p.y) <= kPMax) || !(fmaxf(fabsf(P.x), fabsf(P.y)) <= 16384.0f);
    if (__any_sync(0xffffffffu, bad)) {
      // e of each head moves up to (max over its tokens of logit + log2 max(s_v, 2^-40))
      // - 12: the largest P' lands near 2^12, p stays below 2^52
      float mx = -INFINITY;
      if (v0) mx = lg.x + fmaxf(-40.0f, __log2f(fabsf(sv.x)));
      if (v1) mx = fmaxf(mx, lg.y + fmaxf(-40.0f, __log2f(fabsf(sv.y))));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
      const float e_new = fmaxf(st.e, mx - 12.0f);
      const float al = st.e == -INFINITY ? 0.0f : ex2(st.e - e_new);
      st.e = e_new;
      st.l *= al;
      st.l2 *= al;
      st.zs *= al;
      st.zs2 *= al;
      const float a0 = __shfl_sync(0xffffffffu, al, oh0);
      const float a1 = __shfl_sync(0xffffffffu, al, oh1);
#pragma unroll
      for (int m = 0; m < 8; ++m) {
        st.O[m][0] *= a0;
        st.O[m][1] *= a1;
        st.O[m][2] *= a0;
        st.O[m][3] *= a1;
      }
      dl = f2_add(lg, make_float2(-st.e, -st.e));
      p = make_float2(v0 ? ex2(dl.x) : 0.0f, v1 ? ex2(dl.y) : 0.0f);
      P = f2_mul(p, sv);
    }
    {
      // the two tokens' sums stay apart (l, l2 and zs, zs2) so one packed op adds both
      const float2 l2 = f2_add(make_float2(st.l, st.l2), p);
      const float2 z2 = f2_fma(p, zv, make_float2(st.zs, st.zs2));
      st.l = l2.x;
      st.l2 = l2.y;
      st.zs = z2.x;
      st.zs2 = z2.y;
    }
    // ---- P'^T as the PV product's B fragment (rows = tokens, column g)
    uint32_t b0, b1;
    {
      // fp16 hi and lo parts of both tokens' P', then (hi, lo) per token
      const uint32_t hp = f2_to_h2(P);
      const float2 lo = f2_add(P, neg_f2(h2_to_f2(hp)));
      const uint32_t lp = f2_to_h2(lo);
      const uint32_t W0 = __byte_perm(hp, lp, 0x5410), W1 = __byte_perm(hp, lp, 0x7632);
      const uint32_t x0 = __shfl_sync(0xffffffffu, W0, srcX);
      const uint32_t x1 = __shfl_sync(0xffffffffu, W1, srcX);
      const uint32_t y0 = __shfl_sync(0xffffffffu, W0, srcY);
      const uint32_t y1 = __shfl_sync(0xffffffffu, W1, srcY);
      b0 = __byte_perm(x0, y0, psel);
      b1 = __byte_perm(x1, y1, psel);
    }
    // ---- O^T += C^T P'^T
    {
      const Window w0 = load_window_s(ts + vw0, vsh);
      const Window w1 = load_window_s(ts + vw0 + kRec, vsh);
      const Window w2 = load_window_s(ts + vw0 + 8 * kRec, vsh);
      const Window w3 = load_window_s(ts + vw0 + 9 * kRec, vsh);
      if constexpr (L == 5) {
        // symbol by symbol: after symbol j, rows 0 .. 3j + 2 are ready and the m-blocks
        // up to (3j + 1) / 2 go to the tensor cores
        uint32_t B0[5], B1[5], T0, T1;
        v5_B(w0, w1, hh, ov, B0, T0);
        v5_B(w2, w3, hh, ov, B1, T1);
        uint32_t r0[16], r1[16];
#pragma unroll
        for (int j = 0; j < 5; ++j) {
          v5_digits(B0[j], r0[3 * j], r0[3 * j + 1], r0[3 * j + 2]);
          v5_digits(B1[j], r1[3 * j], r1[3 * j + 1], r1[3 * j + 2]);
#pragma unroll
          for (int m = (3 * j - 2 < 0 ? 0 : (3 * j - 2) / 2 + 1); m <= (3 * j + 1) / 2; ++m)
            mma16816(st.O[m], r0[2 * m], r0[2 * m + 1], r1[2 * m], r1[2 * m + 1], b0, b1);
        }
        r0[15] = v5_tail(T0, tmul, tadd, tneg);
        r1[15] = v5_tail(T1, tmul, tadd, tneg);
        mma16816(st.O[7], r0[14], r0[15], r1[14], r1[15], b0, b1);
      } else {
        uint32_t VA[8][4];
        v_half_pair<L, 0>(w0, w1, tpos, hh, VA);
        v_half_pair<L, 2>(w2, w3, tpos, hh, VA);
#pragma unroll
        for (int m = 0; m < 8; ++m)
          mma16816(st.O[m], VA[m][0], VA[m][1], VA[m][2], VA[m][3], b0, b1);
      }
    }
  };

  const int nchunks = (t_end - t_begin + kChunk - 1) / kChunk;
  const int nmine = nchunks <= warp ? 0 : (nchunks - warp + NW - 1) / NW;
  // first tile of this warp's current chunk (a pool holds fewer than 2^31 slots), the
  // ring position
  int tile = t_begin + warp * kChunk;
  int stage = ring_it % kFastStages;
  uint32_t phase = (uint32_t)((ring_it / kFastStages) & 1);
  bool ok = true;
  int it = 0;
  for (; it < nmine; ++it) {
    if (!mbar_wait(&my_bar[stage], phase)) {
      ok = false;
      break;
    }
    const uint32_t cs = ring_s + stage * kFastStageBytes;
    const int left = (int)count - tile * kTile;  // tokens of the pool from this chunk on
    run_tile(cs, min(kTile, left));
#pragma unroll
    for (int j = 1; j < kChunk; ++j)
      if (tile + j < t_end) run_tile(cs + j * kTileBytes, min(kTile, left - j * kTile));
    __syncwarp();
    // the stage is free again: lane 0 starts the copy of the chunk kFastStages ahead
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    const int nt = tile + kFastStages * NW * kChunk;
    bulk_refill(lane == 0 && it + kFastStages < nmine, my_ring + stage * kFastStageBytes,
                pool_bh + (int64_t)nt * kTileBytes, (uint32_t)min(kChunk, t_end - nt) * kTileBytes,
                &my_bar[stage]);
    tile += NW * kChunk;
    if (++stage == kFastStages) {
      stage = 0;
      phase ^= 1u;
    }
  }
  if (!ok) {
    // a copy never completed: record it, give the copies still in flight a bounded
    // chance to land, and drop this warp's contribution
    if (lane == 0) raise_error(a.err, kDevWaitTimeout);
    for (int j = it; j < nmine && j < it + kFastStages; ++j)
      mbar_wait(&my_bar[(ring_it + j) % kFastStages],
                (uint32_t)(((ring_it + j) / kFastStages) & 1));
    fast_init(st);
  }
  ring_it += nmine;
}

// ------------------------------------------------- TurboQuant-MSE records -----
// Dequantized rows are x^ = (n/128) S H cb[c] (Sec. 4.9), so q . x^ = (n/128) q' . cb[c]
// with q' = H S q, and sum p x^ = S H (sum p (n/128) cb[c]): scores and the weighted
// sum run in the rotated domain and each CTA rotates its partial back at the end.
// One warp per token on the CUDA cores: lane l holds dims 4l..4l+3 of both rows.

// digit k of the group symbol beta (compile-time level, run-time k)
template <int L>
__device__ __forceinline__ uint32_t digit_rt(uint32_t beta, int k) {
  using D = Dec<L>;
  using F = typename D::F;
  if constexpr (D::G == 1) {
    return fdig(beta, (float)L / (float)(1u << F::W));
  } else {
    // chain start and the multiplier of F_k within its chain
    const int k0 = (k >= D::kRestart) ? D::kRestart : 0;
    const uint32_t x = (k0 == 0) ? beta : ((beta * 36u) & 8191u);  // restart: six levels only
    float c = (float)L / (float)(1u << F::W);
    for (int j = k0; j < k; ++j) c *= (float)L;
    const uint32_t Fk = fdig(x, c);
    if (k == k0) return Fk;
    return Fk - (uint32_t)L * fdig(x, c / (float)L);
  }
}
template <int L>
__device__ __forceinline__ uint32_t tail_digit(uint32_t beta, int k) {
  using F = Fmt<L>;
  const float c = (float)L / (float)(1u << F::WT);
  const uint32_t F0 = fdig(beta, c);
  return k == 0 ? F0 : fdig(beta, c * (float)L) - (uint32_t)L * F0;
}
// 96 bits from bit `pos` of a record in global memory, reading no word at or past
// bit `end` (the end of the row): the last record of a pool may end its allocation
__device__ __forceinline__ Window load_window_bounded(const uint8_t* rec, int pos, int end) {
  const uint32_t* w = reinterpret_cast<const uint32_t*>(rec) + (pos >> 5);
  const int first = pos >> 5, last = (end - 1) >> 5;
  uint32_t v[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) v[i] = (first + i <= last) ? w[i] : 0u;
  const int sh = pos & 31;
  Window r;
  r.q0 = __funnelshift_r(v[0], v[1], sh);
  r.q1 = __funnelshift_r(v[1], v[2], sh);
  r.q2 = __funnelshift_r(v[2], v[3], sh);
  return r;
}

// the codes of dims 4l..4l+3 of the row starting at bit `row_bit` of a record
template <int L>
__device__ __forceinline__ void tq_codes4(const uint8_t* rec, int row_bit, int lane, uint32_t c[4]) {
  using D = Dec<L>;
  using F = typename D::F;
  const int q = lane >> 3, i0 = 4 * (lane & 7);
  const Window w = load_window_bounded(rec, row_bit + q * F::QB, row_bit + 8 * F::RB);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int i = i0 + j;
    if (F::R > 0 && i >= 32 - F::R) {
      c[j] = tail_digit<L>(wbits(w, F::NG * F::W, F::WT), i - (32 - F::R));
    } else {
      const int s = i / D::G, k = i % D::G;
      c[j] = digit_rt<L>(wbits_rt(w, s * F::W, F::W), k);
    }
  }
}

template <int L>
__device__ void run_pool_tq(const DecodeArgs& a, const Shared& sh, int which,
                            const uint8_t* pool_bh, int64_t count, int t_begin, int t_end,
                            int G, float* m_out, float* l_out, float* z_out, float* o_out) {
  using F = Fmt<L>;
  constexpr int kRec = 2 * F::RB + 4;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float qf[8][4];
#pragma unroll
  for (int c = 0; c < 8; ++c)
#pragma unroll
    for (int j = 0; j < 4; ++j) qf[c][j] = c < G ? sh.qr[c][4 * lane + j] : 0.0f;
  float m[8], l[8], o[8][4];
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    m[c] = -INFINITY;
    l[c] = 0.0f;
#pragma unroll
    for (int j = 0; j < 4; ++j) o[c][j] = 0.0f;
  }
  const int64_t i_end = min((int64_t)t_end * kTile, count);
  for (int64_t i = (int64_t)t_begin * kTile + warp; i < i_end; i += kWarps) {
    const uint8_t* rec = pool_bh + i * kRec;
    uint32_t ck[4], cv[4];
    tq_codes4<L>(rec, 0, lane, ck);
    tq_codes4<L>(rec, 8 * F::RB, lane, cv);
    const uint32_t nn = *reinterpret_cast<const uint32_t*>(rec + 2 * F::RB);
    const float nk = f16_to_f32((uint16_t)(nn & 0xFFFF)) * (1.0f / 128.0f);
    const float nv = f16_to_f32((uint16_t)(nn >> 16)) * (1.0f / 128.0f);
    float kv[4], vv[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      kv[j] = sh.cb[which][ck[j]] * nk;
      vv[j] = sh.cb[which][cv[j]] * nv;
    }
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      if (c >= G) break;
      float d = qf[c][0] * kv[0] + qf[c][1] * kv[1] + qf[c][2] * kv[2] + qf[c][3] * kv[3];
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off);
      const float lg = d * a.scale_log2;
      const float mn = fmaxf(m[c], lg);
      const float al = m[c] == -INFINITY ? 0.0f : exp2f(m[c] - mn);
      const float pp = exp2f(lg - mn);
      m[c] = mn;
      l[c] = l[c] * al + pp;
#pragma unroll
      for (int j = 0; j < 4; ++j) o[c][j] = o[c][j] * al + pp * vv[j];
    }
  }
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    if (c >= G) break;
    if (lane == 0) {
      m_out[warp * 8 + c] = m[c];
      l_out[warp * 8 + c] = l[c];
      z_out[warp * 8 + c] = 0.0f;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) o_out[mo_at(warp * 8 + c, 4 * lane + j)] = o[c][j];
  }
}

// Dense rotation: q' = M q for the G query heads of each (sequence, KV head); one block
// of 128 threads per pair, thread i taking row i of M (16 independent 16-byte loads)
// against the group's queries staged in shared memory.
__global__ void qrot_dense_kernel(DecodeArgs a) {
  __shared__ float qs[8][128];
  const int b = blockIdx.x / a.H, h = blockIdx.x % a.H;
  const int G = a.Hq / a.H, i = threadIdx.x;
  for (int x = threadIdx.x; x < G * 128; x += blockDim.x)
    qs[x >> 7][x & 127] = f16_to_f32(a.q[((int64_t)b * a.Hq + h * G) * 128 + x]);
  __syncthreads();
  const uint4* row = reinterpret_cast<const uint4*>(a.rot + (((int64_t)a.layer * a.H + h) * 128 + i) * 128);
  uint4 m[16];
#pragma unroll
  for (int c = 0; c < 16; ++c) m[c] = row[c];
  for (int g = 0; g < G; ++g) {
    float acc = 0.0f;
#pragma unroll
    for (int c = 0; c < 16; ++c) {
      const uint32_t w[4] = {m[c].x, m[c].y, m[c].z, m[c].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        acc = fmaf(f16_to_f32((uint16_t)(w[e] & 0xFFFF)), qs[g][8 * c + 2 * e], acc);
        acc = fmaf(f16_to_f32((uint16_t)(w[e] >> 16)), qs[g][8 * c + 2 * e + 1], acc);
      }
    }
    a.qrot[((int64_t)b * a.Hq + h * G + g) * 128 + i] = acc;
  }
}

// ------------------------------------------------------- fp16 stage tokens ----

// Staged tokens are few (< block): one warp per token, lane = 4 dims, CUDA cores.
// Writes rows in natural dim order and zs = 0.
__device__ void run_stage(const DecodeArgs& a, const Shared& sh, int b, int h, int G,
                          float* m_out, float* l_out, float* z_out, float* o_out) {
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
      z_out[warp * 8 + c] = 0.0f;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) o_out[mo_at(warp * 8 + c, 4 * lane + j)] = o[c][j];
  }
}

// -------------------------------------------------------------- kernel --------

// balanced plan: the partial slots of pair bh's hi and lo segments
__host__ __device__ inline int seg_slots(const DecodePlan& P, int64_t s, int64_t e) {
  return e > s ? (int)((e - 1) / P.per - s / P.per + 1) : 0;
}
__host__ __device__ inline void pair_slots(const DecodePlan& P, int64_t bh, int& n_hi, int& n_lo) {
  const int64_t s = bh * P.W, m = s + (int64_t)P.w_hi * P.tiles_hi, e = s + P.W;
  n_hi = seg_slots(P, s, m);
  n_lo = seg_slots(P, m, e);
}
// partial slots used by pair bh (pools, then the stage)
__host__ __device__ inline int pair_partials(const DecodePlan& P, int64_t bh) {
  if (!P.balanced) return P.splits;
  int n_hi, n_lo;
  pair_slots(P, bh, n_hi, n_lo);
  return n_hi + n_lo + P.splits_st;
}

struct MergeArea {
  float m[kMaxWarps * 8], l[kMaxWarps * 8], z[kMaxWarps * 8];
  float scale[kMaxWarps * 8], cta_z[8];
};

// the group's queries of pair (b, h) into shared memory, with their sums and maxima
// (every thread of the CTA calls this; the caller orders it after earlier readers)
// (rotated affine base: also the rotated queries into sh.qr, which the sums then follow)
// A CTA of NW warps' share of the group's query values (thread i: values i, i + 32 NW,
// ...): loaded into registers before a segment's first copies are issued, so that the
// loads do not queue behind the copies
template <int NW>
struct QPrefetch {
  static constexpr int kN = (8 * 128 + NW * 32 - 1) / (NW * 32);
  uint16_t v[kN];
};
template <int NW>
__device__ __forceinline__ void q_prefetch(const DecodeArgs& a, int b, int h, int G,
                                           QPrefetch<NW>& pre) {
#pragma unroll
  for (int k = 0; k < QPrefetch<NW>::kN; ++k) {
    const int i = threadIdx.x + k * NW * 32, c = i >> 7, d = i & 127;
    pre.v[k] = (i < 8 * 128 && c < G) ? a.q[((int64_t)b * a.Hq + h * G + c) * 128 + d] : (uint16_t)0;
  }
}

template <int NW = kWarps>
__device__ void load_group_q(const DecodeArgs& a, Shared& sh, int b, int h, int G,
                             const QPrefetch<NW>* pre = nullptr) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // the Walsh-Hadamard bases take their rotated queries q' = H S q (times fl32(1/sqrt
  // 128) for the rotated affine base, whose rows are stored in the orthonormal frame);
  // the dense rotation's q' = M q comes from qrot_dense_kernel
  const bool wht = a.base == SEMKV_BASE_AFFINE_HAD || a.base == SEMKV_BASE_TQ;
  const bool rot = wht || a.base == SEMKV_BASE_TQ_DENSE;
  if (pre) {
#pragma unroll
    for (int k = 0; k < QPrefetch<NW>::kN; ++k) {
      const int i = threadIdx.x + k * NW * 32;
      if (i < 8 * 128) sh.q[i >> 7][i & 127] = pre->v[k];
    }
  } else {
    for (int i = threadIdx.x; i < 8 * 128; i += NW * 32) {
      const int c = i >> 7, d = i & 127;
      const int64_t at = ((int64_t)b * a.Hq + h * G + c) * 128 + d;
      sh.q[c][d] = c < G ? a.q[at] : (uint16_t)0;
      if (a.base == SEMKV_BASE_TQ_DENSE) sh.qr[c][d] = c < G ? a.qrot[at] : 0.0f;
    }
  }
  __syncthreads();
  // warp w < 8 takes head slot w (a CTA of more warps leaves the rest idle here)
  if (warp < 8) {
  if (wht) {
    // warp w rotates head w: lane l holds dims 4l..4l+3; butterfly stages 1, 2 inside
    // the lane, then 4..64 across lanes, each (a + b, a - b) rounded to nearest
    const int8_t* sg = a.signs + ((int64_t)a.layer * a.H + h) * 128;
    float w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      w[j] = warp < G ? f16_to_f32(sh.q[warp][4 * lane + j]) * (float)sg[4 * lane + j] : 0.0f;
    const float t0 = w[0] + w[1], t1 = w[0] - w[1], t2 = w[2] + w[3], t3 = w[2] - w[3];
    w[0] = t0 + t2;
    w[2] = t0 - t2;
    w[1] = t1 + t3;
    w[3] = t1 - t3;
#pragma unroll
    for (int k = 0; k < 5; ++k) {
      const bool upper = (lane >> k) & 1;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float other = __shfl_xor_sync(0xffffffffu, w[j], 1 << k);
        w[j] = upper ? other - w[j] : w[j] + other;
      }
    }
    const float rs = a.base == SEMKV_BASE_AFFINE_HAD ? kInvSqrtD : 1.0f;
#pragma unroll
    for (int j = 0; j < 4; ++j) sh.qr[warp][4 * lane + j] = w[j] * rs;
    __syncwarp();
  }
  // per head: sum of q (the zero-point weight) and max |q| (the coefficient scale), of
  // the rotated queries for the rotated bases
  float s = 0.0f, mx = 0.0f;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float x = rot ? sh.qr[warp][4 * lane + j] : f16_to_f32(sh.q[warp][4 * lane + j]);
    s += x;
    mx = fmaxf(mx, fabsf(x));
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, off);
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  }
  if (lane == 0) {
    sh.sumq[warp] = s;
    sh.qmax[warp] = mx;
  }
  }
  __syncthreads();
}

// An affine warp's state into the merge area: (e, l, zs) per head and its O^T rows.
// O columns are heads 2t, 2t+1 (for G <= 4, columns 4..7 hold the lo parts of heads
// 0..3; they are written as rows 4..7 and folded in by merge_warps); rows 16m + g (+8)
// are V rows u = 2m (+1) of lane group g, i.e. output dims v_dim(g, u).
__device__ void affine_rows(WarpState& st, int L, int G, MergeArea& mg, float* merge_o) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  // reduce l and zs over the lanes that share a softmax head
#pragma unroll
  for (int off = 1; off <= 16; off <<= 1) {
    if (off == 4 || off == 8 || (off == 16 && G > 4)) continue;
    st.l += __shfl_xor_sync(0xffffffffu, st.l, off);
    st.zs += __shfl_xor_sync(0xffffffffu, st.zs, off);
  }
  __syncthreads();  // every warp is done with the ring: reuse it as the merge area
  if (t == 0 && g < G) {
    mg.m[warp * 8 + g] = st.e;
    mg.l[warp * 8 + g] = st.l;
    mg.z[warp * 8 + g] = st.zs;
  }
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const int qh = 2 * t + c;
    if (qh < G || (G <= 4 && qh >= 4 && qh - 4 < G)) {
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
          merge_o[mo_at(warp * 8 + qh, dim)] = st.O[m][2 * r + c];
        }
      }
    }
  }
}

// Merge the warps' rows into one partial (m, l, o) per head and write it.  kind 0:
// affine pool rows (sum p' c; plus sum p z; lo rows folded for G <= 4); 1: TQ rows
// from the CUDA-core path (rotated back); 2: staged rows (plain sums); 3: TQ rows from
// the tensor-core path (as kind 0, then rotated back).
template <int NW = kWarps>
__device__ void merge_warps(const DecodeArgs& a, int kind, int h, int G, MergeArea& mg,
                            float* merge_o, float* part) {
  constexpr int nw = NW;  // warps of this CTA
  __syncthreads();
  if (threadIdx.x < 8) {
    const int qh = threadIdx.x;
    float M = -INFINITY;
    if (qh < G)
      for (int w = 0; w < nw; ++w) M = fmaxf(M, mg.m[w * 8 + qh]);
    float lsum = 0.0f, zsum = 0.0f;
    for (int w = 0; w < nw; ++w) {
      const float mw = qh < G ? mg.m[w * 8 + qh] : -INFINITY;
      const float sc = (M == -INFINITY || mw == -INFINITY) ? 0.0f : exp2f(mw - M);
      mg.scale[w * 8 + qh] = sc;
      if (sc != 0.0f) {
        lsum += sc * mg.l[w * 8 + qh];
        zsum += sc * mg.z[w * 8 + qh];
      }
    }
    if (qh < G) {
      part[qh] = M;
      part[8 + qh] = lsum;
    }
    mg.cta_z[qh] = zsum;
  }
  __syncthreads();
  // (dense-rotation partials stay in the rotated domain: the combine turns their sum
  // back once per head)
  const bool rotated = (kind == 1 || kind == 3) && a.base != SEMKV_BASE_TQ_DENSE;
  float* merged = merge_o + nw * 8 * kMoStride;  // [8][128], after the warp rows
  for (int i = threadIdx.x; i < G * 128; i += NW * 32) {
    const int qh = i >> 7, d = i & 127;
    float o = 0.0f;
    for (int w = 0; w < nw; ++w) {
      const float sc = mg.scale[w * 8 + qh];
      if (sc != 0.0f) {
        float v = merge_o[mo_at(w * 8 + qh, d)];
        if ((kind == 0 || kind == 3) && G <= 4) v += merge_o[mo_at(w * 8 + qh + 4, d)];
        o += sc * v;
      }
    }
    o = (kind == 0 || kind == 3) ? o + mg.cta_z[qh] : o;
    if (rotated) merged[qh * 128 + d] = o;
    else part[16 + qh * 128 + d] = o;   // nothing to turn back: straight to the partial
  }
  if (!rotated) {
    __syncthreads();  // the merge area (the ring) is free again
    return;
  }
  __syncthreads();
  if (rotated) {
    // back from the rotated domain: o = S H o' (unnormalised transform, stages 1..64)
    for (int hs = 1; hs < 128; hs <<= 1) {
      for (int i = threadIdx.x; i < G * 64; i += NW * 32) {
        const int qh = i >> 6, j = i & 63;
        const int lo = (j / hs) * 2 * hs + (j % hs);
        float* r = merged + qh * 128;
        const float x = r[lo], y = r[lo + hs];
        r[lo] = x + y;
        r[lo + hs] = x - y;
      }
      __syncthreads();
    }
  }
  const int8_t* sg = rotated ? a.signs + ((int64_t)a.layer * a.H + h) * 128 : nullptr;
  // the rotated affine base stores rows in the orthonormal frame: x = S H u / sqrt(128)
  const float rs = a.base == SEMKV_BASE_AFFINE_HAD ? kInvSqrtD : 1.0f;
  for (int i = threadIdx.x; i < G * 128; i += NW * 32) {
    const int qh = i >> 7, d = i & 127;
    const float o = merged[qh * 128 + d];
    part[16 + qh * 128 + d] = rotated ? o * ((float)sg[d] * rs) : o;
  }
  __syncthreads();  // the merge area (the ring) is free again
}

// The first copies of a segment, as run_pool would start them: issued before the
// queries are loaded and the coefficient fragments built, so those overlap the copies.
// The ring must be free (no merge in progress).
__device__ void ring_fill(uint8_t* ring, uint64_t* bars, const uint8_t* pool_bh,
                          uint32_t tile_bytes, int t_begin, int t_end, int ring_it) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nmine = t_end - t_begin <= warp ? 0 : (t_end - t_begin - warp + kWarps - 1) / kWarps;
  uint8_t* my_ring = ring + warp * kStages * kStageBytes;
  uint64_t* my_bar = bars + warp * kStages;
  if (lane == 0) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    for (int i = 0; i < kStages && i < nmine; ++i) {
      const int tile = t_begin + warp + i * kWarps;
      const int sl = (ring_it + i) % kStages;
      mbar_expect_tx(&my_bar[sl], tile_bytes);
      bulk_g2s(my_ring + sl * kStageBytes, pool_bh + (int64_t)tile * tile_bytes, tile_bytes,
               &my_bar[sl]);
    }
  }
  __syncwarp();
}

// The first copies of a fast-path segment (chunks of kChunk tiles), as run_pool_fast
// would start them, issued before the queries are loaded and the coefficient fragments
// built.  The ring must be free (no merge in progress).
template <int NW>
__device__ void ring_fill_fast(uint8_t* ring, uint64_t* bars, const uint8_t* pool_bh,
                               uint32_t tile_bytes, int t_begin, int t_end, int ring_it) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nchunks = (t_end - t_begin + kChunk - 1) / kChunk;
  const int nmine = nchunks <= warp ? 0 : (nchunks - warp + NW - 1) / NW;
  uint8_t* my_ring = ring + warp * kFastStages * kFastStageBytes;
  uint64_t* my_bar = bars + warp * kStages;
  if (lane == 0) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    for (int i = 0; i < kFastStages && i < nmine; ++i) {
      const int first = t_begin + (warp + i * NW) * kChunk;
      const uint32_t bytes = (uint32_t)min(kChunk, t_end - first) * tile_bytes;
      const int sl = (ring_it + i) % kFastStages;
      mbar_expect_tx(&my_bar[sl], bytes);
      bulk_g2s(my_ring + sl * kFastStageBytes, pool_bh + (int64_t)first * tile_bytes, bytes,
               &my_bar[sl]);
    }
  }
  __syncwarp();
}

template <int L>
__device__ void run_pool_any_g(const DecodeArgs& a, const Shared& sh, uint8_t* ring, uint4* aq_all,
                               uint64_t* bars, const uint8_t* pool_bh, int64_t count, int t0,
                               int t1, int G, WarpState& st, int& ring_it) {
  if (G <= 4)
    run_pool<L, true>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it, 0, true);
  else
    run_pool<L, false>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it, 0, true);
}

// Affine pools, balanced plan: CTA c takes the weighted range [c per, (c+1) per) of the
// concatenated [hi | lo] tile sequence of every (b, h) (a tile belongs to the CTA whose
// range holds its start), one partial per (pair, pool) segment it touches.  One wave of
// equal CTAs: no quantisation into waves and no per-split start-up beyond that.
__global__ void __launch_bounds__(kThreads, kCtasAffine) decode_affine_kernel(DecodeArgs a) {
  extern __shared__ __align__(128) uint8_t dyn[];
  __shared__ Shared sh;
  __shared__ MergeArea mg;
  uint8_t* ring = dyn;
  uint4* aq_all = reinterpret_cast<uint4*>(dyn + kRingBytes);
  float* merge_o = reinterpret_cast<float*>(dyn);  // [kWarps][8][128] rows, then [8][128]
  const DecodePlan& P = a.plan;
  const int G = a.Hq / a.H;
  const int64_t pairs = (int64_t)a.B * a.H;
  const int64_t total = pairs * P.W;
  const int64_t start = (int64_t)blockIdx.x * P.per;
  const int64_t end = min(start + P.per, total);

  if (threadIdx.x < kWarps * kStages) mbar_init(&sh.bar[0][0] + threadIdx.x);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncthreads();
  pdl_wait();  // the records, queries and stage partial come from earlier work
  pdl_trigger();
  int ring_it = 0;  // tiles this warp has taken through its ring (barrier phases)
  int64_t loaded = -1;
  for (int64_t bh = start / P.W; bh < pairs && bh * P.W < end; ++bh) {
    const int b = (int)(bh / a.H), h = (int)(bh % a.H);
    for (int src = 0; src < 2; ++src) {
      const int tiles = src ? P.tiles_lo : P.tiles_hi;
      const int w = src ? P.w_lo : P.w_hi;
      const int64_t S = bh * P.W + (src ? (int64_t)P.w_hi * P.tiles_hi : 0);
      const int64_t E = S + (int64_t)w * tiles;
      if (E <= S || E <= start || S >= end) continue;
      const int64_t x0 = max(start, S) - S, x1 = min(end, E) - S;
      const int t0 = (int)((x0 + w - 1) / w);
      const int t1 = (int)min((int64_t)tiles, (x1 + w - 1) / w);
      int n_hi, n_lo;
      pair_slots(P, bh, n_hi, n_lo);
      const int slot = (int)((int64_t)blockIdx.x - S / P.per) + (src ? n_hi : 0);
      const int L = src ? a.L_lo : a.L_hi;
      const int64_t cap = src ? a.lo_cap : a.hi_cap;
      const int64_t count = src ? a.lo_count : a.hi_count;
      const uint8_t* pool = src ? a.lo_pool : a.hi_pool;
      const int rec = record_bytes_rt(SEMKV_BASE_AFFINE, L);
      const uint8_t* pool_bh = pool + (((int64_t)b * a.NL + a.layer) * a.H + h) * cap * rec;
      uint64_t* bars = &sh.bar[0][0];
      ring_fill(ring, bars, pool_bh, (uint32_t)(kTile * rec), t0, t1, ring_it);
      if (bh != loaded) {
        load_group_q(a, sh, b, h, G);
        loaded = bh;
      }
      WarpState st;
      state_init(st);
      switch (L) {
        case 2: run_pool_any_g<2>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        case 3: run_pool_any_g<3>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        case 4: run_pool_any_g<4>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        case 5: run_pool_any_g<5>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        case 6: run_pool_any_g<6>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        case 7: run_pool_any_g<7>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        case 8: run_pool_any_g<8>(a, sh, ring, aq_all, bars, pool_bh, count, t0, t1, G, st, ring_it); break;
        default: break;
      }
      affine_rows(st, L, G, mg, merge_o);
      merge_warps(a, a.base == SEMKV_BASE_AFFINE_HAD ? 3 : 0, h, G, mg, merge_o,
                  a.partials + (bh * P.stride + slot) * kPartialFloats);
    }
  }
}

// A fast-path warp's state into the merge area, in the layout merge_warps reads: per
// head (e, l, zs), and O rows for columns 0..7 (columns 4..7 are the lo parts of
// heads 0..3, folded in by merge_warps); rows 16m + g (+8) are V rows u = 2m (+1) of
// lane group g, i.e. output dims v_dim(g, u).
template <int L>
__device__ void fast_rows(FastState& st, int G, MergeArea& mg, float* merge_o) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  // l and zs of head t: both tokens' sums of the lanes 4g + t for every g
  st.l += st.l2;
  st.zs += st.zs2;
#pragma unroll
  for (int off = 4; off <= 16; off <<= 1) {
    st.l += __shfl_xor_sync(0xffffffffu, st.l, off);
    st.zs += __shfl_xor_sync(0xffffffffu, st.zs, off);
  }
  __syncthreads();  // every warp is done with the ring: reuse it as the merge area
  if (g == 0 && t < G) {
    mg.m[warp * 8 + t] = st.e;
    mg.l[warp * 8 + t] = st.l;
    mg.z[warp * 8 + t] = st.zs;
  }
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const int col = 2 * t + c;
    if ((col & 3) < G) {
#pragma unroll
      for (int m = 0; m < 8; ++m)
#pragma unroll
        for (int r = 0; r < 2; ++r)
          merge_o[mo_at(warp * 8 + col, v_dim<L>(g, 2 * m + r))] = st.O[m][2 * r + c];
    }
  }
}


template <int L, int NW>
__device__ __forceinline__ void run_fast_l(const DecodeArgs& a, const Shared& sh, uint8_t* ring,
                                           uint2* qbs, uint64_t* bars, const uint8_t* pool_bh,
                                           int64_t count, int t0, int t1, int G, FastState& st,
                                           int& ring_it, MergeArea& mg, float* merge_o) {
  run_pool_fast<L, NW>(a, sh, ring, qbs, bars, pool_bh, count, t0, t1, G, st, ring_it);
  fast_rows<L>(st, G, mg, merge_o);
}

// The balanced plan of decode_affine_kernel, run by the fast path: CTA c takes the
// weighted range [c per, (c+1) per) of the concatenated [hi | lo] tile sequence of every
// (b, h), one partial per (pair, pool) segment it touches.
template <int NW>
__global__ void __launch_bounds__(NW * 32, NW == kWarps ? kCtasFast : 1)
    decode_affine_fast_kernel(DecodeArgs a) {
  extern __shared__ __align__(128) uint8_t dyn[];
  __shared__ Shared sh;
  __shared__ MergeArea mg;
  uint8_t* ring = dyn;
  uint2* qbs = reinterpret_cast<uint2*>(dyn + fast_ring_bytes<NW>());  // [8 steps][32 lanes]
  float* merge_o = reinterpret_cast<float*>(dyn);  // [NW][8][128] rows, then [8][128]
  const DecodePlan& P = a.plan;
  const int G = a.Hq / a.H;
  const int64_t pairs = (int64_t)a.B * a.H;
  const int64_t total = pairs * P.W;
  const int64_t start = (int64_t)blockIdx.x * P.per;
  const int64_t end = min(start + P.per, total);

  if (threadIdx.x < NW * kStages) mbar_init(&sh.bar[0][0] + threadIdx.x);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncthreads();
  pdl_wait();  // the records, queries and stage partial come from earlier work
  pdl_trigger();
  int ring_it = 0;  // tiles this warp has taken through its ring (barrier phases)
  int64_t loaded = -1;
  for (int64_t bh = start / P.W; bh < pairs && bh * P.W < end; ++bh) {
    const int b = (int)(bh / a.H), h = (int)(bh % a.H);
    for (int src = 0; src < 2; ++src) {
      const int tiles = src ? P.tiles_lo : P.tiles_hi;
      const int w = src ? P.w_lo : P.w_hi;
      const int64_t S = bh * P.W + (src ? (int64_t)P.w_hi * P.tiles_hi : 0);
      const int64_t E = S + (int64_t)w * tiles;
      if (E <= S || E <= start || S >= end) continue;
      const int64_t x0 = max(start, S) - S, x1 = min(end, E) - S;
      const int t0 = (int)((x0 + w - 1) / w);
      const int t1 = (int)min((int64_t)tiles, (x1 + w - 1) / w);
      int n_hi, n_lo;
      pair_slots(P, bh, n_hi, n_lo);
      const int slot = (int)((int64_t)blockIdx.x - S / P.per) + (src ? n_hi : 0);
      const int L = src ? a.L_lo : a.L_hi;
      const int64_t cap = src ? a.lo_cap : a.hi_cap;
      const int64_t count = src ? a.lo_count : a.hi_count;
      const uint8_t* pool = src ? a.lo_pool : a.hi_pool;
      const int rec = record_bytes_rt(SEMKV_BASE_AFFINE, L);
      const uint8_t* pool_bh = pool + (((int64_t)b * a.NL + a.layer) * a.H + h) * cap * rec;
      uint64_t* bars = &sh.bar[0][0];
      // the queries' loads first, then the segment's first copies, then the queries
      // into shared memory
      const bool new_q = bh != loaded;
      QPrefetch<NW> pre;
      if (new_q) q_prefetch<NW>(a, b, h, G, pre);
      ring_fill_fast<NW>(ring, bars, pool_bh, (uint32_t)(kTile * rec), t0, t1, ring_it);
      if (new_q) {
        load_group_q<NW>(a, sh, b, h, G, &pre);
        loaded = bh;
      }
      FastState st;
      fast_init(st);
      if (L == 5)
        run_fast_l<5, NW>(a, sh, ring, qbs, bars, pool_bh, count, t0, t1, G, st, ring_it, mg,
                          merge_o);
      else
        run_fast_l<6, NW>(a, sh, ring, qbs, bars, pool_bh, count, t0, t1, G, st, ring_it, mg,
                          merge_o);
      merge_warps<NW>(a, a.base == SEMKV_BASE_AFFINE_HAD ? 3 : 0, h, G, mg, merge_o,
                  a.partials + (bh * P.stride + slot) * kPartialFloats);
    }
  }
}

// TQ pools (KIND 1, one CTA per split) and the fp16 stage (KIND 2, one CTA per pair).
template <int KIND>
__global__ void __launch_bounds__(kThreads, kCtasOther) decode_kernel(DecodeArgs a) {
  extern __shared__ __align__(128) uint8_t dyn[];
  __shared__ Shared sh;
  __shared__ MergeArea mg;
  float* merge_o = reinterpret_cast<float*>(dyn);  // [kWarps][8][128] rows, then [8][128]
  const DecodePlan& P = a.plan;
  const int b = blockIdx.z, h = blockIdx.y;
  const int64_t bh = (int64_t)b * a.H + h;
  const int G = a.Hq / a.H;
  int split = blockIdx.x;
  if (KIND == 1) {
    pdl_wait();  // the records and queries (and the dense rotation's q') come from earlier work
    pdl_trigger();
  }
  if (KIND == 2 && !a.stage_overlaps_pools) pdl_wait();
  if (KIND == 2) {
    if (P.balanced) {
      int n_hi, n_lo;
      pair_slots(P, bh, n_hi, n_lo);
      split = n_hi + n_lo;
    } else {
      split = P.splits_hi + P.splits_lo;
    }
  }
  load_group_q(a, sh, b, h, G);
  __shared__ int tq_path;  // TQ: 1 when this pool's codebook takes the tensor-core path
  if (KIND == 1) {
    if (threadIdx.x < 16) {
      const int which = threadIdx.x >> 3, k = threadIdx.x & 7;
      const int L = which == 0 ? a.L_hi : a.L_lo;
      sh.cb[which][k] = k < L ? (which == 0 ? a.cb_hi : a.cb_lo)[k] : 0.0f;
    }
  }
  __syncthreads();
  if (KIND == 1) {
    // rotated queries: sums and maxima for the tensor-core path
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float s = 0.0f, mx = 0.0f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float x = sh.qr[warp][4 * lane + j];
      s += x;
      mx = fmaxf(mx, fabsf(x));
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      s += __shfl_xor_sync(0xffffffffu, s, off);
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    }
    if (lane == 0) {
      sh.sumq[warp] = s;
      sh.qmax[warp] = mx;
    }
    if (threadIdx.x == 0) {
      // centroids as cz + cs c (two levels; three when equally spaced), or for four
      // exactly symmetric levels alpha phi + beta phi^3, phi = 2c - 3
      const int src0 = split < P.splits_hi ? 0 : 1;
      const int L = src0 == 0 ? a.L_hi : a.L_lo;
      const float* cb = sh.cb[src0];
      int path = 0;
      float cs = 0.0f, cz = 0.0f, c3 = 0.0f;
      if (L == 2 || (L == 3 && cb[1] - cb[0] == cb[2] - cb[1])) {
        path = 1;
        cs = cb[1] - cb[0];
        cz = cb[0];
      } else if (L == 4 && cb[0] == -cb[3] && cb[1] == -cb[2]) {
        path = 2;
        const float beta = (cb[3] - 3.0f * cb[2]) / 24.0f;
        const float alpha = cb[2] - beta;
        cs = 2.0f * alpha;
        cz = -3.0f * alpha;
        c3 = beta;
      }
      sh.cdec[src0][0] = cs;
      sh.cdec[src0][1] = cz;
      sh.cdec[src0][2] = c3;
      tq_path = path;
    }
  }
  __syncthreads();
  int kind = KIND;
  if constexpr (KIND == 2) {
    run_stage(a, sh, b, h, G, mg.m, mg.l, mg.z, merge_o);
  } else {
    const int src = split < P.splits_hi ? 0 : 1;
    const int s_idx = src == 0 ? split : split - P.splits_hi;
    const int nsrc = src == 0 ? P.splits_hi : P.splits_lo;
    const int ntiles = src == 0 ? P.tiles_hi : P.tiles_lo;
    const int per = (ntiles + nsrc - 1) / nsrc;
    const int t_begin = min(ntiles, s_idx * per), t_end = min(ntiles, t_begin + per);
    const int L = src == 0 ? a.L_hi : a.L_lo;
    const int64_t cap = src == 0 ? a.hi_cap : a.lo_cap;
    const int64_t count = src == 0 ? a.hi_count : a.lo_count;
    const uint8_t* pool = src == 0 ? a.hi_pool : a.lo_pool;
    const int rec = record_bytes_rt(SEMKV_BASE_TQ, L);
    const uint8_t* pool_bh = pool + (((int64_t)b * a.NL + a.layer) * a.H + h) * cap * rec;
    if (tq_path) {
      uint8_t* ring = dyn;
      uint4* aq_all = reinterpret_cast<uint4*>(dyn + kRingBytes);
      uint64_t* bars = &sh.bar[0][0];
      if (threadIdx.x < kWarps * kStages) mbar_init(bars + threadIdx.x);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      WarpState st;
      state_init(st);
      int ring_it = 0;
      if (L == 2) {
        if (G <= 4) run_pool<2, true, 1>(a, sh, ring, aq_all, bars, pool_bh, count, t_begin, t_end, G, st, ring_it, src);
        else run_pool<2, false, 1>(a, sh, ring, aq_all, bars, pool_bh, count, t_begin, t_end, G, st, ring_it, src);
      } else if (L == 3) {
        if (G <= 4) run_pool<3, true, 1>(a, sh, ring, aq_all, bars, pool_bh, count, t_begin, t_end, G, st, ring_it, src);
        else run_pool<3, false, 1>(a, sh, ring, aq_all, bars, pool_bh, count, t_begin, t_end, G, st, ring_it, src);
      } else {
        if (G <= 4) run_pool<4, true, 2>(a, sh, ring, aq_all, bars, pool_bh, count, t_begin, t_end, G, st, ring_it, src);
        else run_pool<4, false, 2>(a, sh, ring, aq_all, bars, pool_bh, count, t_begin, t_end, G, st, ring_it, src);
      }
      affine_rows(st, L, G, mg, merge_o);
      kind = 3;
    } else {
      switch (L) {
#define SEMKV_TQ_CASE(LV) \
        case LV: run_pool_tq<LV>(a, sh, src, pool_bh, count, t_begin, t_end, G, mg.m, mg.l, mg.z, merge_o); break;
        SEMKV_TQ_CASE(2) SEMKV_TQ_CASE(3) SEMKV_TQ_CASE(4) SEMKV_TQ_CASE(5)
        SEMKV_TQ_CASE(6) SEMKV_TQ_CASE(7) SEMKV_TQ_CASE(8)
#undef SEMKV_TQ_CASE
        default: break;
      }
    }
  }
  merge_warps(a, kind, h, G, mg, merge_o, a.partials + (bh * P.stride + split) * kPartialFloats);
  // a stage kernel that ran alongside the pool kernel completes only after it: the
  // combine, which waits for this kernel, then sees every pool partial too
  if (KIND == 2) pdl_wait();
}

// merge the partials of each (b, qh): one warp per head, 4 dims per lane.  The lanes
// first take the partials' maxima and weights in parallel (weights kept in shared
// memory), then sum the rows with independent loads.
// o = M^T o' for one head (dense rotation): lane l holds dims 4l..4l+3 of o' on entry
// and of o on return; buf is the warp's 128-float scratch, ms the pair's M in shared memory
__device__ __forceinline__ void dense_back(const uint16_t* ms, float* buf, float (&o)[4],
                                           int lane) {
#pragma unroll
  for (int e = 0; e < 4; ++e) buf[4 * lane + e] = o[e];
  __syncwarp();
  const uint16_t* m = ms + 4 * lane;
  float u[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
  for (int j = 0; j < 128; ++j) {
    const uint2 mm = *reinterpret_cast<const uint2*>(m + j * 128);
    const float x = buf[j];
    u[0] = fmaf(f16_to_f32((uint16_t)(mm.x & 0xFFFF)), x, u[0]);
    u[1] = fmaf(f16_to_f32((uint16_t)(mm.x >> 16)), x, u[1]);
    u[2] = fmaf(f16_to_f32((uint16_t)(mm.y & 0xFFFF)), x, u[2]);
    u[3] = fmaf(f16_to_f32((uint16_t)(mm.y >> 16)), x, u[3]);
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) o[e] = u[e];
  __syncwarp();
}

// DENSE: one block of G warps per (sequence, KV head), the pair's rotation staged in
// shared memory for the final M^T.
template <bool DENSE>
__global__ void combine_kernel(DecodeArgs a) {
  constexpr int kHeadsPerCta = 8;
  __shared__ float wsm[kHeadsPerCta][kMaxPartialsPerPair];
  __shared__ float orot[DENSE ? kHeadsPerCta : 1][128];
  __shared__ __align__(16) uint16_t ms[DENSE ? 128 * 128 : 8];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int G = a.Hq / a.H;
  const int gw = DENSE ? (int)blockIdx.x * G + wib : (int)blockIdx.x * kHeadsPerCta + wib;
  if constexpr (DENSE) {
    const int hh = (int)blockIdx.x % a.H;
    const uint4* src = reinterpret_cast<const uint4*>(a.rot + ((int64_t)a.layer * a.H + hh) * 128 * 128);
    for (int x = threadIdx.x; x < 128 * 16; x += blockDim.x) reinterpret_cast<uint4*>(ms)[x] = src[x];
    __syncthreads();
  }
  // launched as a programmatic dependent of the pool kernels: the rotation above is
  // staged while they finish; their partials are read only after this wait
  asm volatile("griddepcontrol.wait;" ::: "memory");
  pdl_trigger();
  if (gw >= a.B * a.Hq) return;
  const int b = gw / a.Hq, qh = gw % a.Hq;
  const int h = qh / G, c = qh % G;
  const int64_t bh = (int64_t)b * a.H + h;
  const int S = pair_partials(a.plan, bh);
  const float* base = a.partials + bh * a.plan.stride * kPartialFloats;
  float M = -INFINITY;
  for (int s = lane; s < S; s += 32) M = fmaxf(M, base[s * kPartialFloats + c]);
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  float lsum = 0.0f;
  for (int s = lane; s < S; s += 32) {
    const float ms = base[s * kPartialFloats + c];
    const float sc = (M == -INFINITY || ms == -INFINITY) ? 0.0f : exp2f(ms - M);
    wsm[wib][s] = sc;
    lsum += sc * base[s * kPartialFloats + 8 + c];
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, off);
  __syncwarp();
  // dense rotation: the pool partials (all but the staged tail's, which comes last) are
  // in the rotated domain; their weighted sum is turned back with M^T before the tail's
  // partial is added
  const int S_rot = DENSE ? S - a.plan.splits_st : -1;
  float o[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
  for (int s = 0; s < S; ++s) {
    if (DENSE && s == S_rot) dense_back(ms, orot[wib], o, lane);
    const float sc = wsm[wib][s];
    if (sc == 0.0f) continue;
    const float4 v = *reinterpret_cast<const float4*>(base + s * kPartialFloats + 16 + c * 128 + 4 * lane);
    o[0] += sc * v.x;
    o[1] += sc * v.y;
    o[2] += sc * v.z;
    o[3] += sc * v.w;
  }
  if (DENSE && S_rot == S) dense_back(ms, orot[wib], o, lane);  // no staged tail
  const float inv = 1.0f / lsum;
  float4 r = make_float4(o[0] * inv, o[1] * inv, o[2] * inv, o[3] * inv);
  *reinterpret_cast<float4*>(a.out + ((int64_t)b * a.Hq + qh) * 128 + 4 * lane) = r;
}

// Merge the partials of one (b, qh) with a CTA of 8 warps: every thread takes partials
// for the maximum and the weights, then warp w sums the rows of partials w, w + 8, ...
// (lane = 4 dims) and the 8 row sums are added in warp order.  For the small batches,
// whose (b, h) pairs are spread over dozens of CTAs, this keeps the combine short.
__global__ void __launch_bounds__(256) combine_wide_kernel(DecodeArgs a) {
  __shared__ float red[8][128];
  __shared__ float red_m[8], red_l[8];
  // launched as a programmatic dependent of the pool kernels: wait for their partials
  asm volatile("griddepcontrol.wait;" ::: "memory");
  pdl_trigger();
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int gw = blockIdx.x;
  const int b = gw / a.Hq, qh = gw % a.Hq;
  const int G = a.Hq / a.H, h = qh / G, c = qh % G;
  const int64_t bh = (int64_t)b * a.H + h;
  const int S = pair_partials(a.plan, bh);
  const float* base = a.partials + bh * a.plan.stride * kPartialFloats;
  // one pass: warp w merges partials w, w + 8, ... (each lane dims 4 lane .. 4 lane + 3)
  // against its own maximum, so every load is issued before any result is needed;
  // then the 8 warps' sums are merged against the overall maximum
  constexpr int kPer = (kMaxPartialsPerPair + 7) / 8;
  float ms[kPer];
  float Mw = -INFINITY;
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int s = w + 8 * i;
    ms[i] = s < S ? base[s * kPartialFloats + c] : -INFINITY;
    Mw = fmaxf(Mw, ms[i]);
  }
  float lw = 0.0f, o[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int s = w + 8 * i;
    if (s >= S || ms[i] == -INFINITY) continue;
    const float sc = exp2f(ms[i] - Mw);
    const float4 v = *reinterpret_cast<const float4*>(base + s * kPartialFloats + 16 + c * 128 + 4 * lane);
    lw += sc * base[s * kPartialFloats + 8 + c];
    o[0] += sc * v.x;
    o[1] += sc * v.y;
    o[2] += sc * v.z;
    o[3] += sc * v.w;
  }
  if (lane == 0) {
    red_m[w] = Mw;
    red_l[w] = lw;
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) red[w][4 * lane + e] = o[e];
  __syncthreads();
  if (w == 0) {
    float M = red_m[0];
#pragma unroll
    for (int i = 1; i < 8; ++i) M = fmaxf(M, red_m[i]);
    float l = 0.0f, r[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float sc = red_m[i] == -INFINITY ? 0.0f : exp2f(red_m[i] - M);
      l += sc * red_l[i];
#pragma unroll
      for (int e = 0; e < 4; ++e) r[e] += sc * red[i][4 * lane + e];
    }
    const float inv = 1.0f / l;
    *reinterpret_cast<float4*>(a.out + ((int64_t)b * a.Hq + qh) * 128 + 4 * lane) =
        make_float4(r[0] * inv, r[1] * inv, r[2] * inv, r[3] * inv);
  }
}

}  // namespace

// relative cost of a 16-token tile per level count (decode instructions per tile)
static int tile_cost(int L) {
  switch (L) {
    case 3: case 6: return 8;   // five-code groups: five multiplies per symbol
    case 5: return 7;
    case 7: case 8: return 6;
    default: return 5;          // L = 2, 4: one code per symbol
  }
}

// the fixed cost of a segment in a CTA (queries, coefficient fragments, the first
// copies' latency, the merge), in tile weights: about 16 five-level tiles
constexpr int64_t kSegmentCost = 16 * 7;

// Replace the balanced plan p by its aligned form (see make_decode_plan) when that is
// cheaper.  target: resident CTAs; st: 1 with a staged tail.
static bool aligned_plan(DecodePlan& p, int64_t pairs, int64_t target, int st, int max_stride,
                         int64_t min_tiles) {
  const int64_t th = p.tiles_hi, tl = p.tiles_lo;
  const int64_t per_pair = target / pairs;
  const int pools = (th > 0) + (tl > 0);
  if (pools == 0 || per_pair < pools) return false;
  const int64_t Th = th > 0 ? th : 1, Tl = tl > 0 ? tl : 1;
  if (Th * Tl > ((int64_t)1 << 40)) return false;  // weights must stay small integers
  // CTAs per segment: min_tiles or more per CTA (a chunk or more per warp), at most the
  // partial slots allow
  const int64_t max_n = (int64_t)max_stride - st;
  const int64_t cap_hi = th > 0 ? (th / min_tiles > 1 ? th / min_tiles : 1) : 0;
  const int64_t cap_lo = tl > 0 ? (tl / min_tiles > 1 ? tl / min_tiles : 1) : 0;
  int64_t best_h = 0, best_l = 0, best = INT64_MAX;
  for (int64_t nh = th > 0 ? 1 : 0; nh <= (th > 0 ? cap_hi : 0); ++nh) {
    int64_t nl = tl > 0 ? per_pair - nh : 0;
    if (nl > cap_lo) nl = cap_lo;
    if (nh + nl > max_n) nl = max_n - nh;
    if (tl > 0 && nl < 1) continue;
    const int64_t ch = nh ? (th + nh - 1) / nh * p.w_hi : 0;
    const int64_t cl = nl ? (tl + nl - 1) / nl * p.w_lo : 0;
    const int64_t c = ch > cl ? ch : cl;
    if (c < best) {
      best = c;
      best_h = nh;
      best_l = nl;
    }
  }
  if (best == INT64_MAX || best >= p.per + kSegmentCost) return false;
  const int64_t wh = best_h * Tl, wl = best_l * Th;
  if (wh > INT32_MAX || wl > INT32_MAX) return false;
  p.w_hi = (int)wh;
  p.w_lo = (int)wl;
  p.per = Th * Tl;
  p.W = (best_h + best_l) * p.per;
  p.ctas = (int)(pairs * (best_h + best_l));
  return true;
}

DecodePlan make_decode_plan(int base, int L_hi, int L_lo, int B, int H, int Hq, int64_t hi_count,
                            int64_t lo_count, int stage_n, int num_sms, int max_stride) {
  DecodePlan p;
  std::memset(&p, 0, sizeof(p));
  p.tiles_hi = (int)((hi_count + kTile - 1) / kTile);
  p.tiles_lo = (int)((lo_count + kTile - 1) / kTile);
  p.tiles_st = (stage_n + kTile - 1) / kTile;
  const int st = stage_n > 0 ? 1 : 0;
  p.splits_st = st;
  const int64_t pairs = (int64_t)B * H;
  if (max_stride > kMaxSplits + 1) max_stride = kMaxSplits + 1;
  if (base == SEMKV_BASE_AFFINE || base == SEMKV_BASE_AFFINE_HAD) {
    // balanced: one wave of equal CTAs over the weighted tiles of every pair
    p.balanced = 1;
    p.fast = (Hq / H <= 4 && (L_hi == 5 || L_hi == 6) && (L_lo == 5 || L_lo == 6)) ? 1 : 0;
    p.w_hi = tile_cost(L_hi);
    p.w_lo = tile_cost(L_lo);
    p.W = (int64_t)p.w_hi * p.tiles_hi + (int64_t)p.w_lo * p.tiles_lo;
    const int64_t total = pairs * p.W;
    if (total == 0) {
      p.per = 1;
      p.ctas = 0;
      p.stride = st;
      return p;
    }
    // A pair's weighted range of length W meets at most ceil(W / per) + 1 CTA ranges,
    // and the hi | lo boundary splits at most one of those pieces in two: the pair
    // writes at most ceil(W / per) + 2 pool partials.  Keep them, plus the stage's,
    // within max_stride: ceil(W / per) <= max_stride - st - 2.
    const int64_t avail = (int64_t)max_stride - st - 2;
    const int64_t w_max = p.w_hi > p.w_lo ? p.w_hi : p.w_lo;
    // equal ranges for `target` CTAs of at least min_tiles tiles' weight each
    auto straddled = [&](int64_t target, int64_t min_tiles) {
      int64_t per = (total + target - 1) / target;
      if (per < w_max * min_tiles) per = w_max * min_tiles;
      const int64_t per_min = (p.W + avail - 1) / avail;
      if (per < per_min) per = per_min;
      p.per = per;
      p.ctas = (int)((total + per - 1) / per);
    };
    if (avail < 1) {
      p.per = 1;
      p.ctas = 0;
      p.stride = max_stride + 1;  // infeasible: the caller reports the workspace as short
      return p;
    }
    // CTAs of 8 warps, two per SM (a copy of one or two tiles per warp and step)
    p.warps = kWarps;
    straddled((int64_t)num_sms * (p.fast ? kCtasFast : kCtasAffine), kWarps * 2);
    // When the CTAs outnumber the pairs' segments (few sequences), ranges of equal
    // weight cut across the hi | lo and pair boundaries, and a CTA whose range holds a
    // boundary sets up, streams and merges two segments.  Aligned alternative: n_hi
    // CTAs per hi segment and n_lo per lo segment, each taking an equal share of its
    // segment's tiles.  It is the same range arithmetic with the weights w_hi' =
    // n_hi T_lo and w_lo' = n_lo T_hi and per' = T_hi T_lo (T = the tile counts, 1 for
    // an empty pool), so that a segment is exactly n_hi (n_lo) ranges long.  Taken when
    // its longest range is shorter than per plus one segment's fixed cost.
    const bool aligned = aligned_plan(p, pairs, (int64_t)num_sms * (p.fast ? kCtasFast : kCtasAffine),
                                      st, max_stride, kWarps * 2);
    // Otherwise the fast kernel runs one CTA of 16 warps per SM (see fast_ring_bytes)
    if (p.fast && !aligned) {
      p.warps = kFastWarps;
      straddled(num_sms, kFastWarps * kChunk);
    }
    int worst = 0;
    for (int64_t bh = 0; bh < pairs; ++bh) {
      int n_hi, n_lo;
      pair_slots(p, bh, n_hi, n_lo);
      if (n_hi + n_lo > worst) worst = n_hi + n_lo;
    }
    p.stride = worst + st;
    p.splits = 0;
    return p;
  }
  // split plan (TQ pools): S CTAs per pair, divided between the pools by tile count
  const int64_t slots = (int64_t)num_sms * kCtasOther;  // resident CTAs
  const int nt = p.tiles_hi + p.tiles_lo;
  const int s_max = max_stride - st < kMaxSplits ? max_stride - st : kMaxSplits;
  int best_s = 1;
  double best_cost = 1e300;
  for (int S = 1; S <= s_max; ++S) {
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
    if (s_max < 2) {
      p.stride = max_stride + 1;  // infeasible
      return p;
    }
    int shi = (int)((double)best_s * p.tiles_hi / nt + 0.5);
    shi = shi < 1 ? 1 : (shi > best_s - 1 ? best_s - 1 : shi);
    p.splits_hi = shi;
    p.splits_lo = best_s - shi;
  } else {
    if (s_max < 1) {
      p.stride = max_stride + 1;
      return p;
    }
    p.splits_hi = p.tiles_hi > 0 ? best_s : 0;
    p.splits_lo = p.tiles_lo > 0 ? best_s : 0;
  }
  p.splits = p.splits_hi + p.splits_lo + p.splits_st;
  p.stride = p.splits;
  return p;
}

size_t decode_workspace_floats(int B, int H, int Hq) {
  return (size_t)B * H * (kMaxSplits + 1) * kPartialFloats + (size_t)B * Hq * 128;
}

cudaError_t launch_decode_attention(const DecodeArgs& a, cudaStream_t stream) {
  static bool attr_set[kAttrDevices] = {};
  {
    const cudaError_t e = once_per_device(attr_set, [] {
      cudaError_t r = cudaFuncSetAttribute(decode_affine_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           kRingBytes + kAqBytes);
      if (r == cudaSuccess)
        r = cudaFuncSetAttribute(decode_affine_fast_kernel<kWarps>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 fast_ring_bytes<kWarps>() + kQbBytes);
      if (r == cudaSuccess)
        r = cudaFuncSetAttribute(decode_affine_fast_kernel<kFastWarps>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 fast_ring_bytes<kFastWarps>() + kQbBytes);
      if (r == cudaSuccess)
        r = cudaFuncSetAttribute(decode_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kRingBytes + kAqBytes);
      if (r == cudaSuccess)
        r = cudaFuncSetAttribute(decode_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kRingBytes);
      return r;
    });
    if (e != cudaSuccess) return e;
  }
  const DecodePlan& P = a.plan;
  if (P.stride < 1 || P.stride > kMaxSplits + 1) return cudaErrorInvalidValue;
  cudaError_t e = cudaSuccess;
  bool pools_launched = false;
  if (a.base == SEMKV_BASE_TQ_DENSE || a.base == SEMKV_BASE_TQ) {
    if (a.base == SEMKV_BASE_TQ_DENSE) {
      qrot_dense_kernel<<<a.B * a.H, 128, 0, stream>>>(a);
      e = cudaGetLastError();
      if (e != cudaSuccess) return e;
    }
    const int pool_splits = P.splits_hi + P.splits_lo;
    if (pool_splits > 0) {
      e = launch_pdl(decode_kernel<1>, dim3(pool_splits, a.H, a.B), dim3(kThreads),
                     kRingBytes + kAqBytes, stream, a);
      if (e != cudaSuccess) return e;
      pools_launched = true;
    }
  } else if (P.ctas > 0) {
    // (the rotated affine base rotates its queries inside the pool and stage kernels)
    if (P.fast)
      e = P.warps == kFastWarps
              ? launch_pdl(decode_affine_fast_kernel<kFastWarps>, dim3(P.ctas),
                           dim3(kFastWarps * 32), fast_ring_bytes<kFastWarps>() + kQbBytes, stream, a)
              : launch_pdl(decode_affine_fast_kernel<kWarps>, dim3(P.ctas), dim3(kWarps * 32),
                           fast_ring_bytes<kWarps>() + kQbBytes, stream, a);
    else
      e = launch_pdl(decode_affine_kernel, dim3(P.ctas), dim3(kThreads), kRingBytes + kAqBytes,
                     stream, a);
    if (e != cudaSuccess) return e;
    pools_launched = true;
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (P.splits_st > 0) {
    // after a pool kernel (which triggers its dependents once it has waited for its own
    // inputs) the stage kernel starts alongside it; otherwise it runs in order
    DecodeArgs as = a;
    as.stage_overlaps_pools = pools_launched ? 1 : 0;
    if (as.stage_overlaps_pools)
      e = launch_pdl(decode_kernel<2>, dim3(1, a.H, a.B), dim3(kThreads), kRingBytes, stream, as);
    else
      decode_kernel<2><<<dim3(1, a.H, a.B), kThreads, kRingBytes, stream>>>(as);
    if (e != cudaSuccess) return e;
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  // the combine starts as a programmatic dependent launch: its launch (and, for the
  // dense rotation, the staging of M) overlaps the tail of the kernels before it
  const int heads = a.B * a.Hq;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.dynamicSmemBytes = 0;
  if (a.base == SEMKV_BASE_TQ_DENSE) {
    cfg.gridDim = dim3((unsigned)(a.B * a.H));
    cfg.blockDim = dim3((unsigned)(32 * (a.Hq / a.H)));
    return cudaLaunchKernelEx(&cfg, combine_kernel<true>, a);
  }
  cfg.gridDim = dim3((unsigned)heads);
  cfg.blockDim = dim3(256);
  return cudaLaunchKernelEx(&cfg, combine_wide_kernel, a);
}

}  // namespace semkv
