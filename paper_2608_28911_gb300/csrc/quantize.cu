// quantize.cu — token-wise mixed-precision quantization and mixed-radix packing
// (Eq. 7; Sec. 4.1 affine base and its Hadamard-rotated form; Sec. 4.9 TurboQuant-MSE
// base with the randomized Hadamard or a dense random rotation), and fake quantization.
//
// Records are built by destination slot: after a slot -> token map (scatter_tok_kernel),
// the affine kernel gives a warp 8 consecutive slots of one pool (lanes own half rows);
// the rotated bases give a 128-thread CTA 64 slots (one thread per row, the whole row
// in registers).  Either way a CTA's level count is uniform and its record writes are
// contiguous.  The dense rotation runs its 128 x 128 product on tcgen05 instead.
//
// Arithmetic (binary32, round to nearest even, no contraction), per row x:
//  affine: s = fp16((max-min)/(L-1)) limited to 65504, z = fp16(min);
//          c = clamp(rint((x - z) * fl(1/s)), 0, L-1)   (all 0 when s == 0)
//  rotated affine: u = fl(1/sqrt 128) * FWHT(x * sign); z = fp16 of min u rounded
//          toward -inf (limited to -65504); s and c as affine on u (all 0 unless s > 0)
//  TQ:     w = FWHT(x * sign) with butterflies h = 1..64; n = fp16(sqrt(sum x^2))
//          with the sum taken as 32 in-order partials of 4 squares then pairwise
//          stages 16, 8, 4, 2, 1; u = w * fl(1/n); c = #{k: u > t_k}
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace semkv {

namespace {

constexpr int kWarpsPerBlock = 8;
constexpr int kMaxRecWords = 27;  // largest record: affine L=7/8, 2*48+8 = 104 B

// ------------------------------------------------- affine pools, by slot -----
// Affine records are built by destination slot: a warp takes units of 4 consecutive
// slots of one pool of one (sequence, layer, KV head), so the level count is uniform
// across the warp and the records it writes are contiguous.  Lane 8i + 4r + q handles
// quarter q (dims 32q..32q+31) of row r (0 = K, 1 = V) of the i-th slot's token: 64
// contiguous bytes in, one quarter bit field out (a quarter per lane keeps the lane's
// state small: 48 registers, 40 warps per SM).  The same arithmetic as the header states, and
// symbols beta = ceil(t 2^W / L^G) (the record format).

constexpr int kAffineSlots = 4;
constexpr int kAffineCtas = 5;  // resident CTAs of 8 warps per SM (48 registers)

// 32 fp16 values of one quarter row (16-byte loads when the source allows)
__device__ __forceinline__ void load_quarter(const uint16_t* src, bool vec16, uint32_t (&h)[16]) {
  if (vec16) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(src) + j);
      h[4 * j] = u.x; h[4 * j + 1] = u.y; h[4 * j + 2] = u.z; h[4 * j + 3] = u.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(src) + j);
      h[2 * j] = u.x; h[2 * j + 1] = u.y;
    }
  }
}

// OR the value v (n bits, n <= 32) in at bit pos of a 3-word field (pos, n compile-time)
__device__ __forceinline__ void put_bits(uint32_t (&w)[3], int pos, int n, uint32_t v) {
  const int wd = pos >> 5, sh = pos & 31;
  w[wd] |= v << sh;
  if (sh + n > 32) w[wd + 1] |= v >> (32 - sh);
}

// The bit field of one quarter from its 32 rounded values: m[j] is the bit pattern of
// 1.5 * 2^23 + c_j, so sums of L-weighted patterns give the radix value t modulo 2^32
// once the weighted 1.5 * 2^23 terms are taken off.
template <int L>
__device__ __forceinline__ void quarter_field(const uint32_t (&m)[32], uint32_t (&w)[3]) {
  using F = Fmt<L>;
  constexpr uint32_t kMagic = 0x4B400000u;
  w[0] = w[1] = w[2] = 0u;
  if constexpr (F::G == 1 && F::LG == (1u << F::W)) {
    // L = 2, 4, 8: ceil(c 2^W / L) = c, each code its own W-bit symbol
#pragma unroll
    for (int sy = 0; sy < 32; ++sy) put_bits(w, sy * F::W, F::W, m[sy] - kMagic);
  } else {
#pragma unroll
    for (int sy = 0; sy < F::NG; ++sy) {
      uint32_t t = 0, wsum = 0;
#pragma unroll
      for (int k = 0; k < F::G; ++k) {
        t = t * (uint32_t)L + m[sy * F::G + k];
        wsum = wsum * (uint32_t)L + 1u;
      }
      t -= wsum * kMagic;
      put_bits(w, sy * F::W, F::W, ((t << F::W) + F::LG - 1u) / F::LG);
    }
    if constexpr (F::R > 0) {
      uint32_t t = 0, wsum = 0;
#pragma unroll
      for (int k = 0; k < F::R; ++k) {
        t = t * (uint32_t)L + m[32 - F::R + k];
        wsum = wsum * (uint32_t)L + 1u;
      }
      t -= wsum * kMagic;
      put_bits(w, F::NG * F::W, F::WT, ((t << F::WT) + F::LR - 1u) / F::LR);
    }
  }
}

// One code of a quarter's field, streamed in order (j = 0..31, compile-time after
// unrolling): m is the magic-number pattern 1.5 * 2^23 + c_j, t the running radix value
// of the open symbol; each completed symbol's beta goes into the field, as quarter_field.
template <int L>
__device__ __forceinline__ void field_push(uint32_t (&w)[3], uint32_t& t, int j, uint32_t m) {
  using F = Fmt<L>;
  constexpr uint32_t kMagic = 0x4B400000u;
  if constexpr (F::G == 1 && F::LG == (1u << F::W)) {
    put_bits(w, j * F::W, F::W, m - kMagic);
  } else {
    if (j < F::NG * F::G) {
      const int k = j % F::G, sy = j / F::G;
      t = (k == 0 ? 0u : t * (uint32_t)L) + m;
      if (k == F::G - 1) {
        uint32_t wsum = 0;
        for (int q = 0; q < F::G; ++q) wsum = wsum * (uint32_t)L + 1u;
        const uint32_t tt = t - wsum * kMagic;
        put_bits(w, sy * F::W, F::W, ((tt << F::W) + F::LG - 1u) / F::LG);
      }
    } else {
      const int k = j - F::NG * F::G;
      t = (k == 0 ? 0u : t * (uint32_t)L) + m;
      if (k == F::R - 1) {
        uint32_t wsum = 0;
        for (int q = 0; q < F::R; ++q) wsum = wsum * (uint32_t)L + 1u;
        const uint32_t tt = t - wsum * kMagic;
        put_bits(w, F::NG * F::W, F::WT, ((tt << F::WT) + F::LR - 1u) / F::LR);
      }
    }
  }
}

template <int L>
__device__ void affine_units(const QuantArgs& a, int b, int l, int h, bool hi, int64_t n_pool,
                             int64_t u_begin, int64_t u_step, bool vec16, uint32_t* img) {
  using F = Fmt<L>;
  constexpr int kRecW = (2 * F::RB + 8) / 4;
  static_assert(F::QB <= 96, "a quarter fits three words");
  const int lane = threadIdx.x & 31;
  const int ti = lane >> 3, row = (lane >> 2) & 1, qd = lane & 3;
  const int64_t cap = hi ? a.hi_cap : a.lo_cap;
  const int64_t base = hi ? a.hi_base : a.lo_base;
  const int64_t bh = ((int64_t)b * a.NL + l) * a.H + h;
  const int32_t* tokmap = (hi ? a.hi_tok : a.lo_tok) + (int64_t)b * cap + base;
  const uint16_t* src = (row ? a.v : a.k) + bh * a.Tsrc * kHeadDim + 32 * qd;
  const int64_t tok_base = a.tok_base;
  uint32_t* recs = reinterpret_cast<uint32_t*>(hi ? a.hi_pool : a.lo_pool) + (bh * cap + base) * kRecW;
  const int64_t units = (n_pool + kAffineSlots - 1) / kAffineSlots;
  for (int64_t u = u_begin; u < units; u += u_step) {
    const int64_t s0 = u * kAffineSlots;
    const int nslots = (int)min((int64_t)kAffineSlots, n_pool - s0);
    const bool active = ti < nslots;
    for (int i = lane; i < kAffineSlots * kRecW; i += 32) img[i] = 0u;
    uint32_t hv[16];
    if (active) {
      load_quarter(src + ((int64_t)tokmap[s0 + ti] - tok_base) * kHeadDim, vec16, hv);
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j) hv[j] = 0u;
    }
    // row minimum and maximum: fp16 pairs (exact), then the row's other quarters
    __half2 mn2 = *reinterpret_cast<const __half2*>(&hv[0]), mx2 = mn2;
#pragma unroll
    for (int j = 1; j < 16; ++j) {
      const __half2 x2 = *reinterpret_cast<const __half2*>(&hv[j]);
      mn2 = __hmin2(mn2, x2);
      mx2 = __hmax2(mx2, x2);
    }
    float mn = fminf(__low2float(mn2), __high2float(mn2));
    float mx = fmaxf(__low2float(mx2), __high2float(mx2));
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, 2));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    // a zero extreme is taken as +0 (min/max may return either signed zero)
    if (mn == 0.0f) mn = 0.0f;
    if (mx == 0.0f) mx = 0.0f;
    const float s32 = __fdiv_rn(__fsub_rn(mx, mn), (float)(L - 1));
    const uint16_t s16 = f16_param(s32), z16 = __half_as_ushort(__float2half_rn(mn));
    const float sc = f16_to_f32(s16), z = f16_to_f32(z16);
    // 1/s, or 0 when s == 0 (then every value rounds to code 0)
    const float inv = sc != 0.0f ? __fdiv_rn(1.0f, sc) : 0.0f;
    __syncwarp();
    // the codes stream into the quarter's field (no array of them: fewer registers)
    uint32_t w[3] = {0u, 0u, 0u}, t = 0u;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float x = f16_to_f32((uint16_t)(hv[j >> 1] >> (16 * (j & 1))));
      // rint((x - z) / s) clamped to L-1 (the difference is >= 0: z is the row
      // minimum); adding 1.5 * 2^23 rounds to nearest even
      const float y = fminf(__fmul_rn(__fsub_rn(x, z), inv), (float)(L - 1));
      field_push<L>(w, t, j, __float_as_uint(__fadd_rn(y, 12582912.0f)));
    }
    if (active) {
      uint32_t* r = img + ti * kRecW;
      const int pos = row * 8 * F::RB + qd * F::QB;  // the quarter's first bit
      const int wd = pos >> 5, sh = pos & 31;
      atomicOr(&r[wd], w[0] << sh);
      if (sh + F::QB > 32) atomicOr(&r[wd + 1], __funnelshift_l(w[0], w[1], sh));
      if (sh + F::QB > 64) atomicOr(&r[wd + 2], __funnelshift_l(w[1], w[2], sh));
      if (sh + F::QB > 96) atomicOr(&r[wd + 3], __funnelshift_l(w[2], 0u, sh));
      if (qd == 0) r[(2 * F::RB) / 4 + row] = (uint32_t)s16 | ((uint32_t)z16 << 16);
    }
    __syncwarp();
    uint32_t* dst = recs + s0 * kRecW;
    for (int i = lane; i < nslots * kRecW; i += 32) dst[i] = img[i];
    __syncwarp();
  }
}

// slot -> token maps of the tokens quantized by this call
__global__ void scatter_tok_kernel(QuantArgs a) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)a.B * a.n) return;
  const int b = (int)(i / a.n), j = (int)(i % a.n);
  const bool hi = a.is_high[(int64_t)b * a.n + j] != 0;
  const int64_t s = (hi ? a.hi_base : a.lo_base) + a.slot[(int64_t)b * a.n + j];
  const int64_t cap = hi ? a.hi_cap : a.lo_cap;
  if (s >= cap) {  // cannot happen after the host's capacity check
    raise_error(a.err, kDevCapacity);
    return;
  }
  (hi ? a.hi_tok : a.lo_tok)[(int64_t)b * cap + s] = (int32_t)(a.tok_base + j);
}

// grid (x, sequence*layer*head, pool): each warp strides over that pool's units
__global__ void __launch_bounds__(kWarpsPerBlock * 32, kAffineCtas)
    quantize_affine_kernel(QuantArgs a, int64_t n_hi, int64_t n_lo) {
  __shared__ __align__(16) uint32_t img_sm[kWarpsPerBlock][kAffineSlots * kMaxRecWords];
  const int wib = threadIdx.x >> 5;
  pdl_wait();  // the slot maps and the rows come from earlier work on the stream
  pdl_trigger();
  const bool hi = blockIdx.z == 0;
  const int64_t n_pool = hi ? n_hi : n_lo;
  const int64_t u_begin = (int64_t)blockIdx.x * kWarpsPerBlock + wib;
  const int64_t u_step = (int64_t)gridDim.x * kWarpsPerBlock;
  const bool vec16 = ((reinterpret_cast<uintptr_t>(a.k) | reinterpret_cast<uintptr_t>(a.v)) & 15u) == 0;
  uint32_t* img = img_sm[wib];
  const int bhs = a.B * a.NL * a.H;
  for (int bhi = blockIdx.y; bhi < bhs; bhi += gridDim.y) {
    const int h = bhi % a.H, l = (bhi / a.H) % a.NL, b = bhi / (a.H * a.NL);
    switch (hi ? a.L_hi : a.L_lo) {
      case 2: affine_units<2>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      case 3: affine_units<3>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      case 4: affine_units<4>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      case 5: affine_units<5>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      case 6: affine_units<6>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      case 7: affine_units<7>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      case 8: affine_units<8>(a, b, l, h, hi, n_pool, u_begin, u_step, vec16, img); break;
      default: break;
    }
  }
}

// ------------------------------ rotated bases by slot, two threads per row -----
// TQ and rotated affine records built by destination slot, as for the affine base: a
// CTA of 256 threads takes 64 consecutive slots of one pool of one (sequence, layer,
// KV head), so the level count is uniform.  Thread tid holds half f = tid & 1 (dims
// 64f .. 64f + 63, quarters 2f and 2f + 1) of row tid >> 1 of the block (K of slot
// tid >> 2 when bit 1 of tid is 0, V when it is 1), in registers as 32 packed pairs
// (x_j, x_{j+32}).  The Walsh-Hadamard butterflies run in the quantizer's stage order
// (the same roundings as any other evaluation of them): stages 1..16 as packed
// operations across pairs, stage 32 inside each pair, stage 64 with the partner lane.
// Then the norm or the min/max (combined across the two halves), the codes, the two
// quarters' bit fields; the threads then assemble the block's record words from the
// rows' bit images and write them in order with 4-byte stores.
constexpr int kRowSlots = 64;
constexpr int kRowStride = 272;  // bytes per staged row: 256 + 16 spreads the banks
constexpr int kRowBitWords = 13;  // words per row's bit image (12 used at most)
constexpr int kRows2Threads = 256;
constexpr int kHalfStride = 144;  // bytes per half-row slot: 128 + 16 (9 x 16 B: the 8 lanes
                                  // of a quarter warp reach distinct banks)
constexpr int kRows2StageBytes = kRows2Threads * kHalfStride;
// resident CTAs per SM (80 registers a thread).  The TQ path at 4 and more levels keeps
// its packed thresholds in registers too and spills a few words at this budget; it still
// ran 6% faster than at 2 CTAs per SM (128 registers, no spills).
constexpr int rows2_ctas(int) { return 3; }
static_assert(kRowBitWords + 1 <= kHalfStride / 4, "bit image and parameters fit a half slot");

// packed binary32 pairs (two independent IEEE operations, rounded to nearest)
__device__ __forceinline__ unsigned long long f2_add(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long f2_sub(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long f2_pack(float lo, float hi) {
  return (unsigned long long)__float_as_uint(lo) | ((unsigned long long)__float_as_uint(hi) << 32);
}
__device__ __forceinline__ float f2_lo(unsigned long long v) { return __uint_as_float((uint32_t)v); }
__device__ __forceinline__ float f2_hi(unsigned long long v) {
  return __uint_as_float((uint32_t)(v >> 32));
}

// OR the 96-bit field v at bit pos (compile-time after unrolling) of a row's words
template <int N>
__device__ __forceinline__ void or_field(uint32_t (&w)[N], int pos, const uint32_t (&v)[3]) {
  const int wd = pos >> 5, sh = pos & 31;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t lo = k < 3 ? v[k] : 0u, prev = k > 0 ? v[k - 1] : 0u;
    const uint32_t part = sh == 0 ? lo : (lo << sh) | (prev >> (32 - sh));
    if (wd + k < N) w[wd + k] |= part;
  }
}

// packed binary32 multiply and fused multiply-add (one rounding each).  The code
// generator may fuse a packed multiply into a packed add or subtract that consumes it,
// .rn notwithstanding (measured), so bit-exact paths use f2_mul only where the product
// is exact (squares of fp16 values) and the scalar __fmul_rn (never fused) elsewhere.
__device__ __forceinline__ unsigned long long f2_mul(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long f2_fma(unsigned long long a, unsigned long long b,
                                                     unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// Butterfly stages 1, 2, 4, 8, 16 and 32 of the row transform over one half of the row,
// held as packed pairs xp[j] = (x_j, x_{j+32}) (half-local indices): stages 1..16 pair
// registers j and j + hs and so run packed, stage 32 works inside each register.  Each
// butterfly is (a + b, a - b), rounded to nearest.
__device__ __forceinline__ void fwht_half(unsigned long long (&xp)[32]) {
#pragma unroll
  for (int hs = 1; hs < 32; hs <<= 1) {
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      if (j & hs) continue;
      const unsigned long long p0 = xp[j], p1 = xp[j + hs];
      xp[j] = f2_add(p0, p1);
      xp[j + hs] = f2_sub(p0, p1);
    }
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float lo = f2_lo(xp[j]), hi = f2_hi(xp[j]);
    xp[j] = f2_pack(__fadd_rn(lo, hi), __fsub_rn(lo, hi));
  }
}

// The bit field of one quarter from its 32 codes c_j = m[j] - kOff (kOff: 1.5 * 2^23 for
// magic-number patterns, 0 for plain codes), as quarter_field.
template <int L, uint32_t kOff>
__device__ __forceinline__ void quarter_field_off(const uint32_t (&m)[32], uint32_t (&w)[3]) {
  using F = Fmt<L>;
  w[0] = w[1] = w[2] = 0u;
  if constexpr (F::G == 1 && F::LG == (1u << F::W)) {
#pragma unroll
    for (int sy = 0; sy < 32; ++sy) put_bits(w, sy * F::W, F::W, m[sy] - kOff);
  } else {
#pragma unroll
    for (int sy = 0; sy < F::NG; ++sy) {
      uint32_t t = 0, wsum = 0;
#pragma unroll
      for (int k = 0; k < F::G; ++k) {
        t = t * (uint32_t)L + m[sy * F::G + k];
        wsum = wsum * (uint32_t)L + 1u;
      }
      t -= wsum * kOff;
      put_bits(w, sy * F::W, F::W, ((t << F::W) + F::LG - 1u) / F::LG);
    }
    if constexpr (F::R > 0) {
      uint32_t t = 0, wsum = 0;
#pragma unroll
      for (int k = 0; k < F::R; ++k) {
        t = t * (uint32_t)L + m[32 - F::R + k];
        wsum = wsum * (uint32_t)L + 1u;
      }
      t -= wsum * kOff;
      put_bits(w, F::NG * F::W, F::WT, ((t << F::WT) + F::LR - 1u) / F::LR);
    }
  }
}

// TQ codes of both quarters of a half, straight into their bit fields.  u2[j] holds the
// pair (u of quarter 0, u of quarter 1) at dim j of the quarters; t2[k] the pair
// (thr_k, thr_k), ascending, with a zero threshold taken as +0.  d = thr_k - u rounds to
// a value below zero exactly when u > thr_k (binary32 subtraction of unequal values is
// never zero, and with +0 thresholds an equal pair gives +0), so bit 31 of d is the
// comparison, and c = sum_k [u > thr_k] is a thermometer code: c = 1 + ... + 1.
//   L = 2, 4, 8: the code's binary digits from those bits (parities and middles of the
//   thermometer), shifted into the field most significant bit first, one funnel shift
//   per bit (code j occupies bits jW .. jW + W - 1 of the field);
//   other L: c as a sum of the bits, radix groups as quarter_field.
template <int L>
__device__ __forceinline__ void tq_fields(const unsigned long long (&u2)[32],
                                          const unsigned long long (&t2)[7],
                                          uint32_t (&w0)[3], uint32_t (&w1)[3]) {
  using F = Fmt<L>;
  w0[0] = w0[1] = w0[2] = 0u;
  w1[0] = w1[1] = w1[2] = 0u;
  if constexpr (F::G == 1 && F::LG == (1u << F::W)) {
    constexpr int W = F::W;
    uint32_t a0 = 0u, a1 = 0u;
#pragma unroll
    for (int j = 31; j >= 0; --j) {
      uint32_t dl[7], dh[7];
#pragma unroll
      for (int k = 0; k < L - 1; ++k) {
        const unsigned long long d = f2_sub(t2[k], u2[j]);
        dl[k] = (uint32_t)d;
        dh[k] = (uint32_t)(d >> 32);
      }
#pragma unroll
      for (int b = W - 1; b >= 0; --b) {
        uint32_t bl, bh;
        if constexpr (L == 2) {
          bl = dl[0]; bh = dh[0];
        } else if constexpr (L == 4) {
          if (b == 1) { bl = dl[1]; bh = dh[1]; }
          else { bl = dl[0] ^ dl[1] ^ dl[2]; bh = dh[0] ^ dh[1] ^ dh[2]; }
        } else {
          if (b == 2) { bl = dl[3]; bh = dh[3]; }
          else if (b == 1) { bl = dl[1] ^ dl[3] ^ dl[5]; bh = dh[1] ^ dh[3] ^ dh[5]; }
          else {
            bl = dl[0] ^ dl[1] ^ dl[2] ^ dl[3] ^ dl[4] ^ dl[5] ^ dl[6];
            bh = dh[0] ^ dh[1] ^ dh[2] ^ dh[3] ^ dh[4] ^ dh[5] ^ dh[6];
          }
        }
        a0 = __funnelshift_l(bl, a0, 1);
        a1 = __funnelshift_l(bh, a1, 1);
        const int pbit = j * W + b;
        if ((pbit & 31) == 0) {
          w0[pbit >> 5] = a0;
          w1[pbit >> 5] = a1;
        }
      }
    }
  } else {
    // c = sum of the comparison bits; symbols beta = ceil(t 2^W / L^G) as quarter_field
    auto code = [&](int j, uint32_t& cl, uint32_t& ch) {
      cl = 0u; ch = 0u;
#pragma unroll
      for (int k = 0; k < L - 1; ++k) {
        const unsigned long long d = f2_sub(t2[k], u2[j]);
        cl += (uint32_t)d >> 31;
        ch += (uint32_t)(d >> 32) >> 31;
      }
    };
#pragma unroll
    for (int sy = 0; sy < F::NG; ++sy) {
      uint32_t tl = 0u, th = 0u;
#pragma unroll
      for (int k = 0; k < F::G; ++k) {
        uint32_t cl, ch;
        code(sy * F::G + k, cl, ch);
        tl = tl * (uint32_t)L + cl;
        th = th * (uint32_t)L + ch;
      }
      put_bits(w0, sy * F::W, F::W, ((tl << F::W) + F::LG - 1u) / F::LG);
      put_bits(w1, sy * F::W, F::W, ((th << F::W) + F::LG - 1u) / F::LG);
    }
    if constexpr (F::R > 0) {
      uint32_t tl = 0u, th = 0u;
#pragma unroll
      for (int k = 0; k < F::R; ++k) {
        uint32_t cl, ch;
        code(32 - F::R + k, cl, ch);
        tl = tl * (uint32_t)L + cl;
        th = th * (uint32_t)L + ch;
      }
      put_bits(w0, F::NG * F::W, F::WT, ((tl << F::WT) + F::LR - 1u) / F::LR);
      put_bits(w1, F::NG * F::W, F::WT, ((th << F::WT) + F::LR - 1u) / F::LR);
    }
  }
}

// One half of every row of a 64-slot block (see above).  stage: the block's half-row
// slots (thread tid's 128 bytes at tid * kHalfStride); smask: the (layer, head)'s sign
// masks, one word per fp16 pair of dims (0x8000 in a half whose sign is -1).
template <int BASE, int L>
__device__ void rows_half(const QuantArgs& a, int b, int l, int h, bool hi, int64_t s0,
                          int nslots, uint8_t* stage, const uint32_t* smask) {
  using F = Fmt<L>;
  constexpr int kWords = (4 * F::QB + 31) / 32;
  constexpr int kRecW = (2 * F::RB + (BASE == SEMKV_BASE_TQ ? 4 : 8)) / 4;
  constexpr int kSh = (2 * F::QB) & 31;        // bit offset of half 1 in its first word
  constexpr int kWb = (2 * F::QB) >> 5;        // that word
  constexpr int kW0 = (2 * F::QB + 31) / 32;   // words half 0 touches
  constexpr int kW1 = (kSh + 2 * F::QB + 31) / 32;  // words half 1 touches, from kWb
  static_assert(kWords <= 12 && F::QB <= 96 && kW1 <= 7, "row image size");
  const int tid = threadIdx.x, f = tid & 1;
  const int64_t cap = hi ? a.hi_cap : a.lo_cap;
  const int64_t pbase = hi ? a.hi_base : a.lo_base;
  const int64_t bh = ((int64_t)b * a.NL + l) * a.H + h;
  // ---- the half, sign-flipped on its fp16 bits (the signs are +-1), as pairs
  unsigned long long xp[32];
  if ((tid >> 2) < nslots) {
    const uint4* src = reinterpret_cast<const uint4*>(stage + tid * kHalfStride);
    const uint4* msk = reinterpret_cast<const uint4*>(smask + 32 * f);
    uint32_t wv[32];
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const uint4 u = src[c], m = msk[c];
      wv[4 * c] = u.x ^ m.x; wv[4 * c + 1] = u.y ^ m.y;
      wv[4 * c + 2] = u.z ^ m.z; wv[4 * c + 3] = u.w ^ m.w;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const uint32_t lo = wv[j >> 1], hi2 = wv[16 + (j >> 1)];
      const int sh = 16 * (j & 1);
      xp[j] = f2_pack(f16_to_f32((uint16_t)(lo >> sh)), f16_to_f32((uint16_t)(hi2 >> sh)));
    }
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j) xp[j] = 0ull;
  }
  uint32_t param;
  float invq;  // TQ: 1/n;  affine: 1/s
  float zq = 0.0f;
  bool live;
  if constexpr (BASE == SEMKV_BASE_TQ) {
    // the norm's fixed tree: 32 in-order partials of 4 squares (this half holds partials
    // 16f + g in the low lanes, 16f + g + 8 in the high ones), then the pairwise stages
    // 16 (across the halves), 8, 4, 2, 1
    // (a square of an fp16 value is exact in binary32, so a fused x * x + v rounds as
    // the separate multiply and add do)
    float pn[8];
#pragma unroll
    for (int g = 0; g < 8; ++g) {
      unsigned long long v = f2_mul(xp[4 * g], xp[4 * g]);
#pragma unroll
      for (int k = 1; k < 4; ++k) v = f2_add(v, f2_mul(xp[4 * g + k], xp[4 * g + k]));
      const float plo = __shfl_xor_sync(0xffffffffu, f2_lo(v), 1);
      const float phi = __shfl_xor_sync(0xffffffffu, f2_hi(v), 1);
      // partials g + (g + 16) and (g + 8) + (g + 24): the same sums in both halves
      const unsigned long long sp = f2_add(v, f2_pack(plo, phi));
      pn[g] = __fadd_rn(f2_lo(sp), f2_hi(sp));
    }
#pragma unroll
    for (int off = 4; off >= 1; off >>= 1)
#pragma unroll
      for (int g = 0; g < off; ++g) pn[g] = __fadd_rn(pn[g], pn[g + off]);
    const uint16_t n16 = f16_param(__fsqrt_rn(pn[0]));
    param = n16;
    const float n = f16_to_f32(n16);
    live = n != 0.0f;
    invq = live ? __fdiv_rn(1.0f, n) : 0.0f;
  }
  // ---- butterflies: stages 1..32 in the thread, stage 64 with the partner half.  Half 0
  // keeps a + b and half 1 a - b (a from half 0): fma(own, +-1, partner), whose product
  // is exact, rounds partner +- own once, which is that sum or difference.
  fwht_half(xp);
  {
    const float sg = f ? -1.0f : 1.0f;
    const unsigned long long sg2 = f2_pack(sg, sg);
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float plo = __shfl_xor_sync(0xffffffffu, f2_lo(xp[j]), 1);
      const float phi = __shfl_xor_sync(0xffffffffu, f2_hi(xp[j]), 1);
      xp[j] = f2_fma(xp[j], sg2, f2_pack(plo, phi));
    }
  }
  if constexpr (BASE == SEMKV_BASE_AFFINE_HAD) {
    float mn = INFINITY, mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      xp[j] = f2_pack(__fmul_rn(f2_lo(xp[j]), kInvSqrtD), __fmul_rn(f2_hi(xp[j]), kInvSqrtD));
      mn = fminf(mn, fminf(f2_lo(xp[j]), f2_hi(xp[j])));
      mx = fmaxf(mx, fmaxf(f2_lo(xp[j]), f2_hi(xp[j])));
    }
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    // a zero extreme is taken as +0 (min/max may return either signed zero)
    if (mn == 0.0f) mn = 0.0f;
    if (mx == 0.0f) mx = 0.0f;
    uint16_t z16 = __half_as_ushort(__float2half_rd(mn));
    if (z16 == 0xFC00u) z16 = 0xFBFFu;
    zq = f16_to_f32(z16);
    const uint16_t s16 = f16_param(__fdiv_rn(__fsub_rn(mx, zq), (float)(L - 1)));
    const float sv = f16_to_f32(s16);
    live = sv > 0.0f;
    // 1/s, or 0 when s == 0: then every (u - z) * 0 clamps and rounds to code 0
    invq = live ? __fdiv_rn(1.0f, sv) : 0.0f;
    param = (uint32_t)s16 | ((uint32_t)z16 << 16);
  }
  // ---- codes, quarter 2f from the low lanes, then quarter 2f + 1 from the high ones
  uint32_t lw[7];
#pragma unroll
  for (int k = 0; k < 7; ++k) lw[k] = 0u;
  const unsigned long long inv2 = f2_pack(invq, invq);
  if constexpr (BASE == SEMKV_BASE_TQ) {
    // c = #{k : u > thr_k} (ties go low); a zero-norm row compares against +inf
    const float* tg = hi ? a.thr_hi : a.thr_lo;
    unsigned long long t2[7];
#pragma unroll
    for (int k = 0; k < L - 1; ++k) {
      const float tk = live ? __fadd_rn(__ldg(tg + k), 0.0f) : INFINITY;
      t2[k] = f2_pack(tk, tk);
    }
    // u = y * fl(1/n), rounded before the comparisons subtract it
#pragma unroll
    for (int j = 0; j < 32; ++j) xp[j] = f2_pack(__fmul_rn(f2_lo(xp[j]), invq), __fmul_rn(f2_hi(xp[j]), invq));
    uint32_t fw0[3], fw1[3];
    tq_fields<L>(xp, t2, fw0, fw1);
    or_field<7>(lw, 0, fw0);
    or_field<7>(lw, F::QB, fw1);
  } else {
    // rint(clamp((u - z) / s)) = clamp(rint(...)) for integer bounds; + 1.5 * 2^23 rounds
    // to nearest even and leaves the code in the low bits of the pattern
    const unsigned long long z2 = f2_pack(zq, zq);
    const unsigned long long mg2 = f2_pack(12582912.0f, 12582912.0f);
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const unsigned long long d = f2_mul(f2_sub(xp[j], z2), inv2);
      const float ylo = fminf(fmaxf(f2_lo(d), 0.0f), (float)(L - 1));
      const float yhi = fminf(fmaxf(f2_hi(d), 0.0f), (float)(L - 1));
      xp[j] = f2_add(f2_pack(ylo, yhi), mg2);
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      uint32_t m[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) m[j] = __float_as_uint(q ? f2_hi(xp[j]) : f2_lo(xp[j]));
      uint32_t fw[3];
      quarter_field_off<L, 0x4B400000u>(m, fw);
      or_field<7>(lw, q * F::QB, fw);
    }
  }
  // ---- the row's bit image and parameters, in half 0's slot: half 0 writes words
  // 0..kWb (word kWb with half 1's low bits when half 1 starts inside it), half 1 the rest
  uint32_t* img = reinterpret_cast<uint32_t*>(stage + (tid & ~1) * kHalfStride);
  if constexpr (kSh != 0) {
#pragma unroll
    for (int k = kW1 - 1; k >= 0; --k) {
      const uint32_t v = (lw[k] << kSh) | (k > 0 ? lw[k - 1] >> (32 - kSh) : 0u);
      if (f) lw[k] = v;
    }
  }
  const uint32_t first1 = __shfl_xor_sync(0xffffffffu, lw[0], 1);
  __syncwarp();  // both halves' values were read from the slots
  if ((tid >> 2) < nslots) {
    if (f == 0) {
#pragma unroll
      for (int k = 0; k < kW0; ++k) img[k] = (kSh != 0 && k == kWb) ? (lw[k] | first1) : lw[k];
      img[kRowBitWords] = param;
    } else {
#pragma unroll
      for (int k = (kSh != 0 ? 1 : 0); k < kW1; ++k) img[kWb + k] = lw[k];
    }
  }
  // ---- records: slot i's two rows are threads 4i .. 4i + 3, so each warp assembles its
  // own 8 slots' records (contiguous words, one 4-byte word per lane and step)
  __syncwarp();
  const int warp = tid >> 5, lane = tid & 31;
  const int ns = min(8, nslots - 8 * warp);
  uint32_t* recs = reinterpret_cast<uint32_t*>(hi ? a.hi_pool : a.lo_pool) +
                   (bh * cap + pbase + s0 + 8 * warp) * kRecW;
  for (int wi = lane; wi < ns * kRecW; wi += 32) {
    const int i = 8 * warp + wi / kRecW, j = wi - (wi / kRecW) * kRecW;
    const uint32_t* K = reinterpret_cast<const uint32_t*>(stage + (4 * i) * kHalfStride);
    const uint32_t* V = reinterpret_cast<const uint32_t*>(stage + (4 * i + 2) * kHalfStride);
    uint32_t word;
    if (4 * j >= 2 * F::RB) {
      const int pj = j - (2 * F::RB) / 4;
      if constexpr (BASE == SEMKV_BASE_TQ) word = K[kRowBitWords] | (V[kRowBitWords] << 16);
      else word = pj ? V[kRowBitWords] : K[kRowBitWords];
    } else if (4 * j + 4 <= F::RB) {
      word = K[j];
    } else {
      const int vb = 4 * j - F::RB;  // byte of the V row at this word's first byte
      if (vb >= 0) word = __funnelshift_r(V[vb >> 2], V[(vb >> 2) + 1], 8 * (vb & 3));
      else word = K[j] | (V[0] << (8 * -vb));
    }
    recs[wi] = word;
  }
}

// ---- shared addresses and mbarriers
__device__ __forceinline__ uint32_t dsmem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void dbar_init(uint64_t* bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(dsmem_u32(bar)) : "memory");
}
// block t of the pass, decoded once: (sequence, layer, KV head), pool, first slot and
// slot count (32-bit arithmetic: the launcher keeps the block count below 2^31)
struct RowsTile {
  int b, l, h;
  bool hi;
  int s0, nslots;
};
__device__ __forceinline__ RowsTile rows_tile(uint32_t t, uint32_t nb_hi, uint32_t per_bh,
                                              uint32_t n_hi, uint32_t n_lo, uint32_t H,
                                              uint32_t NL) {
  RowsTile x;
  const uint32_t bhi = t / per_bh, r = t - bhi * per_bh;
  x.hi = r < nb_hi;
  x.s0 = (int)((x.hi ? r : r - nb_hi) * kRowSlots);
  x.nslots = min(kRowSlots, (int)(x.hi ? n_hi : n_lo) - x.s0);
  const uint32_t q = bhi / H;
  x.h = (int)(bhi - q * H);
  x.b = (int)(q / NL);
  x.l = (int)(q - (uint32_t)x.b * NL);
  return x;
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dsmem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Persistent CTAs of 256 threads over the blocks (64 slots of one pool of one (sequence,
// layer, KV head)), in a two-stage pipeline: while a block is quantized, the halves of
// the CTA's next block are already on their way.  Thread tid brings half tid & 1 of its
// row into its own slot of the stage with eight 16-byte cp.async copies (one commit
// group per block), and the first 64 threads write the next block's sign masks; a
// thread waits for its own group, then the CTA barrier (the only one per block)
// publishes the stage.
template <int BASE>
__global__ void __launch_bounds__(kRows2Threads, rows2_ctas(BASE)) quantize_rows_kernel(QuantArgs a, int64_t n_hi, int64_t n_lo) {
  extern __shared__ __align__(128) uint8_t rstage[];  // 2 stages of 256 half-row slots
  __shared__ __align__(16) uint32_t smask[2][64];
  const int tid = threadIdx.x;
  const uint32_t nb_hi = (uint32_t)((n_hi + kRowSlots - 1) / kRowSlots);
  const uint32_t per_bh = nb_hi + (uint32_t)((n_lo + kRowSlots - 1) / kRowSlots);
  const uint32_t total = (uint32_t)a.B * a.NL * a.H * per_bh;
  auto tile = [&](uint32_t t) {
    return rows_tile(t, nb_hi, per_bh, (uint32_t)n_hi, (uint32_t)n_lo, a.H, a.NL);
  };
  // this thread's half row of block x into stage st (and, for tid < 64, a sign mask word)
  auto issue = [&](const RowsTile& x, int st) {
    if (tid < 64) {
      const char2 s2 = *reinterpret_cast<const char2*>(a.signs + ((int64_t)x.l * a.H + x.h) * kHeadDim + 2 * tid);
      smask[st][tid] = (s2.x < 0 ? 0x8000u : 0u) | (s2.y < 0 ? 0x80000000u : 0u);
    }
    const int i = tid >> 2;
    if (i < x.nslots) {
      const int64_t cap = x.hi ? a.hi_cap : a.lo_cap;
      const int32_t* tokmap = (x.hi ? a.hi_tok : a.lo_tok) + (int64_t)x.b * cap + (x.hi ? a.hi_base : a.lo_base);
      const int64_t tk = (int64_t)tokmap[x.s0 + i] - a.tok_base;
      const int64_t bh = ((int64_t)x.b * a.NL + x.l) * a.H + x.h;
      const uint16_t* src = (((tid >> 1) & 1) ? a.v : a.k) + (bh * a.Tsrc + tk) * kHeadDim + 64 * (tid & 1);
      uint8_t* dst = rstage + st * kRows2StageBytes + tid * kHalfStride;
#pragma unroll
      for (int c = 0; c < 8; ++c) cp_async16(dst + 16 * c, src + 8 * c);
    }
    cp_async_commit();
  };
  uint32_t t = blockIdx.x;
  RowsTile cur{};
  if (t < total) {
    cur = tile(t);
    issue(cur, 0);
  }
  for (int k = 0; t < total; t += gridDim.x, ++k) {
    const int st = k & 1;
    // this thread's copies of block k have landed; after the barrier every thread's have,
    // and every warp is done with the other stage (block k - 1), which the copies of
    // block k + 1 then take over
    cp_async_wait<0>();
    __syncthreads();
    RowsTile nxt{};
    if (t + gridDim.x < total) {
      nxt = tile(t + gridDim.x);
      issue(nxt, st ^ 1);
    }
    uint8_t* stage = rstage + st * kRows2StageBytes;
    switch (cur.hi ? a.L_hi : a.L_lo) {
#define SEMKV_ROWS_CASE(LV) \
      case LV: rows_half<BASE, LV>(a, cur.b, cur.l, cur.h, cur.hi, cur.s0, cur.nslots, stage, smask[st]); break;
      SEMKV_ROWS_CASE(2) SEMKV_ROWS_CASE(3) SEMKV_ROWS_CASE(4) SEMKV_ROWS_CASE(5)
      SEMKV_ROWS_CASE(6) SEMKV_ROWS_CASE(7) SEMKV_ROWS_CASE(8)
#undef SEMKV_ROWS_CASE
      default: break;
    }
    cur = nxt;
  }
}
// ------------------------------------------------- fake quantization ---------
// Every row quantized at its token's precision and reconstructed to fp16 (the quality
// protocol of Sec. 4.1), in binary32 in this order:
//   affine: x^_d = fp16( z + s * c_d )
//   rotated affine: y = FWHT(z + s * c);  x^_d = fp16( (sign_d y_d) * fp32(1/sqrt 128) )
//   TQ:     y = FWHT(cb[c]) (the quantizer's butterflies);  x^_d = fp16( (sign_d y_d) * (n/128) )
// A CTA of 128 threads takes 64 tokens of one (sequence, layer, KV head): thread r
// owns row r (K of token r/2 when r is even, V when odd), in registers; rows are
// staged through shared memory on the way in and out for coalesced transfers.

// Affine base: a CTA per 64-token block, rows staged through shared memory in and out
// (coalesced), each row kept as fp16 pairs (96 registers: 5 CTAs per SM).
__global__ void __launch_bounds__(128, 5) fake_affine_kernel(FakeArgs a) {
  __shared__ __align__(16) uint8_t stage[128 * kRowStride];
  const int tid = threadIdx.x;
  const int64_t bhs = (int64_t)a.B * a.NL * a.H;
  for (int64_t bhi = blockIdx.y; bhi < bhs; bhi += gridDim.y) {
    const int b = (int)(bhi / ((int64_t)a.H * a.NL));
    for (int t0 = blockIdx.x * kRowSlots; t0 < a.T; t0 += gridDim.x * kRowSlots) {
      const int nt = min(kRowSlots, a.T - t0);
      const int64_t row0 = bhi * a.T + t0;
      for (int c = tid; c < 128 * 16; c += 128) {
        const int r = c >> 4, ch = c & 15, i = r >> 1;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (i < nt) v = __ldg(reinterpret_cast<const uint4*>(((r & 1) ? a.v : a.k) + (row0 + i) * kHeadDim) + ch);
        *reinterpret_cast<uint4*>(stage + r * kRowStride + ch * 16) = v;
      }
      __syncthreads();
      const int i = tid >> 1;
      const bool hi = i < nt && (a.is_high == nullptr || a.is_high[(int64_t)b * a.T + t0 + i] != 0);
      const int L = (a.is_high == nullptr || hi) ? a.L_hi : a.L_lo;
      uint32_t ov[64];  // the row's fp16 outputs, in pairs
      {
        // x^_d = fp16(z + s c_d), the row kept as fp16 pairs (fewer registers, more CTAs)
        uint32_t hv[64];
#pragma unroll
        for (int ch = 0; ch < 16; ++ch) {
          const uint4 u = *reinterpret_cast<const uint4*>(stage + tid * kRowStride + ch * 16);
          hv[4 * ch] = u.x;
          hv[4 * ch + 1] = u.y;
          hv[4 * ch + 2] = u.z;
          hv[4 * ch + 3] = u.w;
        }
        // row minimum and maximum on fp16 pairs (exact)
        __half2 mn2 = *reinterpret_cast<const __half2*>(&hv[0]), mx2 = mn2;
#pragma unroll
        for (int j = 1; j < 64; ++j) {
          const __half2 x2 = *reinterpret_cast<const __half2*>(&hv[j]);
          mn2 = __hmin2(mn2, x2);
          mx2 = __hmax2(mx2, x2);
        }
        float mn = fminf(__low2float(mn2), __high2float(mn2));
        float mx = fmaxf(__low2float(mx2), __high2float(mx2));
        if (mn == 0.0f) mn = 0.0f;
        if (mx == 0.0f) mx = 0.0f;
        const uint16_t s16 = f16_param(__fdiv_rn(__fsub_rn(mx, mn), (float)(L - 1)));
        const float sv = f16_to_f32(s16), z = f16_to_f32(__half_as_ushort(__float2half_rn(mn)));
        const float inv = sv != 0.0f ? __fdiv_rn(1.0f, sv) : 0.0f;
        // c = rint(min((x - z) / s, L - 1)) as an integer-valued float (x >= z: z is the
        // row minimum; inv = 0 when s = 0, so every code is 0): adding and taking off
        // 1.5 * 2^23 rounds to nearest even, as the float-to-int conversion would
#pragma unroll
        for (int j = 0; j < 64; ++j) {
          float r[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float x = f16_to_f32((uint16_t)(hv[j] >> (16 * e)));
            const float y = fminf(__fmul_rn(__fsub_rn(x, z), inv), (float)(L - 1));
            const float c = __fsub_rn(__fadd_rn(y, 12582912.0f), 12582912.0f);
            r[e] = __fadd_rn(z, __fmul_rn(sv, c));
          }
          const __half2 h2 = __floats2half2_rn(r[0], r[1]);
          ov[j] = *reinterpret_cast<const uint32_t*>(&h2);
        }
      }
      __syncthreads();  // every row is read: the stage takes the outputs
#pragma unroll
      for (int ch = 0; ch < 16; ++ch)
        *reinterpret_cast<uint4*>(stage + tid * kRowStride + ch * 16) =
            make_uint4(ov[4 * ch], ov[4 * ch + 1], ov[4 * ch + 2], ov[4 * ch + 3]);
      __syncthreads();
      for (int c = tid; c < 128 * 16; c += 128) {
        const int r = c >> 4, ch = c & 15, ii = r >> 1;
        if (ii < nt)
          reinterpret_cast<uint4*>(((r & 1) ? a.v_out : a.k_out) + (row0 + ii) * kHeadDim)[ch] =
              *reinterpret_cast<const uint4*>(stage + r * kRowStride + ch * 16);
      }
      __syncthreads();
    }
  }
}

// Rotated affine and TQ: two threads per row, as the rows quantizer.  Persistent CTAs of
// 256 threads over the 64-token blocks of every (sequence, layer, KV head): thread tid
// holds half f = tid & 1 of row tid >> 1 (K of token tid >> 2 when bit 1 is 0, V when 1)
// as 32 packed pairs (x_j, x_{j+32}), the next block's halves arriving by 16-byte
// cp.async copies under the current block (one CTA barrier per block).  Both
// transforms run the quantizer's butterflies (stages 1..32 in the thread, stage 64 with
// the partner lane); the reconstruction is written back as fp16 with 16-byte stores.

// stage 64 of the butterflies across the two halves of a row (half 0 keeps a + b, half 1
// a - b, a from half 0): fma(own, +-1, partner) rounds partner +- own once
__device__ __forceinline__ void fwht_stage64(unsigned long long (&xp)[32], unsigned long long sg2) {
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float plo = __shfl_xor_sync(0xffffffffu, f2_lo(xp[j]), 1);
    const float phi = __shfl_xor_sync(0xffffffffu, f2_hi(xp[j]), 1);
    xp[j] = f2_fma(xp[j], sg2, f2_pack(plo, phi));
  }
}

// The codebook entry of each of a pair's two values: c = #{k : u > thr_k} over the
// kLmax - 1 thresholds (the row's own L - 1 of them, then +inf), from the sign bits of
// thr_k - u as in tq_fields
template <int kLmax>
__device__ __forceinline__ unsigned long long tq_dequant2(unsigned long long u2,
                                                          const unsigned long long (&t2)[7],
                                                          const float* cb) {
  uint32_t cl = 0u, ch = 0u;
#pragma unroll
  for (int k = 0; k < kLmax - 1; ++k) {
    const unsigned long long d = f2_sub(t2[k], u2);
    cl += (uint32_t)d >> 31;
    ch += (uint32_t)(d >> 32) >> 31;
  }
  return f2_pack(cb[cl], cb[ch]);
}

// One half of a row (see above): slot holds its fp16 values, mask the sign masks of its
// dims; out: the reconstruction's fp16 pairs for dims 64f + 2p, 64f + 2p + 1.
template <int BASE, int kLmax>
__device__ __forceinline__ void fake_half(const uint8_t* slot, const uint32_t* mask, int f, int L,
                                          bool sel_hi, const float (*cbs)[8], const FakeArgs& a,
                                          uint32_t (&out)[32]) {
  unsigned long long xp[32];
  {
    const uint4* src = reinterpret_cast<const uint4*>(slot);
    const uint4* msk = reinterpret_cast<const uint4*>(mask);
    uint32_t wv[32];
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const uint4 u = src[c], m = msk[c];
      wv[4 * c] = u.x ^ m.x; wv[4 * c + 1] = u.y ^ m.y;
      wv[4 * c + 2] = u.z ^ m.z; wv[4 * c + 3] = u.w ^ m.w;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const uint32_t lo = wv[j >> 1], hi2 = wv[16 + (j >> 1)];
      const int sh = 16 * (j & 1);
      xp[j] = f2_pack(f16_to_f32((uint16_t)(lo >> sh)), f16_to_f32((uint16_t)(hi2 >> sh)));
    }
  }
  const float sg = f ? -1.0f : 1.0f;
  const unsigned long long sg2 = f2_pack(sg, sg);
  float post;  // the reconstruction's final factor: fp32(1/sqrt 128), or n / 128
  if constexpr (BASE == SEMKV_BASE_AFFINE_HAD) {
    // y = FWHT(z + s c);  x^_d = fp16((sign_d y_d) * fp32(1/sqrt 128))
    fwht_half(xp);
    fwht_stage64(xp, sg2);
    float mn = INFINITY, mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      xp[j] = f2_pack(__fmul_rn(f2_lo(xp[j]), kInvSqrtD), __fmul_rn(f2_hi(xp[j]), kInvSqrtD));
      mn = fminf(mn, fminf(f2_lo(xp[j]), f2_hi(xp[j])));
      mx = fmaxf(mx, fmaxf(f2_lo(xp[j]), f2_hi(xp[j])));
    }
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    if (mn == 0.0f) mn = 0.0f;
    if (mx == 0.0f) mx = 0.0f;
    uint16_t z16 = __half_as_ushort(__float2half_rd(mn));
    if (z16 == 0xFC00u) z16 = 0xFBFFu;
    const float z = f16_to_f32(z16);
    const float sv = f16_to_f32(f16_param(__fdiv_rn(__fsub_rn(mx, z), (float)(L - 1))));
    const float inv = sv > 0.0f ? __fdiv_rn(1.0f, sv) : 0.0f;
    const unsigned long long z2 = f2_pack(z, z), inv2 = f2_pack(inv, inv), s2 = f2_pack(sv, sv);
    const unsigned long long mg2 = f2_pack(12582912.0f, 12582912.0f);
    const float top = (float)(L - 1);
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      // c = rint(clamp((x - z) / s)) as an integer-valued float (every code 0 when s = 0);
      // z + s c: s c is exact (an fp16 value times an integer below 8), so the fused
      // multiply-add rounds as the separate multiply and add
      const unsigned long long d = f2_mul(f2_sub(xp[j], z2), inv2);
      const float ylo = fminf(fmaxf(f2_lo(d), 0.0f), top), yhi = fminf(fmaxf(f2_hi(d), 0.0f), top);
      const unsigned long long c2 = f2_sub(f2_add(f2_pack(ylo, yhi), mg2), mg2);
      xp[j] = f2_fma(s2, c2, z2);
    }
    post = kInvSqrtD;
  } else {
    // y = FWHT(cb[c]);  x^_d = fp16((sign_d y_d) * (n / 128))
    float pn[8];
#pragma unroll
    for (int g = 0; g < 8; ++g) {
      // (a square of an fp16 value is exact: a fused x * x + v rounds as the separate ops)
      unsigned long long v = f2_mul(xp[4 * g], xp[4 * g]);
#pragma unroll
      for (int k = 1; k < 4; ++k) v = f2_add(v, f2_mul(xp[4 * g + k], xp[4 * g + k]));
      const float plo = __shfl_xor_sync(0xffffffffu, f2_lo(v), 1);
      const float phi = __shfl_xor_sync(0xffffffffu, f2_hi(v), 1);
      const unsigned long long sp = f2_add(v, f2_pack(plo, phi));
      pn[g] = __fadd_rn(f2_lo(sp), f2_hi(sp));
    }
#pragma unroll
    for (int off = 4; off >= 1; off >>= 1)
#pragma unroll
      for (int g = 0; g < off; ++g) pn[g] = __fadd_rn(pn[g], pn[g + off]);
    const float n = f16_to_f32(f16_param(__fsqrt_rn(pn[0])));
    const float inv = n != 0.0f ? __fdiv_rn(1.0f, n) : 0.0f;
    const float* tg = sel_hi ? a.thr_hi : a.thr_lo;
    unsigned long long t2[7];
#pragma unroll
    for (int k = 0; k < kLmax - 1; ++k) {
      // a zero-norm row compares against +inf (all codes 0)
      const float tk = (n != 0.0f && k < L - 1) ? __fadd_rn(__ldg(tg + k), 0.0f) : INFINITY;
      t2[k] = f2_pack(tk, tk);
    }
    fwht_half(xp);
    fwht_stage64(xp, sg2);
    const float* cb = cbs[sel_hi ? 0 : 1];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      // u = y * fl(1/n), rounded before the comparisons subtract it
      const unsigned long long u2 = f2_pack(__fmul_rn(f2_lo(xp[j]), inv), __fmul_rn(f2_hi(xp[j]), inv));
      xp[j] = tq_dequant2<kLmax>(u2, t2, cb);
    }
    post = n * 0.0078125f;
  }
  fwht_half(xp);
  fwht_stage64(xp, sg2);
  // (sign_d y_d) * post = sign_d (y_d * post): the product rounds to fp16 next, no add
  const unsigned long long p2 = f2_pack(post, post);
#pragma unroll
  for (int j = 0; j < 32; ++j) xp[j] = f2_mul(xp[j], p2);
#pragma unroll
  for (int p = 0; p < 16; ++p) {
    const __half2 h0 = __floats2half2_rn(f2_lo(xp[2 * p]), f2_lo(xp[2 * p + 1]));
    const __half2 h1 = __floats2half2_rn(f2_hi(xp[2 * p]), f2_hi(xp[2 * p + 1]));
    out[p] = *reinterpret_cast<const uint32_t*>(&h0) ^ mask[p];
    out[16 + p] = *reinterpret_cast<const uint32_t*>(&h1) ^ mask[16 + p];
  }
}

template <int BASE>
__global__ void __launch_bounds__(kRows2Threads, 2) fake_rows_kernel(FakeArgs a, int Lmax) {
  extern __shared__ __align__(128) uint8_t fstage[];  // 2 stages of 256 half-row slots
  __shared__ __align__(16) uint32_t smask[2][64];
  __shared__ float cbs[2][8];
  const int tid = threadIdx.x, f = tid & 1, r = tid >> 1, i = r >> 1;
  if (BASE == SEMKV_BASE_TQ && tid < 16) {
    const int which = tid >> 3, k = tid & 7;
    const int L = which ? a.L_lo : a.L_hi;
    cbs[which][k] = k < L ? (which ? a.cent_lo : a.cent_hi)[k] : 0.0f;
  }
  const uint32_t nblk = (uint32_t)((a.T + kRowSlots - 1) / kRowSlots);
  const uint32_t total = (uint32_t)a.B * a.NL * a.H * nblk;
  // block t: (sequence, layer, head) index and first token
  auto decode = [&](uint32_t t, uint32_t& bhi, int& t0) {
    bhi = t / nblk;
    t0 = (int)(t - bhi * nblk) * kRowSlots;
  };
  auto issue = [&](uint32_t t, int st) {
    uint32_t bhi;
    int t0;
    decode(t, bhi, t0);
    if (tid < 64) {
      const uint32_t q = bhi / (uint32_t)a.H;
      const int h = (int)(bhi - q * a.H), l = (int)(q % (uint32_t)a.NL);
      const char2 s2 = *reinterpret_cast<const char2*>(a.signs + ((int64_t)l * a.H + h) * kHeadDim + 2 * tid);
      smask[st][tid] = (s2.x < 0 ? 0x8000u : 0u) | (s2.y < 0 ? 0x80000000u : 0u);
    }
    if (i < a.T - t0) {
      const uint16_t* src = ((r & 1) ? a.v : a.k) + ((int64_t)bhi * a.T + t0 + i) * kHeadDim + 64 * f;
      uint8_t* dst = fstage + st * kRows2StageBytes + tid * kHalfStride;
#pragma unroll
      for (int c = 0; c < 8; ++c) cp_async16(dst + 16 * c, src + 8 * c);
    }
    cp_async_commit();
  };
  uint32_t t = blockIdx.x;
  if (t < total) issue(t, 0);
  for (int k = 0; t < total; t += gridDim.x, ++k) {
    const int st = k & 1;
    cp_async_wait<0>();
    __syncthreads();  // the stage and its masks are published; the other stage is free
    if (t + gridDim.x < total) issue(t + gridDim.x, st ^ 1);
    uint32_t bhi;
    int t0;
    decode(t, bhi, t0);
    const int b = (int)(bhi / ((uint32_t)a.H * a.NL));
    const bool live = i < a.T - t0;
    const bool sel_hi = a.is_high == nullptr || (live && a.is_high[(int64_t)b * a.T + t0 + i] != 0);
    const int L = sel_hi ? a.L_hi : a.L_lo;
    const uint8_t* slot = fstage + st * kRows2StageBytes + tid * kHalfStride;
    uint32_t out[32];
    switch (BASE == SEMKV_BASE_TQ ? Lmax : 2) {
#define SEMKV_FAKE_CASE(LV) \
      case LV: fake_half<BASE, LV>(slot, smask[st] + 32 * f, f, L, sel_hi, cbs, a, out); break;
      SEMKV_FAKE_CASE(2) SEMKV_FAKE_CASE(3) SEMKV_FAKE_CASE(4) SEMKV_FAKE_CASE(5)
      SEMKV_FAKE_CASE(6) SEMKV_FAKE_CASE(7) SEMKV_FAKE_CASE(8)
#undef SEMKV_FAKE_CASE
      default: break;
    }
    if (live) {
      uint4* dst = reinterpret_cast<uint4*>(((r & 1) ? a.v_out : a.k_out) + ((int64_t)bhi * a.T + t0 + i) * kHeadDim + 64 * f);
#pragma unroll
      for (int c = 0; c < 8; ++c) dst[c] = make_uint4(out[4 * c], out[4 * c + 1], out[4 * c + 2], out[4 * c + 3]);
    }
  }
}

// ------------------------------------- dense-rotation TQ rows (tcgen05) --------
// Blocks of 64 slots of one pool of one (sequence, layer, KV head), as for the other
// bases: 128 rows (row r: K of slot r/2 when r is even, V when odd), one level count.
// Persistent CTAs of two groups of 4 warps (two CTAs per SM), each CTA over a range of
// blocks of one (sequence, layer, KV head) whose rotation M (128 x 128 fp16, the B
// operand, K-major: output dims x input dims) it stages once.  A group takes every other
// block of the range: thread r of the group brings row r with sixteen 16-byte cp.async
// copies into the group's A tile (K-major 8-row x 16-byte core matrices: byte
// kg * 2048 + r * 16 holds dims 8 kg .. 8 kg + 7), then one thread issues
// D = X M^T on tcgen05 (kind::f16, M = 128 rows, N = 128 output dims, K = 8 x 16) into
// the group's 128 columns of tensor memory, so TMEM lane r is row r and column c its
// output dim c.  While the MMAs run, thread r takes its row's fixed-tree norm from the
// tile; once they have completed it starts the copies of the group's next block and
// reads its row's w = M x a quarter (32 columns) at a time, the next quarter's load in
// flight while one is coded: u = w * fl(1/n), the codes
// from the thresholds, the quarter bit fields, and the row's bytes straight into its
// record.  The two groups' accumulators are distinct, so one group's MMAs overlap the
// other's epilogue.
constexpr int kDenseThreads = 256;
constexpr uint32_t kDenseM = 128 * 128 * 2;   // the rotation, bytes
constexpr uint32_t kDenseA = 128 * 128 * 2;   // one group's tile of 128 rows
constexpr uint32_t kDenseSmem = kDenseM + 2 * kDenseA + 1024;  // + alignment
// instruction descriptor: fp32 accumulate (bits 4-5 = 1), A and B fp16 (formats 0),
// both K-major, N >> 3 at bits 17-22, M >> 4 at bits 24-28
constexpr uint32_t kDenseIdesc = (1u << 4) | ((128u >> 3) << 17) | ((128u >> 4) << 24);

// shared-memory matrix descriptor without swizzle: start >> 4 (bits 0-13), leading
// (K-direction) core-matrix offset >> 4 (bits 16-29), stride (8-row group) offset >> 4
// (bits 32-45), descriptor version 1 (bits 46-47)
__device__ __forceinline__ uint64_t umma_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}
// 32 columns of this warp's 32 TMEM lanes (lane i of the warp <- TMEM lane 32 (w % 4) + i):
// the load, and the wait that makes them readable.  The wait takes the registers as
// in-out operands, so no use of them can be scheduled before it.
__device__ __forceinline__ void tmem_ld32_start(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&v)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]),
                 "+r"(v[6]), "+r"(v[7]), "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]),
                 "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15]), "+r"(v[16]), "+r"(v[17]),
                 "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]), "+r"(v[22]), "+r"(v[23]),
                 "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]), "+r"(v[29]),
                 "+r"(v[30]), "+r"(v[31])
               :
               : "memory");
}
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}
// barrier of the 128 threads of group g (named barrier 1 + g), with an AND of p
__device__ __forceinline__ bool group_sync_and(int g, bool p) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n"
      " barrier.cta.red.and.pred q, %2, 128, p;\n selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r)
      : "r"((uint32_t)p), "r"(1 + g)
      : "memory");
  return r != 0;
}

// The field of one quarter from its 32 values u (thresholds as in tq_fields: t2[k] the
// pair (thr_k, thr_k)); pairs of neighbouring dims share each packed subtraction.
template <int L>
__device__ __forceinline__ void tq_quarter(const float (&u)[32], const unsigned long long (&t2)[7],
                                           uint32_t (&w)[3]) {
  using F = Fmt<L>;
  w[0] = w[1] = w[2] = 0u;
  if constexpr (F::G == 1 && F::LG == (1u << F::W)) {
    constexpr int W = F::W;
    uint32_t acc = 0u;
#pragma unroll
    for (int jp = 15; jp >= 0; --jp) {
      uint32_t dl[7], dh[7];
#pragma unroll
      for (int k = 0; k < L - 1; ++k) {
        const unsigned long long d = f2_sub(t2[k], f2_pack(u[2 * jp], u[2 * jp + 1]));
        dl[k] = (uint32_t)d;
        dh[k] = (uint32_t)(d >> 32);
      }
#pragma unroll
      for (int e = 1; e >= 0; --e) {  // dim 2jp + 1 first: most significant bit first
        const uint32_t* dd = e ? dh : dl;
        const int j = 2 * jp + e;
#pragma unroll
        for (int b = W - 1; b >= 0; --b) {
          uint32_t bit;
          if constexpr (L == 2) bit = dd[0];
          else if constexpr (L == 4) bit = b == 1 ? dd[1] : (dd[0] ^ dd[1] ^ dd[2]);
          else bit = b == 2 ? dd[3] : b == 1 ? (dd[1] ^ dd[3] ^ dd[5])
                                             : (dd[0] ^ dd[1] ^ dd[2] ^ dd[3] ^ dd[4] ^ dd[5] ^ dd[6]);
          acc = __funnelshift_l(bit, acc, 1);
          const int pbit = j * W + b;
          if ((pbit & 31) == 0) w[pbit >> 5] = acc;
        }
      }
    }
  } else {
    uint32_t t = 0u;
#pragma unroll
    for (int jp = 0; jp < 16; ++jp) {
      uint32_t c[2] = {0u, 0u};
#pragma unroll
      for (int k = 0; k < L - 1; ++k) {
        const unsigned long long d = f2_sub(t2[k], f2_pack(u[2 * jp], u[2 * jp + 1]));
        c[0] += (uint32_t)d >> 31;
        c[1] += (uint32_t)(d >> 32) >> 31;
      }
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = 2 * jp + e;
        if (j < F::NG * F::G) {
          const int k = j % F::G, sy = j / F::G;
          t = (k == 0 ? 0u : t * (uint32_t)L) + c[e];
          if (k == F::G - 1) put_bits(w, sy * F::W, F::W, ((t << F::W) + F::LG - 1u) / F::LG);
        } else {
          const int k = j - F::NG * F::G;
          t = (k == 0 ? 0u : t * (uint32_t)L) + c[e];
          if (k == F::R - 1) put_bits(w, F::NG * F::W, F::WT, ((t << F::WT) + F::LR - 1u) / F::LR);
        }
      }
    }
  }
}

// Row r of a block: codes from TMEM (taddr: this warp's lanes, the group's columns), the
// quarter fields, and the row's bytes into its record (rec: the record; kind 0 = K at
// byte 0, 1 = V at byte RB; its fp16 norm at byte 2 RB + 2 kind)
template <int L>
__device__ __forceinline__ void dense_row(uint32_t taddr, const float* thr, float inv, bool live,
                                          uint16_t n16, uint8_t* rec, int kind, bool store) {
  using F = Fmt<L>;
  constexpr int RB = F::RB;
  unsigned long long t2[7];
#pragma unroll
  for (int k = 0; k < L - 1; ++k) {
    const float tk = live ? __fadd_rn(__ldg(thr + k), 0.0f) : INFINITY;
    t2[k] = f2_pack(tk, tk);
  }
  uint32_t w[13];
#pragma unroll
  for (int k = 0; k < 13; ++k) w[k] = 0u;
  // quarter q + 1's columns load while quarter q is coded
  uint32_t vb[2][32];
  tmem_ld32_start(taddr, vb[0]);
  tmem_ld_wait(vb[0]);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    if (q < 3) tmem_ld32_start(taddr + 32 * (q + 1), vb[(q + 1) & 1]);
    float u[32];
    // u = w * fl(1/n), rounded before the comparisons subtract it
#pragma unroll
    for (int j = 0; j < 32; ++j) u[j] = __fmul_rn(__uint_as_float(vb[q & 1][j]), inv);
    if (q < 3) tmem_ld_wait(vb[(q + 1) & 1]);
    uint32_t fw[3];
    tq_quarter<L>(u, t2, fw);
    or_field<13>(w, q * F::QB, fw);
  }
  if (!store) return;
  // the row's RB bytes: word-aligned for K; V starts 2 bytes into a word when RB = 2 mod 4
  if (kind == 0 || (RB & 3) == 0) {
    uint32_t* dst = reinterpret_cast<uint32_t*>(rec + kind * RB);
#pragma unroll
    for (int k = 0; k < RB / 4; ++k) dst[k] = w[k];
    if constexpr ((RB & 3) != 0)
      *reinterpret_cast<uint16_t*>(rec + kind * RB + 4 * (RB / 4)) = (uint16_t)w[RB / 4];
  } else {
    *reinterpret_cast<uint16_t*>(rec + RB) = (uint16_t)w[0];
    uint32_t* dst = reinterpret_cast<uint32_t*>(rec + RB + 2);
#pragma unroll
    for (int k = 0; k < (RB - 2) / 4; ++k) dst[k] = __funnelshift_r(w[k], w[k + 1], 16);
  }
  *reinterpret_cast<uint16_t*>(rec + 2 * RB + 2 * kind) = n16;
}

__global__ void __launch_bounds__(kDenseThreads, 2)
    quantize_tq_dense_kernel(QuantArgs a, int64_t n_hi, int64_t n_lo) {
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~(uintptr_t)1023);
  uint8_t* mb = base;                       // B: the rotation, core-matrix layout
  __shared__ __align__(8) uint64_t mma_bar[2];
  __shared__ uint32_t tmem_base;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int grp = warp >> 2, row = 32 * (warp & 3) + lane;
  uint8_t* xa = base + kDenseM + grp * kDenseA;  // A: this group's rows
  const int64_t bhl = blockIdx.y;
  const int h = (int)(bhl % a.H), l = (int)((bhl / a.H) % a.NL);
  const int b = (int)(bhl / ((int64_t)a.H * a.NL));
  const int nb_hi = (int)((n_hi + kRowSlots - 1) / kRowSlots);
  const int tiles = nb_hi + (int)((n_lo + kRowSlots - 1) / kRowSlots);
  const int per = (tiles + (int)gridDim.x - 1) / (int)gridDim.x;
  const int j0 = min(tiles, (int)blockIdx.x * per), j1 = min(tiles, j0 + per);

  if (tid == 0) {
    dbar_init(&mma_bar[0]);
    dbar_init(&mma_bar[1]);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;" ::"r"(
                     dsmem_u32(&tmem_base))
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // the rotation: 16-byte chunk c = (row group, k group, row in group) at byte 16 c
  const uint4* msrc = reinterpret_cast<const uint4*>(a.rot + ((int64_t)l * a.H + h) * 128 * 128);
  for (int c = tid; c < 128 * 16; c += kDenseThreads) {
    const int rr = c & 7, kg = (c >> 3) & 15, r = (c >> 7) * 8 + rr;
    reinterpret_cast<uint4*>(mb)[c] = msrc[r * 16 + kg];
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tb = tmem_base;
  const uint32_t tcol = tb + (uint32_t)(grp * 128);           // this group's accumulator
  const uint32_t tlane = tcol + ((uint32_t)(32 * (warp & 3)) << 16);
  const int64_t bh = bhl;  // (sequence, layer, head) index of the pools and the rows

  // block j of the range: pool, first slot, slots
  auto block = [&](int j, bool& hi, int& s0, int& ns) {
    hi = j < nb_hi;
    s0 = (hi ? j : j - nb_hi) * kRowSlots;
    ns = (int)min((int64_t)kRowSlots, (hi ? n_hi : n_lo) - s0);
  };
  // this thread's row of block j into the group's tile
  auto load_row = [&](int j) {
    bool hi;
    int s0, ns;
    block(j, hi, s0, ns);
    if ((row >> 1) < ns) {
      const int64_t cap = hi ? a.hi_cap : a.lo_cap;
      const int32_t* tokmap = (hi ? a.hi_tok : a.lo_tok) + (int64_t)b * cap + (hi ? a.hi_base : a.lo_base);
      const int64_t tk = (int64_t)tokmap[s0 + (row >> 1)] - a.tok_base;
      const uint16_t* src = ((row & 1) ? a.v : a.k) + (bh * a.Tsrc + tk) * kHeadDim;
#pragma unroll
      for (int kg = 0; kg < 16; ++kg) cp_async16(xa + kg * 2048 + row * 16, src + 8 * kg);
    }
    cp_async_commit();
  };

  bool ok = true;
  int j = j0 + grp;
  if (j < j1) load_row(j);
  for (int it = 0; j < j1; j += 2, ++it) {
    bool hi;
    int s0, ns;
    block(j, hi, s0, ns);
    const bool mine = (row >> 1) < ns;
    cp_async_wait<0>();
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the rows, for the MMAs
    group_sync_and(grp, true);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (row == 0) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const uint64_t da = umma_desc(dsmem_u32(xa) + k * 4096, 2048, 128);
        const uint64_t db = umma_desc(dsmem_u32(mb) + k * 256, 128, 2048);
        asm volatile(
            "{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n"
            " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tcol),
            "l"(da), "l"(db), "r"(kDenseIdesc), "r"((uint32_t)(k > 0))
            : "memory");
      }
      asm volatile(
          "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
              dsmem_u32(&mma_bar[grp]))
          : "memory");
    }
    // ---- while the MMAs run: the row's norm (fixed tree: 32 in-order partials of 4
    // squares, then the pairwise stages 16, 8, 4, 2, 1).  Partials g and g + 16 are
    // formed as a pair from chunks kg and kg + 8 (a square of an fp16 value is exact, so
    // a fused multiply-add rounds as the separate operations)
    uint16_t n16 = 0;
    float inv = 0.0f;
    {
      const uint32_t xs = dsmem_u32(xa);  // (shared-space loads: the tile is in shared memory)
      float pn[16];
#pragma unroll
      for (int kg = 0; kg < 8; ++kg) {
        const uint4 ua = ld_shared_v4(xs + kg * 2048 + row * 16);
        const uint4 ub = ld_shared_v4(xs + (kg + 8) * 2048 + row * 16);
        const uint32_t wa[4] = {ua.x, ua.y, ua.z, ua.w}, wb[4] = {ub.x, ub.y, ub.z, ub.w};
#pragma unroll
        for (int g2 = 0; g2 < 2; ++g2) {
          unsigned long long acc = 0ull;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const uint32_t xw = wa[2 * g2 + (e >> 1)], yw = wb[2 * g2 + (e >> 1)];
            const int sh = 16 * (e & 1);
            const unsigned long long x2 = f2_pack(f16_to_f32((uint16_t)(xw >> sh)), f16_to_f32((uint16_t)(yw >> sh)));
            acc = e == 0 ? f2_mul(x2, x2) : f2_add(acc, f2_mul(x2, x2));
          }
          // partials 2kg + g2 and 2kg + g2 + 16, then their sum (stage 16)
          pn[2 * kg + g2] = __fadd_rn(f2_lo(acc), f2_hi(acc));
        }
      }
#pragma unroll
      for (int off = 8; off >= 1; off >>= 1)
#pragma unroll
        for (int g = 0; g < off; ++g) pn[g] = __fadd_rn(pn[g], pn[g + off]);
      n16 = f16_param(__fsqrt_rn(pn[0]));
      const float n = f16_to_f32(n16);
      inv = n != 0.0f ? __fdiv_rn(1.0f, n) : 0.0f;
    }
    ok = group_sync_and(grp, mbar_wait_bounded(&mma_bar[grp], (uint32_t)(it & 1)));
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (!ok) break;
    // the MMAs have read the tile and this thread its row: the next block's row
    if (j + 2 < j1) load_row(j + 2);
    // ---- codes and the record
    const int64_t cap = hi ? a.hi_cap : a.lo_cap;
    const int L = hi ? a.L_hi : a.L_lo;
    const int rec_bytes = 2 * row_bytes_rt(L) + 4;
    uint8_t* rec = (hi ? a.hi_pool : a.lo_pool) +
                   (bh * cap + (hi ? a.hi_base : a.lo_base) + s0 + (row >> 1)) * rec_bytes;
    const float* thr = hi ? a.thr_hi : a.thr_lo;
    const bool live = n16 != 0;
    switch (L) {
#define SEMKV_DENSE_CASE(LV) \
      case LV: dense_row<LV>(tlane, thr, inv, live, n16, rec, row & 1, mine); break;
      SEMKV_DENSE_CASE(2) SEMKV_DENSE_CASE(3) SEMKV_DENSE_CASE(4) SEMKV_DENSE_CASE(5)
      SEMKV_DENSE_CASE(6) SEMKV_DENSE_CASE(7) SEMKV_DENSE_CASE(8)
#undef SEMKV_DENSE_CASE
      default: break;
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  }
  if (!ok && row == 0) raise_error(a.err, kDevWaitTimeout);
  cp_async_wait<0>();
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" ::"r"(tb) : "memory");
}

}  // namespace

cudaError_t launch_fake_quant(const FakeArgs& a, int num_sms, cudaStream_t stream) {
  const int64_t total = (int64_t)a.B * a.NL * a.H * a.T;
  if (total == 0) return cudaSuccess;
  const int64_t bhs = (int64_t)a.B * a.NL * a.H;
  const int64_t nblk = ((int64_t)a.T + kRowSlots - 1) / kRowSlots;
  if (a.base == SEMKV_BASE_AFFINE) {
    const dim3 grid((unsigned)(nblk < 65535 ? nblk : 65535), (unsigned)(bhs < 65535 ? bhs : 65535));
    fake_affine_kernel<<<grid, 128, 0, stream>>>(a);
    return cudaGetLastError();
  }
  static bool attr_set[kAttrDevices] = {};
  const cudaError_t e = once_per_device(attr_set, [] {
    cudaError_t r = cudaFuncSetAttribute(fake_rows_kernel<SEMKV_BASE_AFFINE_HAD>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         2 * kRows2StageBytes);
    if (r == cudaSuccess)
      r = cudaFuncSetAttribute(fake_rows_kernel<SEMKV_BASE_TQ>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, 2 * kRows2StageBytes);
    return r;
  });
  if (e != cudaSuccess) return e;
  // persistent: 2 CTAs of 256 threads per SM (128 registers: both transforms' pairs and
  // the dequantization constants spill at 80); block indices are 32-bit
  if (bhs * nblk > INT32_MAX / 2) return cudaErrorInvalidValue;
  int64_t ctas = (int64_t)(num_sms > 0 ? num_sms : 1) * 2;
  if (ctas > bhs * nblk) ctas = bhs * nblk;
  const int Lmax = a.L_hi > a.L_lo ? a.L_hi : a.L_lo;
  if (a.base == SEMKV_BASE_AFFINE_HAD)
    fake_rows_kernel<SEMKV_BASE_AFFINE_HAD>
        <<<(unsigned)ctas, kRows2Threads, 2 * kRows2StageBytes, stream>>>(a, Lmax);
  else
    fake_rows_kernel<SEMKV_BASE_TQ>
        <<<(unsigned)ctas, kRows2Threads, 2 * kRows2StageBytes, stream>>>(a, Lmax);
  return cudaGetLastError();
}

cudaError_t launch_quantize_pack(const QuantArgs& a, int64_t n_hi, int num_sms,
                                 cudaStream_t stream, bool maps_ready) {
  const int64_t total = (int64_t)a.B * a.NL * a.H * a.n;
  if (total == 0) return cudaSuccess;
  if (a.base == SEMKV_BASE_AFFINE) {
    if (!maps_ready) {
      const int64_t pairs = (int64_t)a.B * a.n;
      scatter_tok_kernel<<<(unsigned)((pairs + 255) / 256), 256, 0, stream>>>(a);
      const cudaError_t e = cudaGetLastError();
      if (e != cudaSuccess) return e;
    }
    // grid x from a simple wave model: with R resident CTAs (kAffineCtas per SM), the pass takes
    // about ceil(CTAs / R) waves of ceil(units / (8 bx)) units per warp; take the
    // cheapest bx (at most 16 units per warp).  The (sequence, layer, head) index runs
    // over grid y (and loops past its limit of 65535)
    const int64_t bhs = (int64_t)a.B * a.NL * a.H;
    const int64_t n_max = n_hi > a.n - n_hi ? n_hi : a.n - n_hi;
    const int64_t units = (n_max + kAffineSlots - 1) / kAffineSlots;
    const int64_t resident = (int64_t)(num_sms > 0 ? num_sms : 1) * kAffineCtas;
    const int64_t rows = 2 * (bhs < 65535 ? bhs : 65535);
    int64_t bx = 1, best = -1;
    for (int64_t pw = 16; pw >= 1; --pw) {
      const int64_t cand = (units + pw * kWarpsPerBlock - 1) / (pw * kWarpsPerBlock);
      const int64_t per = (units + cand * kWarpsPerBlock - 1) / (cand * kWarpsPerBlock);
      const int64_t cost = ((cand * rows + resident - 1) / resident) * per;
      if (best < 0 || cost * 50 < best * 49) {  // a near tie keeps the larger units
        best = cost;
        bx = cand;
      }
    }
    if (bx < 1) bx = 1;
    dim3 grid((unsigned)bx, (unsigned)(bhs < 65535 ? bhs : 65535), 2);
    return launch_pdl(quantize_affine_kernel, grid, dim3(kWarpsPerBlock * 32), 0, stream, a, n_hi,
                      a.n - n_hi);
  }
  // TQ, rotated affine and dense-rotation TQ: slot -> token maps, then the rows by slot
  if (!maps_ready) {
    const int64_t pairs = (int64_t)a.B * a.n;
    scatter_tok_kernel<<<(unsigned)((pairs + 255) / 256), 256, 0, stream>>>(a);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (a.base == SEMKV_BASE_TQ_DENSE) {
    static bool attr_set[kAttrDevices] = {};
    const cudaError_t e = once_per_device(attr_set, [] {
      return cudaFuncSetAttribute(quantize_tq_dense_kernel,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kDenseSmem);
    });
    if (e != cudaSuccess) return e;
    const int64_t bhs = (int64_t)a.B * a.NL * a.H;
    if (bhs > 65535) return cudaErrorInvalidValue;
    const int64_t tiles = (n_hi + kRowSlots - 1) / kRowSlots + (a.n - n_hi + kRowSlots - 1) / kRowSlots;
    int64_t splits = (2 * (int64_t)num_sms + bhs - 1) / bhs;  // about two CTAs per SM
    // (each CTA's two groups take alternate blocks of its range)
    if (splits > (tiles + 1) / 2) splits = (tiles + 1) / 2;
    if (splits < 1) splits = 1;
    const dim3 grid((unsigned)splits, (unsigned)bhs);
    quantize_tq_dense_kernel<<<grid, kDenseThreads, kDenseSmem, stream>>>(a, n_hi, a.n - n_hi);
    return cudaGetLastError();
  }
  // persistent CTAs (rows2_ctas per SM) over every block of both pools
  const int64_t bhs = (int64_t)a.B * a.NL * a.H;
  const int64_t blocks = bhs * ((n_hi + kRowSlots - 1) / kRowSlots +
                                (a.n - n_hi + kRowSlots - 1) / kRowSlots);
  int64_t ctas = (int64_t)(num_sms > 0 ? num_sms : 1) * rows2_ctas(a.base);
  if (ctas > blocks) ctas = blocks;
  if (ctas < 1) return cudaSuccess;
  if (blocks + ctas > INT32_MAX) return cudaErrorInvalidValue;  // block indices are 32-bit
  static bool rows_attr[kAttrDevices] = {};
  {
    const cudaError_t e = once_per_device(rows_attr, [] {
      cudaError_t r = cudaFuncSetAttribute(quantize_rows_kernel<SEMKV_BASE_AFFINE_HAD>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           2 * kRows2StageBytes);
      if (r == cudaSuccess)
        r = cudaFuncSetAttribute(quantize_rows_kernel<SEMKV_BASE_TQ>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, 2 * kRows2StageBytes);
      return r;
    });
    if (e != cudaSuccess) return e;
  }
  if (a.base == SEMKV_BASE_AFFINE_HAD)
    quantize_rows_kernel<SEMKV_BASE_AFFINE_HAD>
        <<<(unsigned)ctas, kRows2Threads, 2 * kRows2StageBytes, stream>>>(a, n_hi, a.n - n_hi);
  else
    quantize_rows_kernel<SEMKV_BASE_TQ>
        <<<(unsigned)ctas, kRows2Threads, 2 * kRows2StageBytes, stream>>>(a, n_hi, a.n - n_hi);
  return cudaGetLastError();
}

}  // namespace semkv
