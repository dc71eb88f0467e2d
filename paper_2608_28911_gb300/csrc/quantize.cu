// quantize.cu — token-wise mixed-precision quantization and mixed-radix packing
// (Eq. 7; Sec. 4.1 affine base; Sec. 4.9 TurboQuant-MSE base).
//
// One warp per (sequence, layer, KV head, token): lane l holds dims 4l..4l+3 of the
// token's K row and V row (one 8-byte load each, 256 contiguous bytes per warp per
// row).  The warp reduces the row statistics with shuffles, computes the 4+4 codes
// per lane, stages the 256 codes in shared memory, builds every group symbol of both
// rows in parallel (one lane per symbol), ORs the symbols into a shared record image
// and writes the record to its pool slot with coalesced 4-byte stores.
//
// Arithmetic (binary32, round to nearest even, no contraction), per row x:
//  affine: s = fp16((max-min)/(L-1)) limited to 65504, z = fp16(min);
//          c = clamp(rint((x - z) * fl(1/s)), 0, L-1)   (all 0 when s == 0)
//  TQ:     w = FWHT(x * sign) with butterflies h = 1..64; n = fp16(sqrt(sum x^2))
//          with the sum taken as 32 in-order partials of 4 squares then an xor
//          butterfly over lanes 16, 8, 4, 2, 1; u = w * fl(1/n); c = #{k: u > t_k}
#include "common.cuh"
#include "kernels.h"

namespace semkv {

namespace {

constexpr int kWarpsPerBlock = 8;
constexpr int kMaxRecWords = 27;  // largest record: affine L=7/8, 2*48+8 = 104 B

struct RowOut {
  uint32_t codes;  // four 8-bit codes, dims 4l..4l+3
  uint16_t p0;     // affine: scale; TQ: norm
  uint16_t p1;     // affine: offset
};

__device__ __forceinline__ void load4(const uint16_t* row, int lane, float x[4]) {
  uint2 u = *reinterpret_cast<const uint2*>(row + 4 * lane);
  x[0] = f16_to_f32((uint16_t)(u.x & 0xFFFF));
  x[1] = f16_to_f32((uint16_t)(u.x >> 16));
  x[2] = f16_to_f32((uint16_t)(u.y & 0xFFFF));
  x[3] = f16_to_f32((uint16_t)(u.y >> 16));
}

template <int L>
__device__ __forceinline__ RowOut affine_row(const float x[4]) {
  float mn = fminf(fminf(x[0], x[1]), fminf(x[2], x[3]));
  float mx = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  }
  // a zero extreme is taken as +0 (fmin/fmax may return either signed zero)
  if (mn == 0.0f) mn = 0.0f;
  if (mx == 0.0f) mx = 0.0f;
  const float s32 = __fdiv_rn(__fsub_rn(mx, mn), (float)(L - 1));
  RowOut o;
  o.p0 = f16_param(s32);
  o.p1 = __half_as_ushort(__float2half_rn(mn));
  const float s = f16_to_f32(o.p0), z = f16_to_f32(o.p1);
  o.codes = 0;
  if (s != 0.0f) {
    const float inv = __fdiv_rn(1.0f, s);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int c = __float2int_rn(__fmul_rn(__fsub_rn(x[j], z), inv));
      c = min(max(c, 0), L - 1);
      o.codes |= (uint32_t)c << (8 * j);
    }
  }
  return o;
}

template <int L>
__device__ __forceinline__ RowOut tq_row(const float x[4], const int8_t* sg, int lane,
                                         const float thr[8]) {
  // sign flip (exact) then the Walsh-Hadamard butterflies in stage order
  const char4 s4 = *reinterpret_cast<const char4*>(sg + 4 * lane);
  float w[4] = {x[0] * (float)s4.x, x[1] * (float)s4.y, x[2] * (float)s4.z,
                x[3] * (float)s4.w};
  {  // h = 1: (0,1), (2,3)
    float a = w[0], b = w[1];
    w[0] = __fadd_rn(a, b); w[1] = __fsub_rn(a, b);
    a = w[2]; b = w[3];
    w[2] = __fadd_rn(a, b); w[3] = __fsub_rn(a, b);
  }
  {  // h = 2: (0,2), (1,3)
    float a = w[0], b = w[2];
    w[0] = __fadd_rn(a, b); w[2] = __fsub_rn(a, b);
    a = w[1]; b = w[3];
    w[1] = __fadd_rn(a, b); w[3] = __fsub_rn(a, b);
  }
#pragma unroll
  for (int k = 0; k < 5; ++k) {  // h = 4 << k: partner lane differs in bit k
    const bool upper = (lane >> k) & 1;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float other = __shfl_xor_sync(0xffffffffu, w[j], 1 << k);
      w[j] = upper ? __fsub_rn(other, w[j]) : __fadd_rn(w[j], other);
    }
  }
  // norm with the fixed tree
  float acc = __fmul_rn(x[0], x[0]);
  acc = __fadd_rn(acc, __fmul_rn(x[1], x[1]));
  acc = __fadd_rn(acc, __fmul_rn(x[2], x[2]));
  acc = __fadd_rn(acc, __fmul_rn(x[3], x[3]));
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) acc = __fadd_rn(acc, __shfl_xor_sync(0xffffffffu, acc, off));
  RowOut o;
  o.p0 = f16_param(__fsqrt_rn(acc));
  o.p1 = 0;
  o.codes = 0;
  const float n = f16_to_f32(o.p0);
  if (n != 0.0f) {
    const float inv = __fdiv_rn(1.0f, n);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float u = __fmul_rn(w[j], inv);
      int c = 0;
#pragma unroll
      for (int t = 0; t < L - 1; ++t) c += (u > thr[t]) ? 1 : 0;
      o.codes |= (uint32_t)c << (8 * j);
    }
  }
  return o;
}

// Build every symbol of the K and V rows from the staged codes and OR it into the
// record image (both rows: 2 * 4 * (NG + tail) symbols, one lane per symbol).
template <int L>
__device__ __forceinline__ void pack_rows(const uint8_t* codes, uint32_t* rec, int lane) {
  using F = Fmt<L>;
  constexpr int kSymQ = F::NG + (F::R > 0 ? 1 : 0);
  constexpr int kSymRow = 4 * kSymQ;
  for (int idx = lane; idx < 2 * kSymRow; idx += 32) {
    const int row = idx / kSymRow;
    const int j = idx - row * kSymRow;
    const int q = j / kSymQ;
    const int s = j - q * kSymQ;
    const bool tail = s == F::NG;
    const int n = tail ? F::R : F::G;
    const int w = tail ? F::WT : F::W;
    const uint32_t m = tail ? F::LR : F::LG;
    const int d0 = 32 * q + (tail ? 32 - F::R : s * F::G);
    uint32_t t = 0;
    for (int k = 0; k < n; ++k) t = t * (uint32_t)L + codes[row * 128 + d0 + k];
    const uint32_t beta = ((t << w) + m - 1u) / m;
    const int pos = row * 8 * F::RB + q * F::QB + s * F::W;
    const int word = pos >> 5, sh = pos & 31;
    atomicOr(&rec[word], beta << sh);
    if (sh + w > 32) atomicOr(&rec[word + 1], beta >> (32 - sh));
  }
}

template <int BASE, int L>
__device__ void quantize_pair(const QuantArgs& a, const float kx[4], const float vx[4],
                              const int8_t* sg, const float* thr_g, uint8_t* dst,
                              uint8_t* codes, uint32_t* rec, int lane) {
  using F = Fmt<L>;
  RowOut ko, vo;
  if constexpr (BASE == SEMKV_BASE_AFFINE) {
    ko = affine_row<L>(kx);
    vo = affine_row<L>(vx);
  } else {
    float thr[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) thr[t] = t < L - 1 ? thr_g[t] : 0.0f;
    ko = tq_row<L>(kx, sg, lane, thr);
    vo = tq_row<L>(vx, sg, lane, thr);
  }
  constexpr int kRec = 2 * F::RB + (BASE == SEMKV_BASE_AFFINE ? 8 : 4);
  constexpr int kRecWords = kRec / 4;
  reinterpret_cast<uint32_t*>(codes)[lane] = ko.codes;
  reinterpret_cast<uint32_t*>(codes)[32 + lane] = vo.codes;
  if (lane < kRecWords) rec[lane] = 0u;
  __syncwarp();
  pack_rows<L>(codes, rec, lane);
  if (lane == 0) {
    if constexpr (BASE == SEMKV_BASE_AFFINE) {
      rec[(2 * F::RB) / 4] = (uint32_t)ko.p0 | ((uint32_t)ko.p1 << 16);
      rec[(2 * F::RB) / 4 + 1] = (uint32_t)vo.p0 | ((uint32_t)vo.p1 << 16);
    } else {
      rec[(2 * F::RB) / 4] = (uint32_t)ko.p0 | ((uint32_t)vo.p0 << 16);
    }
  }
  __syncwarp();
  if (lane < kRecWords) reinterpret_cast<uint32_t*>(dst)[lane] = rec[lane];
  __syncwarp();
}

template <int BASE>
__global__ void __launch_bounds__(kWarpsPerBlock * 32)
    quantize_pack_kernel(QuantArgs a) {
  __shared__ __align__(16) uint8_t codes_sm[kWarpsPerBlock][256];
  __shared__ __align__(16) uint32_t rec_sm[kWarpsPerBlock][kMaxRecWords + 1];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int64_t total = (int64_t)a.B * a.NL * a.H * a.n;
  const int64_t nwarps = (int64_t)gridDim.x * kWarpsPerBlock;
  for (int64_t task = (int64_t)blockIdx.x * kWarpsPerBlock + wib; task < total; task += nwarps) {
    const int i = (int)(task % a.n);
    int64_t r = task / a.n;
    const int h = (int)(r % a.H);
    r /= a.H;
    const int l = (int)(r % a.NL);
    const int b = (int)(r / a.NL);
    const bool hi = a.is_high[(int64_t)b * a.n + i] != 0;
    const int64_t s = (hi ? a.hi_base : a.lo_base) + a.slot[(int64_t)b * a.n + i];
    const int64_t cap = hi ? a.hi_cap : a.lo_cap;
    if (s >= cap) {  // cannot happen after the host's capacity check; never write out of range
      if (lane == 0) raise_error(a.err, kDevCapacity);
      continue;
    }
    if (l == 0 && h == 0 && lane == 0) {
      if (hi) a.hi_tok[(int64_t)b * a.hi_cap + s] = (int32_t)(a.tok_base + i);
      else a.lo_tok[(int64_t)b * a.lo_cap + s] = (int32_t)(a.tok_base + i);
    }
    const int64_t row = ((((int64_t)b * a.NL + l) * a.H + h) * a.Tsrc + i) * kHeadDim;
    float kx[4], vx[4];
    load4(a.k + row, lane, kx);
    load4(a.v + row, lane, vx);
    const int L = hi ? a.L_hi : a.L_lo;
    const int rec = record_bytes_rt(BASE, L);
    uint8_t* dst = (hi ? a.hi_pool : a.lo_pool) + ((((int64_t)b * a.NL + l) * a.H + h) * cap + s) * rec;
    const int8_t* sg = a.signs ? a.signs + ((int64_t)l * a.H + h) * kHeadDim : nullptr;
    const float* thr = hi ? a.thr_hi : a.thr_lo;
    uint8_t* cs = codes_sm[wib];
    uint32_t* rs = rec_sm[wib];
    switch (L) {
      case 2: quantize_pair<BASE, 2>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      case 3: quantize_pair<BASE, 3>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      case 4: quantize_pair<BASE, 4>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      case 5: quantize_pair<BASE, 5>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      case 6: quantize_pair<BASE, 6>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      case 7: quantize_pair<BASE, 7>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      case 8: quantize_pair<BASE, 8>(a, kx, vx, sg, thr, dst, cs, rs, lane); break;
      default: break;
    }
  }
}

}  // namespace

cudaError_t launch_quantize_pack(const QuantArgs& a, int num_sms, cudaStream_t stream) {
  const int64_t total = (int64_t)a.B * a.NL * a.H * a.n;
  if (total == 0) return cudaSuccess;
  int64_t blocks = (total + kWarpsPerBlock - 1) / kWarpsPerBlock;
  const int64_t cap_blocks = (int64_t)num_sms * 16;  // grid-stride beyond this
  if (blocks > cap_blocks) blocks = cap_blocks;
  if (a.base == SEMKV_BASE_AFFINE)
    quantize_pack_kernel<SEMKV_BASE_AFFINE><<<(unsigned)blocks, kWarpsPerBlock * 32, 0, stream>>>(a);
  else
    quantize_pack_kernel<SEMKV_BASE_TQ><<<(unsigned)blocks, kWarpsPerBlock * 32, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace semkv
