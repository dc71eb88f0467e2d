/*
 * semkv_oracle.c — the CPU oracle for the bit-exact parts of SemKV.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * statement of what the GPU library must compute.  Only tests/, the smoke check in
 * __graft_entry__ and the CPU-baseline leg of bench.py may load it.  It shares no
 * code, header, table or constant with the CUDA library: every rule below is
 * written here from the paper and from the record format stated in this file.
 *
 * What it computes
 *  - Per-row asymmetric affine quantization with fp16 scale/offset (Sec. 4.1
 *    "Memory accounting": two FP16 parameters per head-token row of dim 128).
 *  - The same affine quantizer on Hadamard-rotated rows (Sec. 4.1: rotation before
 *    the per-row quantizer): orthonormal (1/sqrt 128) H S, offset rounded down.
 *  - TurboQuant-MSE rows with a stored dense random orthogonal rotation (Sec. 4.9
 *    "random rotation"), the rotated row taken as an fp64 sum rounded to binary32.
 *  - TurboQuant-MSE rows (Sec. 4.9): random sign flip + Walsh-Hadamard rotation,
 *    row norm stored in fp16, Gaussian Lloyd-Max codebook with L levels.
 *  - Mixed-radix packing at the paper's rates (Sec. 4.1: 3 five-level codes in
 *    7 bits, 5 six-level codes in 13 bits; Table 6: 3-level at 1.600 bits).
 *  - Token-wise quantization of a whole cache into high/low pools (Eq. 7),
 *    precision broadcast over layers and KV heads (Fig. 5 caption).
 *  - Dequantization of records to exact fp64 rows (used by the fp64 attention).
 *  - The KV-norm importance indicator (Sec. 3.3: key-norm ||K_i||_2 / value-norm
 *    ||V_i||_2 of the tensor being compressed), in a fixed summation order.
 *  - Fake quantization: quantize and reconstruct to fp16 (Sec. 4.1's quality protocol).
 *
 * Floating point: build with -O2 -ffp-contract=off; every float operation below is
 * one IEEE binary32 operation rounded to nearest-even, in the order written.
 *
 * Record format (layout 1), restated here independently of the library:
 *  A 128-value row is four quarters of 32 dims.  In a quarter, codes are grouped
 *  g(L) at a time; group codes c_0..c_{g-1} (increasing dim) form
 *  t = sum_k c_k * L^(g-1-k), stored as the w-bit integer ceil(t * 2^w / L^g), w the
 *  least width with 2^w >= L^g.  The 32 mod g codes left over form one last group
 *  of that size stored the same way.  Symbols follow each other LSB first; quarter
 *  j starts at stream bit j * (bits of a quarter); stream bit i is bit i%8 of byte
 *  i/8; the row is zero-padded to whole bytes.
 *  affine record (also the rotated affine base): [K row][V row][Ks][Kz][Vs][Vz]
 *  (fp16 parameters)
 *  TQ record:     [K row][V row][Kn][Vn]
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define D 128

/* ---------------------------------------------------------------- fp16 -------- */

/* binary32 -> binary16, round to nearest even, with subnormals; overflow -> inf. */
uint16_t orc_f32_to_f16(float f) {
  uint32_t x;
  memcpy(&x, &f, 4);
  uint32_t sign = (x >> 16) & 0x8000u;
  int exp = (int)((x >> 23) & 0xFFu);
  uint32_t mant = x & 0x7FFFFFu;
  if (exp == 0xFF) return (uint16_t)(sign | 0x7C00u | (mant ? 0x200u : 0u));
  if (exp == 0) return (uint16_t)sign; /* binary32 zero/subnormal: far below 2^-25 */
  uint32_t sig = mant | 0x800000u;     /* value = sig * 2^(exp-150) */
  int e = exp - 127 + 15;              /* binary16 biased exponent if normal */
  int shift;
  uint32_t base;
  if (e >= 1) {
    shift = 13;
    base = (uint32_t)(e - 1) << 10; /* + rounded (which carries the hidden bit) */
  } else {
    shift = 13 + (1 - e);
    base = 0;
    if (shift > 24) return (uint16_t)sign; /* below half of the smallest subnormal */
  }
  uint32_t rounded = sig >> shift;
  uint32_t rem = sig & ((1u << shift) - 1u);
  uint32_t half = 1u << (shift - 1);
  if (rem > half || (rem == half && (rounded & 1u))) rounded += 1u;
  uint32_t h = base + rounded;
  if (h >= 0x7C00u) h = 0x7C00u;
  return (uint16_t)(sign | h);
}

/* binary32 -> binary16 rounded toward -infinity (the largest binary16 value not
 * above f), with subnormals; below -65504 -> -inf, above 65504 -> 65504. */
uint16_t orc_f32_to_f16_rd(float f) {
  uint32_t x;
  memcpy(&x, &f, 4);
  uint32_t sign = (x >> 16) & 0x8000u;
  int exp = (int)((x >> 23) & 0xFFu);
  uint32_t mant = x & 0x7FFFFFu;
  if (exp == 0xFF) return (uint16_t)(sign | 0x7C00u | (mant ? 0x200u : 0u));
  uint32_t mag; /* |f| truncated toward zero, as binary16 bits without the sign */
  int inexact;
  if (exp == 0) { /* binary32 zero or subnormal: below every nonzero binary16 */
    mag = 0;
    inexact = mant != 0;
  } else {
    uint32_t sig = mant | 0x800000u;
    int e = exp - 127 + 15;
    int shift;
    uint32_t base;
    if (e >= 1) {
      shift = 13;
      base = (uint32_t)(e - 1) << 10;
    } else {
      shift = 13 + (1 - e);
      base = 0;
    }
    if (shift > 24) {
      mag = 0;
      inexact = 1;
    } else {
      mag = base + (sig >> shift);
      inexact = (sig & ((1u << shift) - 1u)) != 0;
    }
  }
  if (!sign) return (uint16_t)(mag >= 0x7C00u ? 0x7BFFu : mag);
  if (inexact) mag += 1u; /* a negative value rounds away from zero */
  if (mag >= 0x7C00u) mag = 0x7C00u;
  return (uint16_t)(sign | mag);
}

float orc_f16_to_f32(uint16_t h) {
  uint32_t sign = (uint32_t)(h & 0x8000u) << 16;
  int exp = (h >> 10) & 0x1F;
  uint32_t mant = h & 0x3FFu;
  float v;
  if (exp == 0) {
    v = ldexpf((float)mant, -24);
  } else if (exp == 31) {
    v = mant ? NAN : INFINITY;
  } else {
    v = ldexpf((float)(mant | 0x400u), exp - 25);
  }
  uint32_t bits;
  memcpy(&bits, &v, 4);
  bits |= sign;
  memcpy(&v, &bits, 4);
  return v;
}

/* Scale/norm parameters are stored as fp16 rounded to nearest and then limited to
 * the largest finite fp16 (65504) so that a stored parameter is never infinite. */
static uint16_t f16_param(float f) {
  uint16_t h = orc_f32_to_f16(f);
  if ((h & 0x7FFFu) == 0x7C00u) h = (uint16_t)((h & 0x8000u) | 0x7BFFu);
  return h;
}

/* ------------------------------------------------------------- packing -------- */

/* codes per group for each level count (record format, layout 1) */
int orc_group_size(int L) {
  switch (L) {
    case 2: return 1;
    case 3: return 5;
    case 4: return 1;
    case 5: return 3;
    case 6: return 5;
    case 7: return 1;
    case 8: return 1;
    default: return 0;
  }
}

static uint64_t ipow(int b, int e) {
  uint64_t r = 1;
  for (int i = 0; i < e; i++) r *= (uint64_t)b;
  return r;
}

/* least w with 2^w >= L^n (0 when n == 0) */
static int width_for(int L, int n) {
  uint64_t m = ipow(L, n);
  int w = 0;
  while ((1ull << w) < m) w++;
  return w;
}

int orc_symbol_bits(int L) { return width_for(L, orc_group_size(L)); }
int orc_tail_codes(int L) { return 32 % orc_group_size(L); }
int orc_tail_bits(int L) { return width_for(L, orc_tail_codes(L)); }
int orc_quarter_bits(int L) {
  int g = orc_group_size(L);
  return (32 / g) * orc_symbol_bits(L) + orc_tail_bits(L);
}
int orc_row_bytes(int L) {
  if (orc_group_size(L) == 0) return 0;
  return (4 * orc_quarter_bits(L) + 7) / 8;
}
int orc_record_bytes(int base, int L) {
  int rb = orc_row_bytes(L);
  if (rb == 0) return 0;
  return 2 * rb + ((base == 1 || base == 3) ? 4 : 8);
}

static void put_bits(uint8_t* row, int pos, uint64_t val, int nbits) {
  for (int b = 0; b < nbits; b++) {
    int bit = (int)((val >> b) & 1u);
    int p = pos + b;
    row[p / 8] = (uint8_t)(row[p / 8] | (bit << (p % 8)));
  }
}

static uint64_t get_bits(const uint8_t* row, int pos, int nbits) {
  uint64_t v = 0;
  for (int b = 0; b < nbits; b++) {
    int p = pos + b;
    uint64_t bit = (uint64_t)((row[p / 8] >> (p % 8)) & 1);
    v |= bit << b;
  }
  return v;
}

/* one group of n codes (most significant first) -> stored w-bit integer */
static uint64_t encode_group(const uint8_t* c, int n, int L, int w) {
  uint64_t t = 0;
  for (int k = 0; k < n; k++) t = t * (uint64_t)L + c[k];
  uint64_t m = ipow(L, n);
  return ((t << w) + m - 1) / m; /* ceil(t * 2^w / L^n) */
}

/* stored integer -> n codes; t = floor(beta * L^n / 2^w), then base-L digits */
static void decode_group(uint64_t beta, int n, int L, int w, uint8_t* c) {
  uint64_t m = ipow(L, n);
  uint64_t t = (beta * m) >> w;
  for (int k = n - 1; k >= 0; k--) {
    c[k] = (uint8_t)(t % (uint64_t)L);
    t /= (uint64_t)L;
  }
}

/* Pack 128 codes (each < L) into a row of orc_row_bytes(L) bytes. */
void orc_pack_row(const uint8_t* codes, int L, uint8_t* row) {
  int g = orc_group_size(L), w = orc_symbol_bits(L);
  int r = orc_tail_codes(L), wt = orc_tail_bits(L);
  int qb = orc_quarter_bits(L);
  memset(row, 0, (size_t)orc_row_bytes(L));
  for (int q = 0; q < 4; q++) {
    const uint8_t* cq = codes + 32 * q;
    int pos = q * qb;
    for (int s = 0; s < 32 / g; s++) {
      put_bits(row, pos, encode_group(cq + s * g, g, L, w), w);
      pos += w;
    }
    if (r > 0) put_bits(row, pos, encode_group(cq + 32 - r, r, L, wt), wt);
  }
}

void orc_unpack_row(const uint8_t* row, int L, uint8_t* codes) {
  int g = orc_group_size(L), w = orc_symbol_bits(L);
  int r = orc_tail_codes(L), wt = orc_tail_bits(L);
  int qb = orc_quarter_bits(L);
  for (int q = 0; q < 4; q++) {
    uint8_t* cq = codes + 32 * q;
    int pos = q * qb;
    for (int s = 0; s < 32 / g; s++) {
      decode_group(get_bits(row, pos, w), g, L, w, cq + s * g);
      pos += w;
    }
    if (r > 0) decode_group(get_bits(row, pos, wt), r, L, wt, cq + 32 - r);
  }
}

/* ------------------------------------------------------------ quantizers ------ */

/* Affine row quantizer Q_b (Eq. 7 with the Sec. 4.1 per-row asymmetric quantizer):
 *   mn, mx = min, max of the row (a zero extreme taken as +0);
 *   s32 = (mx - mn) / (L - 1)
 *   s16 = fp16(s32) (limited to 65504);  z16 = fp16(mn)  (= mn, an fp16 value)
 *   codes c_j = clamp(rint((x_j - z) * fl(1/s)), 0, L-1) with z, s the fp32 values
 *   of the stored parameters; all codes 0 when s == 0. */
void orc_affine_row(const uint16_t* x, int L, uint8_t* codes, uint16_t* s_out,
                    uint16_t* z_out) {
  float xf[D];
  float mn = INFINITY, mx = -INFINITY;
  for (int j = 0; j < D; j++) {
    xf[j] = orc_f16_to_f32(x[j]);
    if (xf[j] < mn) mn = xf[j];
    if (xf[j] > mx) mx = xf[j];
  }
  /* a zero extreme is taken as +0, so the stored offset does not depend on the
   * order in which equal zeros of either sign were met */
  if (mn == 0.0f) mn = 0.0f;
  if (mx == 0.0f) mx = 0.0f;
  float range = mx - mn;
  float s32 = range / (float)(L - 1);
  uint16_t s16 = f16_param(s32);
  uint16_t z16 = orc_f32_to_f16(mn);
  float s = orc_f16_to_f32(s16);
  float z = orc_f16_to_f32(z16);
  if (s == 0.0f) {
    memset(codes, 0, D);
  } else {
    float inv = 1.0f / s;
    for (int j = 0; j < D; j++) {
      float d = xf[j] - z;
      float qv = d * inv;
      float rq = nearbyintf(qv); /* default rounding: to nearest, ties to even */
      int c = (int)rq;
      if (c < 0) c = 0;
      if (c > L - 1) c = L - 1;
      codes[j] = (uint8_t)c;
    }
  }
  *s_out = s16;
  *z_out = z16;
}

/* 1/sqrt(128) = (1/sqrt 2)/8 rounded once to binary32: the normalisation of the
 * orthonormal rotation (1/sqrt D) H S of the rotated affine base. */
static const float kInvSqrtD = 0.0883883476483184405501f;
float orc_inv_sqrt_d(void) { return kInvSqrtD; }

void orc_fwht_f32(float* w);

/* Hadamard-rotated affine row quantizer (Sec. 4.1: the per-row affine quantizer is
 * applied after a Hadamard rotation; Sec. 4.9 names the rotation family).  In binary32:
 *   u = fp32(1/sqrt 128) * FWHT(x * sign)             (orthonormal rotation of the row)
 *   z16 = fp16 rounded toward -inf of min u, limited to >= -65504, so z <= min u
 *   s16 = fp16_param((max u - z) / (L - 1))
 *   c_j = clamp(rint((u_j - z) * fl(1/s)), 0, L-1), all 0 unless s > 0.
 * Rows holding NaN or infinity are outside the supported inputs. */
void orc_affine_had_row(const uint16_t* x, const int8_t* sgn, int L, uint8_t* codes,
                        uint16_t* s_out, uint16_t* z_out) {
  float u[D];
  for (int j = 0; j < D; j++) u[j] = orc_f16_to_f32(x[j]) * (float)sgn[j];
  orc_fwht_f32(u);
  float mn = INFINITY, mx = -INFINITY;
  for (int j = 0; j < D; j++) {
    u[j] = u[j] * kInvSqrtD;
    if (u[j] < mn) mn = u[j];
    if (u[j] > mx) mx = u[j];
  }
  if (mn == 0.0f) mn = 0.0f;
  if (mx == 0.0f) mx = 0.0f;
  uint16_t z16 = orc_f32_to_f16_rd(mn);
  if (z16 == 0xFC00u) z16 = 0xFBFFu;
  float z = orc_f16_to_f32(z16);
  float s32 = (mx - z) / (float)(L - 1);
  uint16_t s16 = f16_param(s32);
  float s = orc_f16_to_f32(s16);
  if (!(s > 0.0f)) {
    memset(codes, 0, D);
  } else {
    float inv = 1.0f / s;
    for (int j = 0; j < D; j++) {
      float d = u[j] - z;
      float qv = d * inv;
      int c = (int)nearbyintf(qv);
      if (c < 0) c = 0;
      if (c > L - 1) c = L - 1;
      codes[j] = (uint8_t)c;
    }
  }
  *s_out = s16;
  *z_out = z16;
}

/* Unnormalised Walsh-Hadamard transform in binary32, butterfly stages h = 1, 2,
 * ..., 64; each butterfly maps (a, b) -> (a + b, a - b). */
void orc_fwht_f32(float* w) {
  for (int h = 1; h < D; h <<= 1) {
    for (int i = 0; i < D; i++) {
      if (i & h) continue;
      float a = w[i], b = w[i + h];
      w[i] = a + b;
      w[i + h] = a - b;
    }
  }
}

/* Row norm in binary32 with a fixed summation tree: 32 partial sums of four
 * consecutive squares each (summed in order), then five pairwise stages that add
 * partials whose indices differ in bit 4, 3, 2, 1, 0. */
float orc_row_norm(const float* x) {
  float p[32], np[32];
  for (int l = 0; l < 32; l++) {
    float acc = x[4 * l] * x[4 * l];
    for (int k = 1; k < 4; k++) {
      float sq = x[4 * l + k] * x[4 * l + k];
      acc = acc + sq;
    }
    p[l] = acc;
  }
  for (int off = 16; off >= 1; off >>= 1) {
    for (int l = 0; l < 32; l++) np[l] = p[l] + p[l ^ off];
    memcpy(p, np, sizeof(p));
  }
  return sqrtf(p[0]);
}

/* TurboQuant-MSE row quantizer (Sec. 4.9): y = x * sign; w = FWHT(y);
 * n16 = fp16(||x||); u_j = w_j * fl(1/n) ~ N(0,1); c_j = #{k : u_j > thr_k}.
 * All codes 0 when n == 0. */
void orc_tq_row(const uint16_t* x, const int8_t* sgn, int L, const float* thr,
                uint8_t* codes, uint16_t* n_out) {
  float xf[D], w[D];
  for (int j = 0; j < D; j++) {
    xf[j] = orc_f16_to_f32(x[j]);
    w[j] = xf[j] * (float)sgn[j];
  }
  orc_fwht_f32(w);
  float n32 = orc_row_norm(xf);
  uint16_t n16 = f16_param(n32);
  float n = orc_f16_to_f32(n16);
  if (n == 0.0f) {
    memset(codes, 0, D);
  } else {
    float inv = 1.0f / n;
    for (int j = 0; j < D; j++) {
      float u = w[j] * inv;
      int c = 0;
      for (int k = 0; k < L - 1; k++)
        if (u > thr[k]) c++;
      codes[j] = (uint8_t)c;
    }
  }
  *n_out = n16;
}

/* TurboQuant-MSE row with a dense random rotation (Sec. 4.9: "random rotation" before
 * the Lloyd-Max codebook; here a stored orthogonal matrix instead of the randomized
 * Hadamard transform).  rot: the fp16 matrix M ~ sqrt(128) Q (Q orthogonal), row-major
 * [128][128] fp16 bits, so that w = M x plays the part of H S x:
 *   w_i = sum_j M_ij x_j                 (exact products, summed in fp64 in index order,
 *                                        rounded once to binary32)
 *   n16 = fp16(||x||) (the fixed tree of orc_row_norm); u_i = w_i * fl(1/n);
 *   c_i = #{k : u_i > thr_k}; all codes 0 when n == 0. */
void orc_tq_dense_w(const uint16_t* x, const uint16_t* rot, float* w) {
  for (int i = 0; i < D; i++) {
    double acc = 0.0;
    for (int j = 0; j < D; j++)
      acc += (double)orc_f16_to_f32(rot[i * D + j]) * (double)orc_f16_to_f32(x[j]);
    w[i] = (float)acc;
  }
}

void orc_tq_dense_row(const uint16_t* x, const uint16_t* rot, int L, const float* thr,
                      uint8_t* codes, uint16_t* n_out) {
  float xf[D], w[D];
  for (int j = 0; j < D; j++) xf[j] = orc_f16_to_f32(x[j]);
  orc_tq_dense_w(x, rot, w);
  uint16_t n16 = f16_param(orc_row_norm(xf));
  float n = orc_f16_to_f32(n16);
  if (n == 0.0f) {
    memset(codes, 0, D);
  } else {
    float inv = 1.0f / n;
    for (int j = 0; j < D; j++) {
      float u = w[j] * inv;
      int c = 0;
      for (int k = 0; k < L - 1; k++)
        if (u > thr[k]) c++;
      codes[j] = (uint8_t)c;
    }
  }
  *n_out = n16;
}

/* --------------------------------------------------------- whole cache -------- */

/* Quantize tokens 0..n-1 of a source K/V tensor [B][NL][H][Tsrc][128] (fp16 bits)
 * into the pools (Eq. 7; the precision of token i is broadcast over every layer
 * and KV head).  Token i of sequence b goes to slot base + slot[b][i] of the high
 * pool when is_high[b][i], else of the low pool, and its token index tok_base + i
 * is written to hi_tok / lo_tok.  signs: [NL][H][128] (TQ only).  Returns 0, or -1
 * when a slot is beyond the capacity. */
int orc_quantize_tokens(int base, int Lhi, int Llo, const uint16_t* k, const uint16_t* v,
                        int B, int NL, int H, int Tsrc, int n, const uint8_t* is_high,
                        const uint32_t* slot, int64_t hi_base, int64_t lo_base,
                        int64_t tok_base, const int8_t* signs, const float* thr_hi,
                        const float* thr_lo, uint8_t* hi_pool, uint8_t* lo_pool,
                        int64_t hi_cap, int64_t lo_cap, int32_t* hi_tok, int32_t* lo_tok,
                        const uint16_t* rot) {
  int rec_hi = orc_record_bytes(base, Lhi), rec_lo = orc_record_bytes(base, Llo);
  for (int b = 0; b < B; b++) {
    for (int i = 0; i < n; i++) {
      int hi = is_high[(int64_t)b * n + i] != 0;
      int64_t s = (hi ? hi_base : lo_base) + slot[(int64_t)b * n + i];
      if (s >= (hi ? hi_cap : lo_cap)) return -1;
      if (hi)
        hi_tok[(int64_t)b * hi_cap + s] = (int32_t)(tok_base + i);
      else
        lo_tok[(int64_t)b * lo_cap + s] = (int32_t)(tok_base + i);
      int L = hi ? Lhi : Llo;
      int rec = hi ? rec_hi : rec_lo;
      int rb = orc_row_bytes(L);
      for (int l = 0; l < NL; l++) {
        for (int h = 0; h < H; h++) {
          int64_t row = ((((int64_t)b * NL + l) * H + h) * Tsrc + i) * D;
          int64_t cap = hi ? hi_cap : lo_cap;
          uint8_t* r = (hi ? hi_pool : lo_pool) + ((((int64_t)b * NL + l) * H + h) * cap + s) * rec;
          uint8_t ck[D], cv[D];
          memset(r, 0, (size_t)rec);
          if (base == 0) {
            uint16_t p[4];
            orc_affine_row(k + row, L, ck, &p[0], &p[1]);
            orc_affine_row(v + row, L, cv, &p[2], &p[3]);
            memcpy(r + 2 * rb, p, 8);
          } else if (base == 2) {
            uint16_t p[4];
            const int8_t* sg = signs + ((int64_t)l * H + h) * D;
            orc_affine_had_row(k + row, sg, L, ck, &p[0], &p[1]);
            orc_affine_had_row(v + row, sg, L, cv, &p[2], &p[3]);
            memcpy(r + 2 * rb, p, 8);
          } else if (base == 3) {
            uint16_t p[2];
            const uint16_t* m = rot + ((int64_t)l * H + h) * D * D;
            const float* thr = hi ? thr_hi : thr_lo;
            orc_tq_dense_row(k + row, m, L, thr, ck, &p[0]);
            orc_tq_dense_row(v + row, m, L, thr, cv, &p[1]);
            memcpy(r + 2 * rb, p, 4);
          } else {
            uint16_t p[2];
            const int8_t* sg = signs + ((int64_t)l * H + h) * D;
            const float* thr = hi ? thr_hi : thr_lo;
            orc_tq_row(k + row, sg, L, thr, ck, &p[0]);
            orc_tq_row(v + row, sg, L, thr, cv, &p[1]);
            memcpy(r + 2 * rb, p, 4);
          }
          orc_pack_row(ck, L, r);
          orc_pack_row(cv, L, r + rb);
        }
      }
    }
  }
  return 0;
}

/* fp64 Walsh-Hadamard transform (unnormalised), used only for dequantization. */
static void fwht_f64(double* w) {
  for (int h = 1; h < D; h <<= 1)
    for (int i = 0; i < D; i++) {
      if (i & h) continue;
      double a = w[i], b = w[i + h];
      w[i] = a + b;
      w[i + h] = a - b;
    }
}

/* Dequantize `count` records of one (b, layer, head) into exact fp64 rows.
 *  affine:         x^ = z + s * c                        (exact in fp64)
 *  rotated affine: x^ = S H (z + s * c) / sqrt(128)      (the rotation's inverse)
 *  TQ:             x^ = (n / 128) * S H cb[c]   (x = S H (H S x) / 128, H H = 128 I)
 *  dense TQ:       x^ = (n / 128) * M^T cb[c]   (M = rot, M M^T ~ 128 I) */
void orc_dequant_records(int base, int L, const uint8_t* recs, int64_t count,
                         const int8_t* sgn, const double* centroids, double* kout,
                         double* vout, const uint16_t* rot) {
  int rb = orc_row_bytes(L), rec = orc_record_bytes(base, L);
  for (int64_t i = 0; i < count; i++) {
    const uint8_t* r = recs + i * rec;
    uint8_t ck[D], cv[D];
    orc_unpack_row(r, L, ck);
    orc_unpack_row(r + rb, L, cv);
    uint16_t p[4];
    memcpy(p, r + 2 * rb, (base == 1 || base == 3) ? 4 : 8);
    double* ko = kout + i * D;
    double* vo = vout + i * D;
    if (base == 0 || base == 2) {
      double ks = orc_f16_to_f32(p[0]), kz = orc_f16_to_f32(p[1]);
      double vs = orc_f16_to_f32(p[2]), vz = orc_f16_to_f32(p[3]);
      for (int j = 0; j < D; j++) {
        ko[j] = kz + ks * ck[j];
        vo[j] = vz + vs * cv[j];
      }
      if (base == 2) {
        fwht_f64(ko);
        fwht_f64(vo);
        const double r = 1.0 / sqrt((double)D);
        for (int j = 0; j < D; j++) {
          ko[j] = ko[j] * sgn[j] * r;
          vo[j] = vo[j] * sgn[j] * r;
        }
      }
    } else if (base == 3) {
      double kn = orc_f16_to_f32(p[0]), vn = orc_f16_to_f32(p[1]);
      for (int d = 0; d < D; d++) {
        double sk = 0.0, sv = 0.0;
        for (int i2 = 0; i2 < D; i2++) {
          const double m = orc_f16_to_f32(rot[i2 * D + d]);
          sk += m * centroids[ck[i2]];
          sv += m * centroids[cv[i2]];
        }
        ko[d] = sk * kn / D;
        vo[d] = sv * vn / D;
      }
    } else {
      double kn = orc_f16_to_f32(p[0]), vn = orc_f16_to_f32(p[1]);
      for (int j = 0; j < D; j++) {
        ko[j] = centroids[ck[j]];
        vo[j] = centroids[cv[j]];
      }
      fwht_f64(ko);
      fwht_f64(vo);
      for (int j = 0; j < D; j++) {
        ko[j] = ko[j] * sgn[j] * kn / D;
        vo[j] = vo[j] * sgn[j] * vn / D;
      }
    }
  }
}

/* Element-wise conversions over arrays (for tests that sweep many values). */
/* Fake quantization (Sec. 4.1: the quality experiments quantize and dequantize and
 * compute in fp16): every row of K and V quantized at its token's precision (Eq. 7;
 * is_high NULL puts every token at Lhi, a uniform grid point) and reconstructed to
 * fp16 in binary32, in this order:
 *   affine: x^_d = fp16( z + s * c_d )                       (multiply, then add)
 *   rotated affine: y = FWHT(z + s * c);  x^_d = fp16( (sign_d y_d) * fp32(1/sqrt 128) )
 *   TQ:     y = FWHT(cb[c]) (the quantizer's butterflies);  x^_d = fp16( (sign_d y_d) * (n / 128) )
 * cent_*: fp32 centroids (TQ); x, out: [B][NL][H][T][128] fp16 bits. */
static void fake_row(int base, const uint16_t* x, int L, const int8_t* sgn, const float* cent,
                     const float* thr, uint16_t* out) {
  uint8_t c[D];
  if (base == 2) {
    uint16_t s16, z16;
    orc_affine_had_row(x, sgn, L, c, &s16, &z16);
    const float s = orc_f16_to_f32(s16), z = orc_f16_to_f32(z16);
    float y[D];
    for (int j = 0; j < D; j++) {
      const float t = s * (float)c[j];
      y[j] = z + t;
    }
    orc_fwht_f32(y);
    for (int j = 0; j < D; j++) out[j] = orc_f32_to_f16((y[j] * (float)sgn[j]) * kInvSqrtD);
  } else if (base == 0) {
    uint16_t s16, z16;
    orc_affine_row(x, L, c, &s16, &z16);
    const float s = orc_f16_to_f32(s16), z = orc_f16_to_f32(z16);
    for (int j = 0; j < D; j++) {
      const float t = s * (float)c[j];
      out[j] = orc_f32_to_f16(z + t);
    }
  } else {
    uint16_t n16;
    orc_tq_row(x, sgn, L, thr, c, &n16);
    const float nq = orc_f16_to_f32(n16) * 0.0078125f;
    float y[D];
    for (int j = 0; j < D; j++) y[j] = cent[c[j]];
    orc_fwht_f32(y);
    for (int j = 0; j < D; j++) out[j] = orc_f32_to_f16((y[j] * (float)sgn[j]) * nq);
  }
}

void orc_fake_quant(int base, int Lhi, int Llo, const uint16_t* k, const uint16_t* v, int B,
                    int NL, int H, int T, const uint8_t* is_high, const int8_t* signs,
                    const float* cent_hi, const float* thr_hi, const float* cent_lo,
                    const float* thr_lo, uint16_t* kout, uint16_t* vout) {
  for (int b = 0; b < B; b++)
    for (int l = 0; l < NL; l++)
      for (int h = 0; h < H; h++)
        for (int t = 0; t < T; t++) {
          const int hi = is_high ? is_high[(int64_t)b * T + t] != 0 : 1;
          const int64_t row = ((((int64_t)b * NL + l) * H + h) * T + t) * D;
          const int8_t* sg = signs ? signs + ((int64_t)l * H + h) * D : NULL;
          fake_row(base, k + row, hi ? Lhi : Llo, sg, hi ? cent_hi : cent_lo,
                   hi ? thr_hi : thr_lo, kout + row);
          fake_row(base, v + row, hi ? Lhi : Llo, sg, hi ? cent_hi : cent_lo,
                   hi ? thr_hi : thr_lo, vout + row);
        }
}

/* KV-norm indicator (Sec. 3.3, "KV-norm" family): token t of sequence b scores
 * ||x_{b,t}||_2 over the rows of layers [lb, le) and every KV head, x being the K or V
 * cache [B][NL][H][T][128] (fp16 bits).  Summation order, fixed so that equal inputs
 * give equal scores (and hence equal rankings) everywhere: the 128 dims of a row are
 * 32 consecutive groups of 4; group j's square sum ((x0^2 + x1^2) + x2^2) + x3^2 is
 * added to accumulator j, rows taken layer by layer, head by head; then the 32
 * accumulators are combined pairwise a[j] + a[j ^ o] for o = 16, 8, 4, 2, 1 (which
 * leaves the same total in every a[j]); the score is sqrtf of that total. */
void orc_score_kv_norm(const uint16_t* x, int B, int NL, int H, int T, int lb, int le,
                       float* scores) {
  for (int b = 0; b < B; b++) {
    for (int t = 0; t < T; t++) {
      float acc[32];
      for (int j = 0; j < 32; j++) acc[j] = 0.0f;
      for (int l = lb; l < le; l++) {
        for (int h = 0; h < H; h++) {
          const uint16_t* row = x + ((((int64_t)b * NL + l) * H + h) * T + t) * D;
          for (int j = 0; j < 32; j++) {
            float x0 = orc_f16_to_f32(row[4 * j]), x1 = orc_f16_to_f32(row[4 * j + 1]);
            float x2 = orc_f16_to_f32(row[4 * j + 2]), x3 = orc_f16_to_f32(row[4 * j + 3]);
            float sq = x0 * x0;
            sq = sq + x1 * x1;
            sq = sq + x2 * x2;
            sq = sq + x3 * x3;
            acc[j] = acc[j] + sq;
          }
        }
      }
      for (int o = 16; o >= 1; o >>= 1) {
        float nxt[32];
        for (int j = 0; j < 32; j++) nxt[j] = acc[j] + acc[j ^ o];
        for (int j = 0; j < 32; j++) acc[j] = nxt[j];
      }
      scores[(int64_t)b * T + t] = sqrtf(acc[0]);
    }
  }
}

void orc_f32_to_f16_array(const float* x, uint16_t* h, int64_t n) {
  for (int64_t i = 0; i < n; i++) h[i] = orc_f32_to_f16(x[i]);
}
void orc_f16_to_f32_array(const uint16_t* h, float* x, int64_t n) {
  for (int64_t i = 0; i < n; i++) x[i] = orc_f16_to_f32(h[i]);
}
