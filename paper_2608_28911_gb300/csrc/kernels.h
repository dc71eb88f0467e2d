// kernels.h — launch interfaces between the C ABI (api.cu) and the kernels.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace semkv {

// Quantize tokens 0..n-1 of a source K/V tensor [B][NL][H][Tsrc][128] into the
// pools at slot base + slot[b][i] (Eq. 7).
struct QuantArgs {
  int base, L_hi, L_lo;
  const uint16_t* k;
  const uint16_t* v;
  int B, NL, H, Tsrc, n;
  const uint8_t* is_high;   // [B][n]
  const uint32_t* slot;     // [B][n]
  int64_t hi_base, lo_base, tok_base;
  const int8_t* signs;      // [NL][H][128] (TQ)
  const uint16_t* rot;      // [NL][H][128][128] fp16 (dense TQ)
  const float* thr_hi;
  const float* thr_lo;
  uint8_t* hi_pool;
  uint8_t* lo_pool;
  int64_t hi_cap, lo_cap;
  int32_t* hi_tok;
  int32_t* lo_tok;
  int32_t* err;
};
// n_hi: how many of the n tokens go to the high pool (the rest go to the low pool).
// maps_ready: the slot -> token maps of these tokens are already written (by the rank
// kernel of a block append); otherwise a scatter kernel writes them first.
cudaError_t launch_quantize_pack(const QuantArgs& a, int64_t n_hi, int num_sms,
                                 cudaStream_t stream, bool maps_ready = false);

// Top-r selection of each sequence (Eqs. 4-5).
struct RankArgs {
  const float* scores;      // [B][T] (row stride ld)
  int B, T;
  int64_t ld;
  uint32_t n_high;
  uint8_t* is_high;         // [B][T]
  uint32_t* slot;           // [B][T]
  uint32_t* rank;           // [B][T] or null
  uint32_t* ws;             // rank_workspace_words(B, T) words when rank is set
  // Optional, T <= 1024 only (a block append): when hi_tok is set the kernel also
  // writes the pools' slot -> token maps, hi_tok[b][hi_base + slot] = tok_base + i
  // (lo likewise), and raises kDevCapacity in err for a slot past the capacity.
  int32_t* hi_tok = nullptr;
  int32_t* lo_tok = nullptr;
  int64_t hi_base = 0, lo_base = 0, hi_cap = 0, lo_cap = 0, tok_base = 0;
  int32_t* err = nullptr;
};
size_t rank_workspace_words(int B, int T);
cudaError_t launch_rank_assign(const RankArgs& a, cudaStream_t stream);

// Fake quantization: quantize + reconstruct every row to fp16 (Sec. 4.1 protocol).
struct FakeArgs {
  int base, L_hi, L_lo;
  const uint16_t* k;
  const uint16_t* v;
  int B, NL, H, T;
  const uint8_t* is_high;   // [B][T] or null (every token at L_hi)
  const int8_t* signs;      // [NL][H][128] (TQ)
  const float* thr_hi;
  const float* thr_lo;
  const float* cent_hi;
  const float* cent_lo;
  uint16_t* k_out;
  uint16_t* v_out;
  int32_t* err = nullptr;   // device error word, or null (the call has none)
};
cudaError_t launch_fake_quant(const FakeArgs& a, int num_sms, cudaStream_t stream);

// KV-norm importance scores (Sec. 3.3): ||x_{b,t}|| over layers [lb, le), all heads.
struct ScoreArgs {
  const uint16_t* x;        // [B][NL][H][T][128] fp16
  int B, NL, H, T, lb, le;
  float* scores;            // [B][T]
};
cudaError_t launch_score_kv_norm(const ScoreArgs& a, int num_sms, cudaStream_t stream);

// Decode attention over one layer of the cache (split-K + combine).
struct DecodePlan {
  int tiles_hi, tiles_lo, tiles_st;     // 16-token tiles per (b, h) per source
  int splits_hi, splits_lo, splits_st;  // split plan: CTAs per (b, h) per source
  int splits;                            // split plan: partials per (b, h)
  int stride;                            // partial slots reserved per (b, h)
  // balanced plan (affine pools): one wave of CTAs over the weighted tiles of every
  // (b, h) in the order [hi | lo]; a hi tile weighs w_hi, a lo tile w_lo
  int balanced;
  int w_hi, w_lo;
  int64_t W;                             // weighted length of one (b, h)
  int64_t per;                           // weighted length per CTA
  int ctas;
  // affine pools with five- and six-level codes and GQA groups of up to 4 heads: the
  // fast kernel runs the balanced plan, with CTAs of `warps` warps (8: two per SM, 16: one)
  int fast;
  int warps;
};
struct DecodeArgs {
  int base, L_hi, L_lo;
  int B, NL, H, Hq, layer;
  const uint8_t* hi_pool;
  const uint8_t* lo_pool;
  int64_t hi_cap, lo_cap, hi_count, lo_count;
  const uint16_t* stage_k;   // [B][NL][H][block][128]
  const uint16_t* stage_v;
  int block, stage_n;
  const uint16_t* q;         // [B][Hq][128]
  float* out;                // [B][Hq][128]
  float scale_log2;          // softmax scale * log2(e)
  float* partials;           // [B][H][splits][kPartialFloats]
  const int8_t* signs;       // TQ
  const uint16_t* rot;       // dense TQ: [NL][H][128][128] fp16
  const float* cb_hi;        // TQ centroids
  const float* cb_lo;
  float* qrot;               // TQ: [B][Hq][128] rotated queries (workspace)
  int32_t* err;
  // the fp16 stage kernel runs as a programmatic dependent of the affine pool kernel:
  // it reads its inputs at once and waits for that kernel only before it exits
  int stage_overlaps_pools;
  DecodePlan plan;
};
constexpr int kPartialFloats = 16 + 8 * 128;  // m[8], l[8], o[8][128]
// max_stride: partial slots available per (b, h); a plan whose stride exceeds it
// cannot be run with that workspace
DecodePlan make_decode_plan(int base, int L_hi, int L_lo, int B, int H, int Hq, int64_t hi_count,
                            int64_t lo_count, int stage_n, int num_sms, int max_stride);
constexpr int kMaxPartialsPerPair = 65;
size_t decode_workspace_floats(int B, int H, int Hq);
cudaError_t launch_decode_attention(const DecodeArgs& a, cudaStream_t stream);

int device_sm_count();

}  // namespace semkv
