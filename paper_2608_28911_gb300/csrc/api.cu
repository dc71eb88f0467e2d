// api.cu — the C ABI declared in include/semkv.h: argument checks, capacity
// accounting and kernel launches.  No entry point allocates, frees or synchronises.
#include <cmath>
#include <cstdint>
#include <cstring>

#include "checks.h"
#include "common.cuh"
#include "kernels.h"

using namespace semkv;

namespace {

semkv_status from_cuda(cudaError_t e) { return e == cudaSuccess ? SEMKV_OK : SEMKV_ECUDA; }

}  // namespace

namespace semkv {
int device_sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64 && cached[dev]) return cached[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64) cached[dev] = n;
  return n;
}
}  // namespace semkv

extern "C" {

size_t semkv_row_bytes(int32_t levels) { return level_ok(levels) ? (size_t)row_bytes_rt(levels) : 0; }

size_t semkv_record_bytes(int32_t base, int32_t levels) {
  if (!level_ok(levels) || base < SEMKV_BASE_AFFINE || base > SEMKV_BASE_TQ_DENSE) return 0;
  return (size_t)record_bytes_rt(base, levels);
}

uint32_t semkv_high_count_floor(uint32_t T, uint32_t r_num, uint32_t r_den) {
  if (r_den == 0) return 0;
  uint64_t k = (uint64_t)T * r_num / r_den;
  return (uint32_t)(k > T ? T : k);
}

uint32_t semkv_block_high_count(uint32_t n, uint32_t r_num, uint32_t r_den) {
  if (r_den == 0) return 0;
  uint64_t k = (2ull * r_num * n + r_den) / (2ull * r_den);
  return (uint32_t)(k > n ? n : k);
}

const char* semkv_status_string(semkv_status s) {
  switch (s) {
    case SEMKV_OK: return "ok";
    case SEMKV_EINVAL: return "invalid argument";
    case SEMKV_EALIGN: return "misaligned pointer or capacity";
    case SEMKV_ECAPACITY: return "pool or staging capacity exceeded";
    case SEMKV_EUNSUPPORTED: return "unsupported level count, base or shape";
    case SEMKV_ECUDA: return "CUDA error";
    case SEMKV_EWORKSPACE: return "workspace missing or too small";
  }
  return "unknown status";
}

// Lloyd-Max quantizer of N(0,1) (Sec. 4.9): Lloyd iteration in fp64 until the
// centroids stop moving; thresholds are centroid midpoints.
semkv_status semkv_lloyd_max_gaussian(int32_t levels, float* centroids, float* thresholds) {
  const TraceRange trace("semkv_lloyd_max_gaussian");
  if (levels < 2 || levels > 64 || !centroids || !thresholds) return SEMKV_EINVAL;
  const int L = levels;
  double c[64], nc[64], t[65];
  for (int i = 0; i < L; ++i) c[i] = 2.0 * (-1.0 + 2.0 * (i + 0.5) / L);
  const double inv_sqrt2 = 1.0 / std::sqrt(2.0), inv_sqrt2pi = 1.0 / std::sqrt(2.0 * M_PI);
  auto pdf = [&](double x) { return std::isinf(x) ? 0.0 : std::exp(-0.5 * x * x) * inv_sqrt2pi; };
  auto cdf = [&](double x) {
    if (x == INFINITY) return 1.0;
    if (x == -INFINITY) return 0.0;
    return 0.5 * std::erfc(-x * inv_sqrt2);
  };
  for (int iter = 0; iter < 200000; ++iter) {
    t[0] = -INFINITY;
    t[L] = INFINITY;
    for (int i = 1; i < L; ++i) t[i] = 0.5 * (c[i - 1] + c[i]);
    double delta = 0.0;
    for (int i = 0; i < L; ++i) {
      nc[i] = (pdf(t[i]) - pdf(t[i + 1])) / (cdf(t[i + 1]) - cdf(t[i]));
      delta = std::fmax(delta, std::fabs(nc[i] - c[i]));
    }
    std::memcpy(c, nc, sizeof(double) * L);
    if (delta < 1e-15) break;
  }
  // the codebook of a symmetric density is symmetric: make it so exactly
  for (int i = 0; i < L; ++i) nc[i] = 0.5 * (c[i] - c[L - 1 - i]);
  std::memcpy(c, nc, sizeof(double) * L);
  for (int i = 0; i < L; ++i) centroids[i] = (float)c[i];
  for (int i = 0; i + 1 < L; ++i) thresholds[i] = (float)(0.5 * (c[i] + c[i + 1]));
  return SEMKV_OK;
}

size_t semkv_rank_workspace_bytes(int32_t batch, int32_t T, int32_t want_rank) {
  if (!want_rank || batch < 1 || T < 1) return 0;
  return rank_workspace_words(batch, T) * sizeof(uint32_t);
}

semkv_status semkv_rank_assign(const float* scores, int32_t batch, int32_t T, uint32_t n_high,
                               uint8_t* is_high, uint32_t* slot, uint32_t* rank, void* ws,
                               size_t ws_bytes, void* stream) {
  const TraceRange trace("semkv_rank_assign");
  if (!scores || !is_high || !slot || batch < 0 || T < 1 || T > (1 << 24)) return SEMKV_EINVAL;
  if (n_high > (uint32_t)T) return SEMKV_EINVAL;
  if (rank) {
    if (!ws || ws_bytes < semkv_rank_workspace_bytes(batch, T, 1)) return SEMKV_EWORKSPACE;
    if (!aligned(ws, 4)) return SEMKV_EALIGN;
  }
  RankArgs a;
  a.rank = rank;
  a.ws = static_cast<uint32_t*>(ws);
  a.scores = scores;
  a.B = batch;
  a.T = T;
  a.ld = T;
  a.n_high = n_high;
  a.is_high = is_high;
  a.slot = slot;
  return from_cuda(launch_rank_assign(a, (cudaStream_t)stream));
}

semkv_status semkv_fake_quant(const semkv_quant_desc* desc, const uint16_t* k, const uint16_t* v,
                              int32_t batch, int32_t layers, int32_t kv_heads, int32_t T,
                              const uint8_t* is_high, uint16_t* k_out, uint16_t* v_out,
                              void* stream) {
  const TraceRange trace("semkv_fake_quant");
  semkv_status s = check_desc(desc);
  if (s != SEMKV_OK) return s;
  if (desc->base == SEMKV_BASE_TQ_DENSE) return SEMKV_EUNSUPPORTED;
  if (!k || !v || !k_out || !v_out || batch < 1 || layers < 1 || kv_heads < 1 || T < 1)
    return SEMKV_EINVAL;
  if (!aligned(k, 16) || !aligned(v, 16) || !aligned(k_out, 16) || !aligned(v_out, 16))
    return SEMKV_EALIGN;
  FakeArgs a;
  a.base = desc->base;
  a.L_hi = desc->levels_hi;
  a.L_lo = desc->levels_lo;
  a.k = k;
  a.v = v;
  a.B = batch;
  a.NL = layers;
  a.H = kv_heads;
  a.T = T;
  a.is_high = is_high;
  a.signs = desc->signs;
  a.thr_hi = desc->thresholds_hi;
  a.thr_lo = desc->thresholds_lo;
  a.cent_hi = desc->centroids_hi;
  a.cent_lo = desc->centroids_lo;
  a.k_out = k_out;
  a.v_out = v_out;
  return from_cuda(launch_fake_quant(a, device_sm_count(), (cudaStream_t)stream));
}

semkv_status semkv_score_kv_norm(const uint16_t* x, int32_t batch, int32_t layers,
                                 int32_t kv_heads, int32_t T, int32_t layer_begin,
                                 int32_t layer_end, float* scores, void* stream) {
  const TraceRange trace("semkv_score_kv_norm");
  if (!x || !scores || batch < 1 || layers < 1 || kv_heads < 1 || T < 1) return SEMKV_EINVAL;
  if (layer_begin < 0 || layer_end > layers || layer_begin >= layer_end) return SEMKV_EINVAL;
  if (!aligned(x, 8) || !aligned(scores, 4)) return SEMKV_EALIGN;
  ScoreArgs a;
  a.x = x;
  a.B = batch;
  a.NL = layers;
  a.H = kv_heads;
  a.T = T;
  a.lb = layer_begin;
  a.le = layer_end;
  a.scores = scores;
  return from_cuda(launch_score_kv_norm(a, device_sm_count(), (cudaStream_t)stream));
}

semkv_status semkv_quantize_pack(const semkv_quant_desc* desc, const uint16_t* k,
                                 const uint16_t* v, int32_t T, const uint8_t* is_high,
                                 const uint32_t* slot, uint32_t n_high, semkv_cache* cache,
                                 void* stream) {
  const TraceRange trace("semkv_quantize_pack");
  semkv_status s = check_desc(desc);
  if (s != SEMKV_OK) return s;
  s = check_cache(cache);
  if (s != SEMKV_OK) return s;
  if (!k || !v || !is_high || !slot || T < 1) return SEMKV_EINVAL;
  if (!aligned(k, 8) || !aligned(v, 8)) return SEMKV_EALIGN;
  if (desc->base != SEMKV_BASE_AFFINE && (!aligned(k, 16) || !aligned(v, 16)))
    return SEMKV_EALIGN;  // the rows arrive by async or tensor copies in 16-byte units
  if (n_high > (uint32_t)T) return SEMKV_EINVAL;
  if ((int64_t)n_high > cache->hi_cap || (int64_t)(T - n_high) > cache->lo_cap)
    return SEMKV_ECAPACITY;
  QuantArgs a;
  a.base = desc->base;
  a.L_hi = desc->levels_hi;
  a.L_lo = desc->levels_lo;
  a.k = k;
  a.v = v;
  a.B = cache->batch;
  a.NL = cache->layers;
  a.H = cache->kv_heads;
  a.Tsrc = T;
  a.n = T;
  a.is_high = is_high;
  a.slot = slot;
  a.hi_base = 0;
  a.lo_base = 0;
  a.tok_base = 0;
  a.signs = desc->signs;
  a.rot = desc->rotation;
  a.thr_hi = desc->thresholds_hi;
  a.thr_lo = desc->thresholds_lo;
  a.hi_pool = cache->hi_pool;
  a.lo_pool = cache->lo_pool;
  a.hi_cap = cache->hi_cap;
  a.lo_cap = cache->lo_cap;
  a.hi_tok = cache->hi_tok;
  a.lo_tok = cache->lo_tok;
  a.err = cache->dev_error;
  s = from_cuda(launch_quantize_pack(a, n_high, device_sm_count(), (cudaStream_t)stream));
  if (s != SEMKV_OK) return s;
  cache->hi_count = n_high;
  cache->lo_count = T - (int64_t)n_high;
  cache->n_tokens = T;
  cache->stage_n = 0;
  return SEMKV_OK;
}

semkv_status semkv_append_block(const semkv_quant_desc* desc, semkv_cache* cache,
                                uint32_t r_num, uint32_t r_den, void* stream) {
  const TraceRange trace("semkv_append_block");
  semkv_status s = check_desc(desc);
  if (s != SEMKV_OK) return s;
  s = check_cache(cache);
  if (s != SEMKV_OK) return s;
  if (r_den == 0 || r_num > r_den) return SEMKV_EINVAL;
  const int n = cache->stage_n;
  if (n == 0) return SEMKV_OK;
  if (!cache->stage_k || !cache->stage_v || !cache->stage_score || !cache->blk_is_high ||
      !cache->blk_slot)
    return SEMKV_EINVAL;
  if (!aligned(cache->stage_k, 8) || !aligned(cache->stage_v, 8)) return SEMKV_EALIGN;
  if (desc->base != SEMKV_BASE_AFFINE &&
      (!aligned(cache->stage_k, 16) || !aligned(cache->stage_v, 16)))
    return SEMKV_EALIGN;
  const uint32_t n_high = semkv_block_high_count((uint32_t)n, r_num, r_den);
  if (cache->hi_count + n_high > cache->hi_cap || cache->lo_count + (n - n_high) > cache->lo_cap)
    return SEMKV_ECAPACITY;
  RankArgs r;
  r.scores = cache->stage_score;
  r.B = cache->batch;
  r.T = n;
  r.ld = cache->block;
  r.n_high = n_high;
  r.is_high = cache->blk_is_high;
  r.slot = cache->blk_slot;
  r.rank = nullptr;
  r.ws = nullptr;
  // a block of at most 1024 tokens is ranked by one single-pass kernel, which then
  // writes the slot -> token maps too (no separate scatter launch)
  const bool maps_in_rank = n <= 1024 && desc->base != SEMKV_BASE_TQ_DENSE;
  if (maps_in_rank) {
    r.hi_tok = cache->hi_tok;
    r.lo_tok = cache->lo_tok;
    r.hi_base = cache->hi_count;
    r.lo_base = cache->lo_count;
    r.hi_cap = cache->hi_cap;
    r.lo_cap = cache->lo_cap;
    r.tok_base = cache->n_tokens;
    r.err = cache->dev_error;
  }
  s = from_cuda(launch_rank_assign(r, (cudaStream_t)stream));
  if (s != SEMKV_OK) return s;
  QuantArgs a;
  a.base = desc->base;
  a.L_hi = desc->levels_hi;
  a.L_lo = desc->levels_lo;
  a.k = cache->stage_k;
  a.v = cache->stage_v;
  a.B = cache->batch;
  a.NL = cache->layers;
  a.H = cache->kv_heads;
  a.Tsrc = cache->block;
  a.n = n;
  a.is_high = cache->blk_is_high;
  a.slot = cache->blk_slot;
  a.hi_base = cache->hi_count;
  a.lo_base = cache->lo_count;
  a.tok_base = cache->n_tokens;
  a.signs = desc->signs;
  a.rot = desc->rotation;
  a.thr_hi = desc->thresholds_hi;
  a.thr_lo = desc->thresholds_lo;
  a.hi_pool = cache->hi_pool;
  a.lo_pool = cache->lo_pool;
  a.hi_cap = cache->hi_cap;
  a.lo_cap = cache->lo_cap;
  a.hi_tok = cache->hi_tok;
  a.lo_tok = cache->lo_tok;
  a.err = cache->dev_error;
  s = from_cuda(launch_quantize_pack(a, n_high, device_sm_count(), (cudaStream_t)stream,
                                     maps_in_rank));
  if (s != SEMKV_OK) return s;
  cache->hi_count += n_high;
  cache->lo_count += n - (int64_t)n_high;
  cache->n_tokens += n;
  cache->stage_n = 0;
  return SEMKV_OK;
}

size_t semkv_decode_workspace_bytes(const semkv_cache* cache) {
  if (!cache || cache->batch < 1 || cache->kv_heads < 1) return 0;
  return decode_workspace_floats(cache->batch, cache->kv_heads, cache->q_heads) * sizeof(float);
}

semkv_status semkv_decode_attention(const semkv_quant_desc* desc, const semkv_cache* cache,
                                    int32_t layer, const uint16_t* q, float* out,
                                    float softmax_scale, void* ws, size_t ws_bytes,
                                    void* stream) {
  const TraceRange trace("semkv_decode_attention");
  semkv_status s = check_decode(desc, cache, layer, q, out);
  if (s != SEMKV_OK) return s;
  if (!ws || !aligned(ws, 16)) return SEMKV_EWORKSPACE;
  if (ws_bytes < semkv_decode_workspace_bytes(cache)) return SEMKV_EWORKSPACE;
  const int sms = device_sm_count();
  if (sms <= 0) return SEMKV_ECUDA;
  DecodeArgs a = decode_args(desc, cache, layer, q, out, softmax_scale);
  a.partials = reinterpret_cast<float*>(ws);
  // rotated queries (TQ and rotated affine bases) after the split-K partials
  // in the workspace
  a.qrot = a.partials + (decode_workspace_floats(a.B, a.H, a.Hq) - (size_t)a.B * a.Hq * 128);
  a.plan = make_decode_plan(a.base, a.L_hi, a.L_lo, a.B, a.H, a.Hq, a.hi_count, a.lo_count, a.stage_n,
                            sms, kMaxPartialsPerPair);
  return from_cuda(launch_decode_attention(a, (cudaStream_t)stream));
}

}  // extern "C"
