// checks.h — host-side argument checks shared by the C-ABI entry points (api.cu,
// noalloc.cu), so that every entry point accepts exactly the same descriptors and
// caches, and the decode arguments are filled in one place.
#pragma once
#include <cstdint>
#include <cstring>

#include <nvtx3/nvToolsExt.h>

#include "../../include/semkv.h"
#include "kernels.h"

namespace semkv {

// An NVTX range named after the C-ABI call, open for the call's host-side extent (its
// checks and launches), so a profiler's timeline shows which call enqueued which kernels.
// Without a profiler attached the push and pop do nothing.
struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};

inline bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

inline bool level_ok(int L) { return L >= 2 && L <= SEMKV_MAX_LEVELS; }

inline semkv_status check_desc(const semkv_quant_desc* d) {
  if (!d) return SEMKV_EINVAL;
  if (d->head_dim != SEMKV_HEAD_DIM) return SEMKV_EUNSUPPORTED;
  if (d->base != SEMKV_BASE_AFFINE && d->base != SEMKV_BASE_TQ &&
      d->base != SEMKV_BASE_AFFINE_HAD && d->base != SEMKV_BASE_TQ_DENSE)
    return SEMKV_EUNSUPPORTED;
  if (!level_ok(d->levels_hi) || !level_ok(d->levels_lo)) return SEMKV_EUNSUPPORTED;
  if (d->base == SEMKV_BASE_AFFINE_HAD) {
    if (!d->signs) return SEMKV_EINVAL;
    if (!aligned(d->signs, 4)) return SEMKV_EALIGN;
  }
  if (d->base == SEMKV_BASE_TQ_DENSE) {
    if (!d->rotation || !d->thresholds_hi || !d->thresholds_lo || !d->centroids_hi ||
        !d->centroids_lo)
      return SEMKV_EINVAL;
    if (!aligned(d->rotation, 16)) return SEMKV_EALIGN;
  }
  if (d->base == SEMKV_BASE_TQ) {
    if (!d->signs || !d->thresholds_hi || !d->thresholds_lo || !d->centroids_hi ||
        !d->centroids_lo)
      return SEMKV_EINVAL;
    if (!aligned(d->signs, 4)) return SEMKV_EALIGN;
  }
  return SEMKV_OK;
}

inline semkv_status check_cache(const semkv_cache* c) {
  if (!c) return SEMKV_EINVAL;
  if (c->batch < 1 || c->layers < 1 || c->kv_heads < 1 || c->q_heads < 1) return SEMKV_EINVAL;
  if (c->head_dim != SEMKV_HEAD_DIM) return SEMKV_EUNSUPPORTED;
  if (c->q_heads % c->kv_heads != 0) return SEMKV_EINVAL;
  if (c->q_heads / c->kv_heads > 8) return SEMKV_EUNSUPPORTED;
  if (c->block < 1 || c->block > 1024) return SEMKV_EINVAL;
  if (!c->hi_pool || !c->lo_pool || !c->hi_tok || !c->lo_tok) return SEMKV_EINVAL;
  if (!aligned(c->hi_pool, 16) || !aligned(c->lo_pool, 16)) return SEMKV_EALIGN;
  if (c->hi_cap < 0 || c->lo_cap < 0 || c->hi_cap % 16 || c->lo_cap % 16) return SEMKV_EALIGN;
  // slot and tile indices are 32-bit inside the kernels
  if (c->hi_cap > (int64_t)1 << 30 || c->lo_cap > (int64_t)1 << 30) return SEMKV_EUNSUPPORTED;
  if (c->hi_count < 0 || c->lo_count < 0 || c->hi_count > c->hi_cap || c->lo_count > c->lo_cap)
    return SEMKV_EINVAL;
  if (c->stage_n < 0 || c->stage_n > c->block) return SEMKV_EINVAL;
  return SEMKV_OK;
}

// Everything a decode call checks before it plans, whatever holds its partials.
inline semkv_status check_decode(const semkv_quant_desc* desc, const semkv_cache* cache,
                                 int32_t layer, const uint16_t* q, const float* out) {
  semkv_status s = check_desc(desc);
  if (s != SEMKV_OK) return s;
  s = check_cache(cache);
  if (s != SEMKV_OK) return s;
  if (!q || !out || layer < 0 || layer >= cache->layers) return SEMKV_EINVAL;
  if (!aligned(out, 16)) return SEMKV_EALIGN;
  if (cache->hi_count + cache->lo_count + cache->stage_n == 0) return SEMKV_EINVAL;
  if (cache->stage_n > 0 && (!cache->stage_k || !cache->stage_v)) return SEMKV_EINVAL;
  if (cache->stage_n > 0 && (!aligned(cache->stage_k, 8) || !aligned(cache->stage_v, 8)))
    return SEMKV_EALIGN;
  return SEMKV_OK;
}

// The launch arguments of a decode call; the caller sets partials, qrot and plan.
inline DecodeArgs decode_args(const semkv_quant_desc* desc, const semkv_cache* cache,
                              int32_t layer, const uint16_t* q, float* out,
                              float softmax_scale) {
  DecodeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.base = desc->base;
  a.L_hi = desc->levels_hi;
  a.L_lo = desc->levels_lo;
  a.B = cache->batch;
  a.NL = cache->layers;
  a.H = cache->kv_heads;
  a.Hq = cache->q_heads;
  a.layer = layer;
  a.hi_pool = cache->hi_pool;
  a.lo_pool = cache->lo_pool;
  a.hi_cap = cache->hi_cap;
  a.lo_cap = cache->lo_cap;
  a.hi_count = cache->hi_count;
  a.lo_count = cache->lo_count;
  a.stage_k = cache->stage_k;
  a.stage_v = cache->stage_v;
  a.block = cache->block;
  a.stage_n = cache->stage_n;
  a.q = q;
  a.out = out;
  a.scale_log2 = softmax_scale * 1.4426950408889634f;
  a.signs = desc->signs;
  a.rot = desc->rotation;
  a.cb_hi = desc->centroids_hi;
  a.cb_lo = desc->centroids_lo;
  a.err = cache->dev_error;
  return a;
}

}  // namespace semkv
