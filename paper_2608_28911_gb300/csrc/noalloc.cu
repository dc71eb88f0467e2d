// noalloc.cu — decode attention whose split-K scratch lives in a fixed device array,
// for callers that cannot allocate device memory.
//
// semkv_decode_attention needs a caller-provided workspace for its per-CTA partial
// results.  Some callers have no way to provide one: a host framework that owns all
// device memory and hands this library only the cache and the tensors of the call,
// or a serving loop that must not call cudaMalloc between steps (an allocation can
// synchronise the device and stalls every stream).  semkv_decode_attention_noalloc
// runs the same kernels with the partials in the array below instead.
#include <cstring>

#include "common.cuh"
#include "kernels.h"

// 8 MiB of split-K partials: 2016 partial results of kPartialFloats floats each.
// Every GPU that loads the library holds this array until the process exits.
static constexpr size_t kScratchFloats = (size_t)2016 * semkv::kPartialFloats;
static __device__ __align__(256) float g_decode_scratch[kScratchFloats];
// 2 MiB of rotated queries (the rotated bases): 4096 query heads of 128 floats
static constexpr size_t kQrotFloats = (size_t)4096 * 128;
static __device__ __align__(256) float g_qrot_scratch[kQrotFloats];

namespace {

constexpr int kMaxDevices = 64;
float* g_scratch_addr[kMaxDevices] = {nullptr};
float* g_qrot_addr[kMaxDevices] = {nullptr};

// The device addresses of the arrays on the current device.  In host code their names
// are only host-side stand-ins, so the addresses are looked up once per device (with
// that device current) and cached.
semkv_status scratch_address(float** out, float** qrot) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SEMKV_ECUDA;
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    void* r = nullptr;
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || !p) return SEMKV_ECUDA;
    if (cudaGetSymbolAddress(&r, g_qrot_scratch) != cudaSuccess || !r) return SEMKV_ECUDA;
    g_scratch_addr[dev] = static_cast<float*>(p);
    g_qrot_addr[dev] = static_cast<float*>(r);
  }
  *out = g_scratch_addr[dev];
  *qrot = g_qrot_addr[dev];
  return SEMKV_OK;
}

bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

}  // namespace

extern "C" semkv_status semkv_decode_attention_noalloc(const semkv_quant_desc* desc,
                                                       const semkv_cache* cache, int32_t layer,
                                                       const uint16_t* q, float* out,
                                                       float softmax_scale, void* stream) {
  using namespace semkv;
  if (!desc || !cache) return SEMKV_EINVAL;
  if (desc->head_dim != SEMKV_HEAD_DIM || cache->head_dim != SEMKV_HEAD_DIM)
    return SEMKV_EUNSUPPORTED;
  if (desc->base < SEMKV_BASE_AFFINE || desc->base > SEMKV_BASE_TQ_DENSE) return SEMKV_EUNSUPPORTED;
  if (desc->levels_hi < 2 || desc->levels_hi > SEMKV_MAX_LEVELS || desc->levels_lo < 2 ||
      desc->levels_lo > SEMKV_MAX_LEVELS)
    return SEMKV_EUNSUPPORTED;
  if (desc->base == SEMKV_BASE_TQ || desc->base == SEMKV_BASE_AFFINE_HAD) {
    if (!desc->signs) return SEMKV_EINVAL;
    if (!aligned(desc->signs, 4)) return SEMKV_EALIGN;
  }
  if (desc->base == SEMKV_BASE_TQ_DENSE) {
    if (!desc->rotation) return SEMKV_EINVAL;
    if (!aligned(desc->rotation, 16)) return SEMKV_EALIGN;
  }
  if ((desc->base == SEMKV_BASE_TQ || desc->base == SEMKV_BASE_TQ_DENSE) &&
      (!desc->centroids_hi || !desc->centroids_lo || !desc->thresholds_hi || !desc->thresholds_lo))
    return SEMKV_EINVAL;
  const semkv_cache* c = cache;
  if (c->batch < 1 || c->layers < 1 || c->kv_heads < 1 || c->q_heads < 1) return SEMKV_EINVAL;
  if (c->q_heads % c->kv_heads != 0) return SEMKV_EINVAL;
  if (c->q_heads / c->kv_heads > 8) return SEMKV_EUNSUPPORTED;
  if (c->block < 1 || c->block > 1024) return SEMKV_EINVAL;
  if (!c->hi_pool || !c->lo_pool) return SEMKV_EINVAL;
  if (!aligned(c->hi_pool, 16) || !aligned(c->lo_pool, 16)) return SEMKV_EALIGN;
  if (c->hi_cap < 0 || c->lo_cap < 0 || c->hi_cap % 16 || c->lo_cap % 16) return SEMKV_EALIGN;
  if (c->hi_count < 0 || c->lo_count < 0 || c->hi_count > c->hi_cap || c->lo_count > c->lo_cap)
    return SEMKV_EINVAL;
  if (c->stage_n < 0 || c->stage_n > c->block) return SEMKV_EINVAL;
  if (!q || !out || layer < 0 || layer >= c->layers) return SEMKV_EINVAL;
  if (!aligned(out, 16)) return SEMKV_EALIGN;
  if (c->hi_count + c->lo_count + c->stage_n == 0) return SEMKV_EINVAL;
  if (c->stage_n > 0 && (!c->stage_k || !c->stage_v)) return SEMKV_EINVAL;
  if (c->stage_n > 0 && (!aligned(c->stage_k, 8) || !aligned(c->stage_v, 8))) return SEMKV_EALIGN;

  const int sms = device_sm_count();
  if (sms <= 0) return SEMKV_ECUDA;
  // Fit the plan to the array: each (sequence, KV head) gets at most
  // cap = capacity / (batch * kv_heads) partial slots.
  const int64_t pairs = (int64_t)c->batch * c->kv_heads;
  const int64_t cap64 = (int64_t)(kScratchFloats / kPartialFloats) / pairs;
  const int cap = (int)(cap64 < kMaxPartialsPerPair ? cap64 : kMaxPartialsPerPair);
  const DecodePlan plan = make_decode_plan(desc->base, desc->levels_hi, desc->levels_lo, c->batch,
                                           c->kv_heads, c->hi_count, c->lo_count, c->stage_n,
                                           sms, cap);
  if (cap < 1 || plan.stride > cap) return SEMKV_EWORKSPACE;  // exceeds the static scratch

  const bool rotated = desc->base != SEMKV_BASE_AFFINE;
  if (rotated && (size_t)c->batch * c->q_heads * 128 > kQrotFloats) return SEMKV_EWORKSPACE;

  float* scratch = nullptr;
  float* qrot = nullptr;
  semkv_status s = scratch_address(&scratch, &qrot);
  if (s != SEMKV_OK) return s;

  DecodeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.base = desc->base;
  a.L_hi = desc->levels_hi;
  a.L_lo = desc->levels_lo;
  a.B = c->batch;
  a.NL = c->layers;
  a.H = c->kv_heads;
  a.Hq = c->q_heads;
  a.layer = layer;
  a.hi_pool = c->hi_pool;
  a.lo_pool = c->lo_pool;
  a.hi_cap = c->hi_cap;
  a.lo_cap = c->lo_cap;
  a.hi_count = c->hi_count;
  a.lo_count = c->lo_count;
  a.stage_k = c->stage_k;
  a.stage_v = c->stage_v;
  a.block = c->block;
  a.stage_n = c->stage_n;
  a.q = q;
  a.out = out;
  a.scale_log2 = softmax_scale * 1.4426950408889634f;
  a.partials = scratch;  // fully overwritten by each call: nothing needs clearing
  a.signs = desc->signs;
  a.rot = desc->rotation;
  a.cb_hi = desc->centroids_hi;
  a.cb_lo = desc->centroids_lo;
  a.qrot = rotated ? qrot : nullptr;
  a.err = c->dev_error;
  a.plan = plan;
  return launch_decode_attention(a, (cudaStream_t)stream) == cudaSuccess ? SEMKV_OK : SEMKV_ECUDA;
}
