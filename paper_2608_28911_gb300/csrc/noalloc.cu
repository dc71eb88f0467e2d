// noalloc.cu — decode attention whose split-K scratch lives in a fixed device array,
// for callers that cannot allocate device memory.
//
// semkv_decode_attention needs a caller-provided workspace for its per-CTA partial
// results.  Some callers have no way to provide one: a host framework that owns all
// device memory and hands this library only the cache and the tensors of the call,
// or a serving loop that must not call cudaMalloc between steps (an allocation can
// synchronise the device and stalls every stream).  semkv_decode_attention_noalloc
// runs the same kernels with the partials in the array below instead.
#include <atomic>

#include "checks.h"
#include "common.cuh"
#include "kernels.h"

// 8 MiB of split-K partials: 2016 partial results of kPartialFloats floats each.
// Every GPU that loads the library holds this array until the process exits.
static constexpr size_t kScratchPartials = 2016;
static constexpr size_t kScratchFloats = kScratchPartials * semkv::kPartialFloats;
static __device__ __align__(256) float g_decode_scratch[kScratchFloats];
// 2 MiB of rotated queries (the dense-rotation base): 4096 query heads of 128 floats
static constexpr size_t kQrotFloats = (size_t)4096 * 128;
static __device__ __align__(256) float g_qrot_scratch[kQrotFloats];

namespace {

constexpr int kMaxDevices = 64;
// Device addresses of the two arrays, per device.  Host threads may make their first
// call on a device at the same time: each may look the addresses up (the lookups agree),
// and the atomics make the cached values safe to share.
std::atomic<float*> g_scratch_addr[kMaxDevices];
std::atomic<float*> g_qrot_addr[kMaxDevices];

// The device addresses of the arrays on the current device.  In host code their names
// are only host-side stand-ins, so the addresses are looked up once per device (with
// that device current) and cached.  The cache is not refreshed after cudaDeviceReset.
semkv_status scratch_address(float** out, float** qrot) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SEMKV_ECUDA;
  float* s = g_scratch_addr[dev].load(std::memory_order_acquire);
  float* r = g_qrot_addr[dev].load(std::memory_order_acquire);
  if (!s || !r) {
    void* p = nullptr;
    void* q = nullptr;
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || !p) return SEMKV_ECUDA;
    if (cudaGetSymbolAddress(&q, g_qrot_scratch) != cudaSuccess || !q) return SEMKV_ECUDA;
    s = static_cast<float*>(p);
    r = static_cast<float*>(q);
    g_scratch_addr[dev].store(s, std::memory_order_release);
    g_qrot_addr[dev].store(r, std::memory_order_release);
  }
  *out = s;
  *qrot = r;
  return SEMKV_OK;
}

}  // namespace

extern "C" semkv_status semkv_decode_attention_noalloc(const semkv_quant_desc* desc,
                                                       const semkv_cache* cache, int32_t layer,
                                                       const uint16_t* q, float* out,
                                                       float softmax_scale, void* stream) {
  const semkv::TraceRange trace("semkv_decode_attention_noalloc");
  using namespace semkv;
  semkv_status st = check_decode(desc, cache, layer, q, out);
  if (st != SEMKV_OK) return st;
  const semkv_cache* c = cache;
  const int sms = device_sm_count();
  if (sms <= 0) return SEMKV_ECUDA;
  // Fit the plan to the array: each (sequence, KV head) gets at most
  // cap = capacity / (batch * kv_heads) partial slots.
  const int64_t pairs = (int64_t)c->batch * c->kv_heads;
  const int64_t cap64 = (int64_t)kScratchPartials / pairs;
  const int cap = (int)(cap64 < kMaxPartialsPerPair ? cap64 : kMaxPartialsPerPair);
  const DecodePlan plan = make_decode_plan(desc->base, desc->levels_hi, desc->levels_lo, c->batch,
                                           c->kv_heads, c->q_heads, c->hi_count, c->lo_count, c->stage_n,
                                           sms, cap);
  if (cap < 1 || plan.stride > cap) return SEMKV_EWORKSPACE;  // exceeds the static scratch

  // only the dense rotation keeps its rotated queries in memory (the Walsh-Hadamard bases
  // rotate them inside the kernels)
  const bool rotated = desc->base == SEMKV_BASE_TQ_DENSE;
  if (rotated && (size_t)c->batch * c->q_heads * 128 > kQrotFloats) return SEMKV_EWORKSPACE;

  float* scratch = nullptr;
  float* qrot = nullptr;
  st = scratch_address(&scratch, &qrot);
  if (st != SEMKV_OK) return st;

  DecodeArgs a = decode_args(desc, cache, layer, q, out, softmax_scale);
  a.partials = scratch;  // fully overwritten by each call: nothing needs clearing
  a.qrot = rotated ? qrot : nullptr;
  a.plan = plan;
  return launch_decode_attention(a, (cudaStream_t)stream) == cudaSuccess ? SEMKV_OK : SEMKV_ECUDA;
}
