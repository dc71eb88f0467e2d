// common.cuh — record format, fp16 helpers and error plumbing shared by the
// SemKV kernels (sm_103a).
//
// Record format (layout 1): a 128-value row is four quarters of 32 dims; in a
// quarter, codes are grouped G at a time and a group (c_0 = lowest dim) is stored
// as the W-bit integer ceil(t * 2^W / L^G) with t = sum_k c_k L^(G-1-k); the 32 % G
// codes left over form one shorter group.  This "fixed-point fraction" form of the
// mixed-radix value lets a kernel peel the digits most-significant first with one
// integer multiply each: y = x * L, digit = y >> W, x = y mod 2^W.
#pragma once
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/semkv.h"

namespace semkv {

constexpr int kHeadDim = 128;

// ---------------------------------------------------------------- format ------

__host__ __device__ constexpr int group_codes(int L) {
  return L == 3 ? 5 : L == 5 ? 3 : L == 6 ? 5 : 1;  // 2, 4, 7, 8: one code per symbol
}
__host__ __device__ constexpr uint64_t ipow_c(int b, int e) {
  return e == 0 ? 1ull : (uint64_t)b * ipow_c(b, e - 1);
}
__host__ __device__ constexpr int bits_for(uint64_t m) {  // least w with 2^w >= m
  return m <= 1 ? 0 : 1 + bits_for((m + 1) / 2);
}
template <int L>
struct Fmt {
  static constexpr int G = group_codes(L);             // codes per symbol
  static constexpr int W = bits_for(ipow_c(L, G));     // bits per symbol
  static constexpr int NG = 32 / G;                    // full symbols per quarter
  static constexpr int R = 32 % G;                     // codes in the tail symbol
  static constexpr int WT = bits_for(ipow_c(L, R));    // bits of the tail symbol
  static constexpr int QB = NG * W + WT;               // bits per quarter
  static constexpr int RB = (4 * QB + 7) / 8;          // bytes per row
  static constexpr uint32_t LG = (uint32_t)ipow_c(L, G);
  static constexpr uint32_t LR = (uint32_t)ipow_c(L, R);
};

__host__ __device__ inline int row_bytes_rt(int L) {
  switch (L) {
    case 2: return Fmt<2>::RB;
    case 3: return Fmt<3>::RB;
    case 4: return Fmt<4>::RB;
    case 5: return Fmt<5>::RB;
    case 6: return Fmt<6>::RB;
    case 7: return Fmt<7>::RB;
    case 8: return Fmt<8>::RB;
    default: return 0;
  }
}
__host__ __device__ inline int record_bytes_rt(int base, int L) {
  int rb = row_bytes_rt(L);
  return rb == 0 ? 0 : 2 * rb + ((base == SEMKV_BASE_TQ || base == SEMKV_BASE_TQ_DENSE) ? 4 : 8);
}

// --------------------------------------------------------------- helpers ------

// fp16 parameter: round to nearest, then limited to the largest finite fp16 so a
// stored scale or norm is never infinite.
__device__ __forceinline__ uint16_t f16_param(float f) {
  uint16_t h = __half_as_ushort(__float2half_rn(f));
  if ((h & 0x7FFFu) == 0x7C00u) h = (uint16_t)((h & 0x8000u) | 0x7BFFu);
  return h;
}
// 1/sqrt(128) rounded to binary32: the normalisation of the rotation (1/sqrt 128) H S
constexpr float kInvSqrtD = 0x1.6a09e6p-4f;

__device__ __forceinline__ float f16_to_f32(uint16_t h) {
  return __half2float(__ushort_as_half(h));
}

// device error codes written to the cache's error word (first error wins)
enum DevError : int32_t { kDevOk = 0, kDevWaitTimeout = 1, kDevCapacity = 2 };

__device__ __forceinline__ void raise_error(int32_t* err, int32_t code) {
  if (err) atomicCAS(err, 0, code);
}

// Bounded mbarrier wait, the one every kernel uses: polls the barrier's phase at most
// `polls` times and returns false if it never completed, so a copy that never lands
// cannot hang a kernel (the caller records kDevWaitTimeout and returns).
constexpr uint32_t kWaitPolls = 1u << 22;
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint32_t polls = kWaitPolls) {
  const uint32_t addr = (uint32_t)__cvta_generic_to_shared(bar);
  for (uint32_t i = 0; i < polls; ++i) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(addr), "r"(parity)
        : "memory");
    if (ok) return true;
  }
  return false;
}

// Kernel attributes (the opt-in dynamic shared memory size) are per device: set() runs
// the first time a launcher is called on each device.
constexpr int kAttrDevices = 64;
template <typename F>
inline cudaError_t once_per_device(bool (&done)[kAttrDevices], F set) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kAttrDevices) return cudaErrorInvalidDevice;
  if (done[dev]) return cudaSuccess;
  e = set();
  if (e == cudaSuccess) done[dev] = true;
  return e;
}

// Programmatic dependent launch: the kernel may be scheduled while the previous kernel
// on the stream drains; it must call pdl_wait() before touching what that kernel (or
// anything earlier on the stream) wrote.  pdl_wait is a no-op for an ordinary launch.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Let the next kernel on the stream be scheduled now (its CTAs take SM slots as this
// kernel's CTAs leave).  It fires once every CTA of this grid has issued it or exited,
// so a dependent never holds resources that a CTA of this grid still waits for, and
// the dependent still waits (pdl_wait) before it reads what this kernel writes.
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
template <typename... Params, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

}  // namespace semkv
