// score.cu — the KV-norm importance indicator (Sec. 3.3, "KV-norm" family: key-norm
// ||K_i||_2 and value-norm ||V_i||_2, the magnitude of the very tensor compressed).
//
// score[b][t] = ||x_{b,t}||_2 over the rows of layers [lb, le) and every KV head of the
// fp16 cache x [B][NL][H][T][128].  One warp per token: lane j keeps the square sum of
// dims 4j..4j+3 of every row, ((x0^2 + x1^2) + x2^2) + x3^2 added row by row (layers,
// then heads), and the 32 partials are combined with an xor butterfly (16, 8, 4, 2, 1).
// That summation order is fixed, so equal inputs give bit-identical scores -- and the
// top-r selection over them is reproducible.  Binary32, round to nearest, no
// contraction.  Bound: HBM (every row is read once).
#include "common.cuh"
#include "kernels.h"

namespace semkv {

namespace {

constexpr int kWarpsPerBlock = 8;

__global__ void __launch_bounds__(kWarpsPerBlock * 32)
    score_kv_norm_kernel(ScoreArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t total = (int64_t)a.B * a.T;
  const int64_t nw = (int64_t)gridDim.x * kWarpsPerBlock;
  for (int64_t w = (int64_t)blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5); w < total; w += nw) {
    const int b = (int)(w / a.T), t = (int)(w % a.T);
    float acc = 0.0f;
    for (int l = a.lb; l < a.le; ++l) {
      const uint16_t* lrow = a.x + (((int64_t)b * a.NL + l) * a.H * a.T + t) * kHeadDim + 4 * lane;
#pragma unroll 8
      for (int h = 0; h < a.H; ++h) {
        const uint2 u = *reinterpret_cast<const uint2*>(lrow + (int64_t)h * a.T * kHeadDim);
        const float x0 = f16_to_f32((uint16_t)(u.x & 0xFFFF)), x1 = f16_to_f32((uint16_t)(u.x >> 16));
        const float x2 = f16_to_f32((uint16_t)(u.y & 0xFFFF)), x3 = f16_to_f32((uint16_t)(u.y >> 16));
        float sq = __fmul_rn(x0, x0);
        sq = __fadd_rn(sq, __fmul_rn(x1, x1));
        sq = __fadd_rn(sq, __fmul_rn(x2, x2));
        sq = __fadd_rn(sq, __fmul_rn(x3, x3));
        acc = __fadd_rn(acc, sq);
      }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) acc = __fadd_rn(acc, __shfl_xor_sync(0xffffffffu, acc, off));
    if (lane == 0) a.scores[w] = __fsqrt_rn(acc);
  }
}

}  // namespace

cudaError_t launch_score_kv_norm(const ScoreArgs& a, int num_sms, cudaStream_t stream) {
  const int64_t total = (int64_t)a.B * a.T;
  if (total == 0) return cudaSuccess;
  int64_t blocks = (total + kWarpsPerBlock - 1) / kWarpsPerBlock;
  const int64_t cap = (int64_t)num_sms * 32;  // grid-stride beyond this
  if (blocks > cap) blocks = cap;
  score_kv_norm_kernel<<<(unsigned)blocks, kWarpsPerBlock * 32, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace semkv
