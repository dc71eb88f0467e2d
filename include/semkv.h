/*
 * semkv.h — C ABI of the SemKV packed mixed-precision KV cache (sm_103a).
 *
 * SemKV keeps every token of the KV cache (Eqs. 8-9) and gives each token one of
 * two adjacent fractional precisions: the top-r fraction by importance score gets
 * b_high, the rest b_low (Eqs. 4-5).  A "fractional" precision is an integer level
 * count L with log2(L) bits (Sec. 4.1: 2.585 = log2 6, 2.322 = log2 5).  Codes are
 * stored by mixed-radix packing (Sec. 4.1: 3 five-level codes in 7 bits, 5 six-level
 * codes in 13 bits) with per-row fp16 metadata (two parameters per 128-value row
 * for the affine base; one norm per row for the TurboQuant-MSE base, Sec. 4.9).
 * Generated tokens are staged at fp16 and quantized a block at a time, exactly
 * round(r*B) of each block at b_high (Sec. 3.7, Algorithm 2).
 *
 * Conventions shared by every entry point
 *  - The caller owns every buffer.  No entry point allocates, frees or synchronises;
 *    all device work is enqueued on the caller's stream `stream` (a cudaStream_t
 *    passed as void*; NULL = legacy default stream).
 *  - Pointers documented as "device" must be device (or managed) memory.
 *  - Host-checkable errors (NULL pointers, bad sizes, misalignment, unsupported
 *    level counts, capacity overflow) return an error status before anything is
 *    launched.  A failed launch returns SEMKV_ECUDA.  Kernels never trap: an
 *    anomaly seen on the device (e.g. a bulk-copy wait that timed out) is written
 *    to cache->dev_error (when given) and the host reads it when it chooses.
 *  - fp16 tensors are passed as uint16_t bit patterns (IEEE binary16).
 *  - head_dim is 128 in this version (the shape of Llama-3.1-8B / Mistral-7B KV).
 *
 * Record format (layout 1).  For level count L a 128-value row is four quarters
 * of 32 consecutive dims.  Inside a quarter the codes are grouped g(L) at a time;
 * a group's codes c_0..c_{g-1} (c_0 = lowest dim) form t = sum_k c_k L^(g-1-k) and
 * are stored as the w(L)-bit integer ceil(t * 2^w / L^g); the 32 mod g codes left at
 * the end of the quarter form one shorter group stored the same way in
 * ceil(log2 L^(32 mod g)) bits.  Quarters are concatenated least-significant-bit
 * first (stream bit i is bit i%8 of byte i/8); unused bits are zero.
 *      L : g  w   bits/quarter  row bytes RB(L)
 *      2 : 1  1        32            16
 *      3 : 5  8        52            26
 *      4 : 1  2        64            32
 *      5 : 3  7        75            38
 *      6 : 5 13        84            42
 *      7 : 1  3        96            48
 *      8 : 1  3        96            48
 *  affine record = [K row RB][V row RB][Ks f16][Kz f16][Vs f16][Vz f16]  (2RB+8 B)
 *  TQ record     = [K row RB][V row RB][Kn f16][Vn f16]                   (2RB+4 B)
 *  Pools are [batch][layers][kv_heads][cap][record]; slot s of the high pool of
 *  sequence b holds the s-th high-precision token of b in token order.
 */
#ifndef SEMKV_H_
#define SEMKV_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SEMKV_OK = 0,
  SEMKV_EINVAL = 1,         /* NULL pointer, bad size or inconsistent arguments   */
  SEMKV_EALIGN = 2,         /* a pointer or capacity violates an alignment rule    */
  SEMKV_ECAPACITY = 3,      /* a pool or the staging buffer would overflow         */
  SEMKV_EUNSUPPORTED = 4,   /* level count / base / head_dim not supported         */
  SEMKV_ECUDA = 5,          /* a CUDA launch or query failed                       */
  SEMKV_EWORKSPACE = 6      /* workspace NULL or smaller than the size query says  */
} semkv_status;

enum { SEMKV_BASE_AFFINE = 0, SEMKV_BASE_TQ = 1, SEMKV_BASE_AFFINE_HAD = 2,
       SEMKV_BASE_TQ_DENSE = 3 };
enum { SEMKV_HEAD_DIM = 128, SEMKV_MAX_LEVELS = 8 };

/* Quantizer description (host struct; the pointers inside are device pointers).
 * base AFFINE: per-row asymmetric min/max quantizer with fp16 scale and offset
 *   (Sec. 4.1 "two FP16 parameters (offset and scale) per head-token row").
 * base AFFINE_HAD: the same affine quantizer applied to the Hadamard-rotated row
 *   (Sec. 4.1: rows are rotated before quantization), in binary32:
 *     u = fp32(1/sqrt 128) * FWHT(x * sign)   (orthonormal (1/sqrt 128) H S; butterfly
 *                                              stages 1, 2, ..., 64, each (a+b, a-b))
 *     z = fp16 of min u rounded toward -infinity (limited to >= -65504), so z <= min u
 *     s = fp16((max u - z) / (L - 1)), rounded to nearest and limited to 65504
 *     c_j = clamp(rint((u_j - z) * fl(1/s)), 0, L - 1); all 0 unless s > 0.
 *   Records as AFFINE; decoding rotates each query once and the output back once.
 *   Needs signs.  Rows holding NaN or infinity are outside the supported inputs.
 * base TQ: TurboQuant-MSE (Sec. 4.9): sign flip + unnormalised Walsh-Hadamard
 *   transform of the row, divided by the row's fp16 norm, then a Gaussian Lloyd-Max
 *   scalar codebook with L levels (thresholds strictly-greater: ties go low).
 * base TQ_DENSE: TurboQuant-MSE with a dense random rotation (Sec. 4.9 "random
 *   rotation"): w = M x with M the stored fp16 matrix ~ sqrt(128) Q (Q orthogonal) in
 *   place of H S x; the rest as TQ (fp16 norm, u = w * fl(1/n), codebook).  w is formed
 *   on the tensor cores (exact fp16 products, fp32 accumulation), so a code can differ
 *   from the exactly rounded product's where u lies within rounding of a threshold.
 *   Records as TQ; rows dequantize to (n/128) M^T cb[c].  Needs rotation + codebooks.
 * levels_hi / levels_lo: L for b_high / b_low, each in 2..8; equal = uniform. */
typedef struct {
  int32_t base;
  int32_t levels_hi, levels_lo;
  int32_t head_dim;                 /* must be 128 */
  const int8_t* signs;              /* TQ, AFFINE_HAD: device [layers][kv_heads][128]
                                       of +-1, 4-byte aligned                       */
  const float* centroids_hi;        /* TQ, TQ_DENSE: device [levels_hi] ascending   */
  const float* thresholds_hi;       /* TQ: device [levels_hi-1] ascending           */
  const float* centroids_lo;        /* TQ: device [levels_lo]                       */
  const float* thresholds_lo;       /* TQ: device [levels_lo-1]                     */
  const uint16_t* rotation;         /* TQ_DENSE: device fp16 [layers][kv_heads][128][128]
                                       row-major (w_i = sum_j M_ij x_j), 16-byte
                                       aligned; NULL for the other bases             */
} semkv_quant_desc;

/* One mixed-precision cache Ĉ_KV (Algorithm 1 output, extended by Algorithm 2).
 * Every sequence of the batch has the same prompt length and the same r, so the
 * pool counts are equal across the batch and kept on the host.  Fields marked
 * (lib) are updated by the library; the caller initialises them to 0. */
typedef struct {
  int32_t batch, layers, kv_heads, q_heads, head_dim;  /* q_heads % kv_heads == 0 */
  int32_t block;               /* B of Algorithm 2 (1..1024)                       */
  uint8_t* hi_pool;            /* device [batch][layers][kv_heads][hi_cap][rec_hi], 16-B aligned */
  uint8_t* lo_pool;            /* device [batch][layers][kv_heads][lo_cap][rec_lo], 16-B aligned */
  int64_t hi_cap, lo_cap;      /* slots per (b, layer, head); multiples of 16, at
                                  most 2^30 (else SEMKV_EUNSUPPORTED)               */
  int32_t* hi_tok;             /* device [batch][hi_cap]: token index of each slot */
  int32_t* lo_tok;             /* device [batch][lo_cap]                            */
  int64_t hi_count, lo_count;  /* (lib) slots in use, same for every sequence      */
  int64_t n_tokens;            /* (lib) tokens quantized so far (prompt + blocks)  */
  uint16_t* stage_k;           /* device fp16 [batch][layers][kv_heads][block][128] */
  uint16_t* stage_v;           /* device fp16, same shape                           */
  float* stage_score;          /* device [batch][block]: scores of staged tokens    */
  int32_t stage_n;             /* tokens currently staged (caller writes the data
                                  at index stage_n, then increments it)            */
  uint8_t* blk_is_high;        /* device scratch [batch][block]                     */
  uint32_t* blk_slot;          /* device scratch [batch][block]                     */
  int32_t* dev_error;          /* device int32 error word (may be NULL)             */
} semkv_cache;

/* Bytes of one packed 128-value row with L levels (RB(L) above); 0 if unsupported. */
size_t semkv_row_bytes(int32_t levels);
/* Bytes of one record of the given base and level count; 0 if unsupported. */
size_t semkv_record_bytes(int32_t base, int32_t levels);

/* K = floor(r*T) with r = r_num/r_den, in 64-bit integers (Eq. 4). */
uint32_t semkv_high_count_floor(uint32_t T, uint32_t r_num, uint32_t r_den);
/* round(r*n), nearest integer with halves rounded up, in integers (Algorithm 2:
 * exactly round(rB) per block; the flush of a partial block uses n = |S|). */
uint32_t semkv_block_high_count(uint32_t n, uint32_t r_num, uint32_t r_den);

/* Gaussian N(0,1) Lloyd-Max codebook with L levels (Sec. 4.9: "Gaussian-optimal
 * Lloyd-Max codebook", extended to any integer L).  Computed on the host in fp64
 * by Lloyd iteration to convergence, then made exactly symmetric (c_l = -c_{L-1-l});
 * centroids[L] = fp32(c_l), thresholds[L-1] = fp32((c_l + c_{l+1})/2) taken in fp64.
 * Host pointers. */
semkv_status semkv_lloyd_max_gaussian(int32_t levels, float* centroids, float* thresholds);

/* Top-r selection, Eqs. 4-5 / Algorithm 1.  For each sequence b of `batch`:
 * H = the n_high tokens with the largest score, ties broken by lower token index
 * (NaN ranks below every number, -0 equals +0).  Outputs (device):
 *   is_high[b][i] = 1 if i in H else 0            (u8  [batch][T])
 *   slot[b][i]    = #{j < i : is_high[b][j] == is_high[b][i]}   (u32 [batch][T])
 *   rank[b][i]    = position of i in the (score desc, index asc) order, 0-based
 *                   (u32 [batch][T]; may be NULL).
 * scores: device f32 [batch][T].  ws/ws_bytes: device workspace of at least
 * semkv_rank_workspace_bytes(batch, T, rank != NULL) bytes, 4-byte aligned, owned by
 * the caller: 16 * batch * T bytes when ranks are wanted (keys and indices of a
 * stable radix sort, double-buffered), else 0 and ws may be NULL.
 * Errors: SEMKV_EINVAL (null pointers, T outside 1..2^24, n_high > T),
 * SEMKV_EWORKSPACE (rank set and ws missing or too small), SEMKV_EALIGN. */
size_t semkv_rank_workspace_bytes(int32_t batch, int32_t T, int32_t want_rank);
semkv_status semkv_rank_assign(const float* scores, int32_t batch, int32_t T,
                               uint32_t n_high, uint8_t* is_high, uint32_t* slot,
                               uint32_t* rank, void* ws, size_t ws_bytes, void* stream);

/* Fake quantization (Sec. 4.1: the quality experiments quantize, dequantize and compute
 * in fp16).  Every row of K and V is quantized with the same arithmetic as
 * semkv_quantize_pack at its token's level count (levels_hi where is_high[b][t], else
 * levels_lo; is_high NULL puts every token at levels_hi, a uniform grid point) and
 * reconstructed to fp16, in binary32 in this order:
 *   affine: out_d = fp16( z + s * c_d )
 *   TQ:     y = unnormalised FWHT(cb[c]) (stages 1..64);  out_d = fp16( (sign_d * y_d) * (n/128) )
 * k, v, k_out, v_out: device fp16 [batch][layers][kv_heads][T][128], 16-byte aligned
 * (rows move in 16-byte chunks), caller-owned (outputs may not alias inputs); is_high:
 * device u8 [batch][T] or NULL.
 * Errors: SEMKV_EINVAL, SEMKV_EALIGN, SEMKV_EUNSUPPORTED (level counts, base).  There is
 * no device error word: the rotated bases move rows with bulk copies whose waits are
 * bounded, and a copy that never completed would stop its CTA, leaving the rows it had
 * not yet written unchanged. */
semkv_status semkv_fake_quant(const semkv_quant_desc* desc, const uint16_t* k, const uint16_t* v,
                              int32_t batch, int32_t layers, int32_t kv_heads, int32_t T,
                              const uint8_t* is_high, uint16_t* k_out, uint16_t* v_out,
                              void* stream);

/* KV-norm importance indicator (Sec. 3.3, "KV-norm" family: key-norm ||K_i||_2 and
 * value-norm ||V_i||_2, the magnitude of the tensor being compressed; Sec. 4.5 finds
 * value-norm the cheapest indicator profiled).  Writes
 *   scores[b][t] = || x[b][l][h][t][:] ||_2 over l in [layer_begin, layer_end) and all h
 * (a layer range restricts the score to the last m layers, as Eq. 3 does).
 * x: device fp16 [batch][layers][kv_heads][T][128] (pass the K cache for key-norm, the V
 * cache for value-norm), 8-byte aligned; scores: device f32 [batch][T], 4-byte aligned,
 * both caller-owned.  The summation order is fixed (per dim group of 4, row by row, then
 * a pairwise tree over the 32 groups), so equal inputs give bit-identical scores.
 * The scores feed semkv_rank_assign directly (only their ranking matters).
 * Errors: SEMKV_EINVAL (null pointers, empty or inverted ranges), SEMKV_EALIGN. */
semkv_status semkv_score_kv_norm(const uint16_t* x, int32_t batch, int32_t layers,
                                 int32_t kv_heads, int32_t T, int32_t layer_begin,
                                 int32_t layer_end, float* scores, void* stream);

/* Token-wise quantization, Eq. 7 / Algorithm 1: quantize every row of the prompt
 * K/V with Q_{b_i} and write token i's record (for every layer and KV head) to
 * slot[b][i] of the high pool if is_high[b][i] else of the low pool; writes
 * hi_tok/lo_tok[b][slot] = i.  k, v: device fp16 [batch][layers][kv_heads][T][128],
 * 8-byte aligned for AFFINE, 16-byte aligned for the other bases (their rows arrive by
 * bulk or tensor copies in 16-byte units); the same holds for the stage buffers in
 * semkv_append_block.  is_high, slot: as produced by semkv_rank_assign for this T.  n_high: the number
 * of high tokens per sequence (used for the capacity check and the counts).
 * Sets cache->hi_count = n_high, lo_count = T - n_high, n_tokens = T and resets
 * stage_n to 0 (a prompt replaces whatever the cache held). */
semkv_status semkv_quantize_pack(const semkv_quant_desc* desc, const uint16_t* k,
                                 const uint16_t* v, int32_t T, const uint8_t* is_high,
                                 const uint32_t* slot, uint32_t n_high, semkv_cache* cache,
                                 void* stream);

/* Block-exact deferred quantization, Sec. 3.7 / Algorithm 2: quantizes the n =
 * cache->stage_n staged tokens, exactly semkv_block_high_count(n, r_num, r_den) of
 * them (the highest staged scores, ties to the earlier token) at levels_hi, the rest
 * at levels_lo, appends them to the pools after the current counts, records their
 * token indices n_tokens + j, then advances hi_count / lo_count / n_tokens and sets
 * stage_n = 0.  Call it when stage_n == block (a full block) or at the end of a
 * turn with 0 < stage_n < block (the residual flush).  stage_n == 0 is a no-op. */
semkv_status semkv_append_block(const semkv_quant_desc* desc, semkv_cache* cache,
                                uint32_t r_num, uint32_t r_den, void* stream);

/* Single-query decode attention over the whole cache of one layer ("use Ĉ_KV for
 * decoding", Algorithm 1; the staged fp16 tokens take part, Algorithm 2):
 *   out[b][qh] = sum_i softmax_i(scale * q[b][qh] . k^_i) * v^_i
 * over i = all hi_count + lo_count quantized tokens and the stage_n staged tokens
 * of sequence b, with KV head h = qh / (q_heads / kv_heads) and k^, v^ the
 * dequantized rows (affine: z + s*c; TQ: n/128 * S H cb[c]).  Computed split-K over
 * the tokens with an online softmax and a final combine.
 * q: device fp16 [batch][q_heads][128]; out: device f32 [batch][q_heads][128].
 * ws: device workspace of semkv_decode_workspace_bytes(cache) bytes, 16-B aligned.
 * Accuracy: against fp64 attention over the same dequantized cache, max-abs error
 * <= 2e-3 and relative L2 <= 1e-3 for values of magnitude below 64; binary32 carries
 * relative error, so for larger values the absolute error grows as up to 8e-6 *
 * max|v^| (all of fp16's range, including subnormal steps, is supported). */
size_t semkv_decode_workspace_bytes(const semkv_cache* cache);
semkv_status semkv_decode_attention(const semkv_quant_desc* desc, const semkv_cache* cache,
                                    int32_t layer, const uint16_t* q, float* out,
                                    float softmax_scale, void* ws, size_t ws_bytes,
                                    void* stream);

/* Decode attention for callers that cannot allocate device memory.  The paper has
 * no counterpart: this is a deployment variant of semkv_decode_attention.
 * Who needs it: a caller whose host framework owns all device memory and gives this
 * library only the cache and the tensors of the call, or a serving loop that must
 * not call cudaMalloc between decode steps (an allocation can synchronise the device).
 * It computes what semkv_decode_attention computes, for every base, with the same
 * kernels, but keeps the split-K partial results in a static device array of 8 MiB
 * (2016 partials) that the library owns, instead of a caller workspace; it calls no
 * cudaMalloc, cudaFree or allocating routine.  Every GPU that loads the library
 * holds that array until the process exits.
 *  - Set-up: the first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress) with that device current and caches it; make that first
 *    call before any stream capture.  The cached address is not refreshed after
 *    cudaDeviceReset.  Host threads may make their first calls concurrently.
 *  - Limit: each (sequence, KV head) pair gets cap = min(65, 2016 / (batch *
 *    kv_heads)) partial slots, and the split count is reduced to fit them.  The
 *    affine bases (balanced plan) need cap >= 3 + stage, i.e. batch * kv_heads <= 672,
 *    or <= 504 with staged tokens; the TQ bases (split plan) need cap >= one per
 *    non-empty pool + stage, i.e. batch * kv_heads * (pools + stage) <= 2016.
 *    Larger requests return SEMKV_EWORKSPACE before anything is launched.  The dense-
 *    rotation base (TQ_DENSE) also keeps its rotated queries in a second static array
 *    of 4096 query heads (batch * q_heads beyond it: SEMKV_EWORKSPACE).
 *  - All calls share the array, which keeps the last call's contents (each call
 *    overwrites every partial it reads, so nothing needs clearing).  Calls whose
 *    kernels overlap on the GPU (e.g. on two streams, or two host threads) race on
 *    it: serialise them.
 * Arguments and errors otherwise as semkv_decode_attention (no ws / ws_bytes). */
semkv_status semkv_decode_attention_noalloc(const semkv_quant_desc* desc,
                                            const semkv_cache* cache, int32_t layer,
                                            const uint16_t* q, float* out, float softmax_scale,
                                            void* stream);

/* Failure-detection check (not a step of the paper's method).  Every kernel that
 * waits on a bulk copy uses one bounded mbarrier wait: after a fixed number of polls
 * (2^22) it gives up, writes 1 (a wait that timed out) into the device error word and
 * the kernel returns, so a lost copy never hangs the GPU and the context stays usable.
 * This entry point runs that same wait in one CTA of 4 warps on a barrier that nothing
 * arrives on, with the caller's poll limit `polls` (1 .. 2^22): each warp's wait runs
 * out and writes 1 into *dev_error (device int32, 4-byte aligned; the first error
 * written wins, so clear it first to see this one).  It lets a test make a wait run
 * out on purpose without faulting or hanging anything.  Stream-ordered; errors:
 * SEMKV_EINVAL (NULL dev_error, polls out of range), SEMKV_EALIGN, SEMKV_ECUDA. */
semkv_status semkv_debug_wait_timeout(int32_t* dev_error, uint32_t polls, void* stream);

/* Human-readable name of a status code (static string). */
const char* semkv_status_string(semkv_status s);

#ifdef __cplusplus
}
#endif
#endif /* SEMKV_H_ */
