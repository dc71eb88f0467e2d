// rank.cu — top-r selection of Eqs. 4-5 / Algorithm 1 (and of each block in
// Algorithm 2): is_high marks the n_high largest scores of a sequence, ties going to
// the lower token index; slot is each token's position in its pool.
//
// One 1024-thread CTA per sequence.  Sequences of at most 1024 tokens (the blocks of
// Algorithm 2) take a single pass: each thread counts the keys ahead of its own.
// Longer ones: scores become order-preserving 32-bit keys
// (NaN -> 0, below every number; -0 -> +0), kept in shared memory for sequences of up
// to 40960 tokens.  A 4-pass MSB-first radix select over 8-bit digits finds theta,
// the key of the n_high-th largest score, and `need`, how many keys equal to theta
// are taken (the earliest ones).  One sweep with a block
// scan of packed (greater, equal) counts then gives, for token i,
//   high(i)        = key_i > theta  or  (key_i == theta and eq_before(i) < need)
//   high_before(i) = gt_before(i) + min(eq_before(i), need)
//   slot(i)        = high(i) ? high_before(i) : i - high_before(i).
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace semkv {

namespace {

constexpr int kThreads = 1024;
constexpr int kItems = 4;

__device__ __forceinline__ uint32_t order_key(float f) {
  if (f != f) return 0u;  // NaN ranks below every number
  uint32_t b = __float_as_uint(f);
  if (f == 0.0f) b = 0u;  // -0 == +0
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// exclusive scan of a 64-bit value over the CTA; returns the prefix, sets *total
__device__ __forceinline__ uint64_t block_exclusive_scan(uint64_t v, uint64_t* warp_sums,
                                                         uint64_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint64_t x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    uint64_t y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint64_t w = warp_sums[lane];
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      uint64_t y = __shfl_up_sync(0xffffffffu, w, off);
      if (lane >= off) w += y;
    }
    warp_sums[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  const uint64_t before_warp = warp == 0 ? 0ull : warp_sums[warp - 1];
  *total = warp_sums[31];
  const uint64_t r = before_warp + x - v;
  __syncthreads();  // warp_sums is reused by the next call
  return r;
}

// Short sequences (T <= 1024, e.g. a block of Algorithm 2): thread i counts the keys
// that precede token i in the (key desc, index asc) order -- its rank -- by comparing
// against all T keys in shared memory; is_high = rank < n_high, and the slot is the
// count of earlier tokens of the same class (a block scan of the flags).
__global__ void __launch_bounds__(kThreads) rank_small_kernel(RankArgs a) {
  __shared__ uint32_t keys[kThreads];
  __shared__ uint32_t warp_hi[32];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = a.T;
  pdl_wait();  // the scores (and the maps) belong to earlier work on the stream
  pdl_trigger();
  const float* s = a.scores + (int64_t)b * a.ld;
  const uint32_t mine = tid < T ? order_key(s[tid]) : 0u;
  keys[tid] = mine;
  __syncthreads();
  uint32_t rank = 0;
  if (tid < T) {
#pragma unroll 8
    for (int j = 0; j < T; ++j) {
      const uint32_t kj = keys[j];
      rank += (kj > mine || (kj == mine && j < tid)) ? 1u : 0u;
    }
  }
  const bool hi = tid < T && rank < a.n_high;
  // exclusive count of earlier high tokens
  const uint32_t bal = __ballot_sync(0xffffffffu, hi);
  if (lane == 0) warp_hi[warp] = __popc(bal);
  __syncthreads();
  uint32_t before = __popc(bal & ((1u << lane) - 1u));
  for (int w = 0; w < warp; ++w) before += warp_hi[w];
  if (tid < T) {
    const uint32_t slot = hi ? before : (uint32_t)tid - before;
    a.is_high[(int64_t)b * T + tid] = hi ? 1 : 0;
    a.slot[(int64_t)b * T + tid] = slot;
    if (a.hi_tok != nullptr) {
      // a block append: the pools' slot -> token maps as well
      const int64_t s = (hi ? a.hi_base : a.lo_base) + slot;
      const int64_t cap = hi ? a.hi_cap : a.lo_cap;
      if (s >= cap)  // cannot happen after the host's capacity check
        raise_error(a.err, kDevCapacity);
      else
        (hi ? a.hi_tok : a.lo_tok)[(int64_t)b * cap + s] = (int32_t)(a.tok_base + tid);
    }
  }
}

// keys of sequences up to this length are kept in shared memory across the passes
constexpr uint32_t kSmemKeys = 40960;
constexpr int kSelItems = 8;  // keys per thread per loop trip (independent loads)

// warp 0: the bin holding the k-th largest key among the 256 counts, and how many
// larger keys the bins above it hold (a suffix scan, 8 bins per lane)
__device__ __forceinline__ void select_bin(const uint32_t* hist, uint32_t k, uint32_t* bin_out,
                                           uint32_t* above_out) {
  const int lane = threadIdx.x & 31;
  // lane l owns bins 255 - 8l down to 248 - 8l (descending key order)
  uint32_t c[8], sum = 0;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    c[e] = hist[255 - 8 * lane - e];
    sum += c[e];
  }
  uint32_t incl = sum;  // inclusive scan over lanes of the per-lane sums
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += y;
  }
  const uint32_t excl = incl - sum;  // keys in bins above this lane's
  const bool mine = excl < k && incl >= k;
  if (mine) {
    uint32_t cum = excl;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      if (cum + c[e] >= k) {
        *bin_out = 255u - 8u * lane - (uint32_t)e;
        *above_out = cum;
        break;
      }
      cum += c[e];
    }
  }
}

__global__ void __launch_bounds__(kThreads) rank_assign_kernel(RankArgs a) {
  extern __shared__ uint32_t skeys[];  // the sequence's keys when T <= kSmemKeys
  __shared__ uint32_t hist[256];
  __shared__ uint32_t whist[kThreads / 32][256];  // one histogram per warp: no contention
  __shared__ uint32_t sel_bin, sel_above;
  __shared__ uint64_t warp_sums[32];
  const int b = blockIdx.x;
  const float* s = a.scores + (int64_t)b * a.ld;
  uint8_t* is_high = a.is_high + (int64_t)b * a.T;
  uint32_t* slot = a.slot + (int64_t)b * a.T;
  const uint32_t T = (uint32_t)a.T;
  const int tid = threadIdx.x;

  if (a.n_high == 0 || a.n_high == T) {
    const uint8_t all = a.n_high == T ? 1 : 0;
    for (uint32_t i = tid; i < T; i += kThreads) {
      is_high[i] = all;
      slot[i] = i;
    }
    return;
  }
  const bool in_smem = T <= kSmemKeys;
  if (in_smem) {
    for (uint32_t i = tid; i < T; i += kThreads) skeys[i] = order_key(s[i]);
    __syncthreads();
  }

  // ---- radix select: theta = key of the n_high-th largest, need = ties taken
  uint32_t prefix = 0, mask = 0, k = a.n_high;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    uint32_t* wh = whist[tid >> 5];
    for (int i = tid; i < (kThreads / 32) * 256; i += kThreads) (&whist[0][0])[i] = 0;
    __syncthreads();
    for (uint32_t i0 = 0; i0 < T; i0 += kThreads * kSelItems) {
      uint32_t key[kSelItems];
#pragma unroll
      for (int j = 0; j < kSelItems; ++j) {
        const uint32_t i = i0 + j * kThreads + tid;
        key[j] = i < T ? (in_smem ? skeys[i] : order_key(s[i])) : 0u;
      }
#pragma unroll
      for (int j = 0; j < kSelItems; ++j) {
        const uint32_t i = i0 + j * kThreads + tid;
        const bool cand = i < T && (key[j] & mask) == prefix;
        const uint32_t bin = (key[j] >> shift) & 0xFFu;
        // the warp's own histogram: shared-memory atomics without cross-warp contention
        if (cand) atomicAdd(&wh[bin], 1u);
      }
    }
    __syncthreads();
    for (int i = tid; i < 256; i += kThreads) {
      uint32_t c = 0;
#pragma unroll 8
      for (int w = 0; w < kThreads / 32; ++w) c += whist[w][i];
      hist[i] = c;
    }
    __syncthreads();
    if (tid < 32) select_bin(hist, k, &sel_bin, &sel_above);
    __syncthreads();
    prefix |= sel_bin << shift;
    k -= sel_above;
    mask |= 0xFFu << shift;
    __syncthreads();
  }
  const uint32_t theta = prefix, need = k;

  // ---- one sweep: flags and slots from a scan of packed (eq << 32 | gt) counts
  uint64_t run = 0;  // totals of all earlier chunks
  for (uint32_t c0 = 0; c0 < T; c0 += kThreads * kItems) {
    uint32_t keys[kItems];
    uint64_t local = 0;
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      const uint32_t i = c0 + tid * kItems + j;
      keys[j] = i < T ? (in_smem ? skeys[i] : order_key(s[i])) : 0u;
      if (i < T) local += (keys[j] > theta ? 1ull : 0ull) | ((keys[j] == theta ? 1ull : 0ull) << 32);
    }
    uint64_t total;
    uint64_t before = run + block_exclusive_scan(local, warp_sums, &total);
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      const uint32_t i = c0 + tid * kItems + j;
      if (i >= T) break;
      const uint32_t gt_b = (uint32_t)(before & 0xFFFFFFFFu);
      const uint32_t eq_b = (uint32_t)(before >> 32);
      const bool gt = keys[j] > theta, eq = keys[j] == theta;
      const bool hi = gt || (eq && eq_b < need);
      const uint32_t hib = gt_b + min(eq_b, need);
      is_high[i] = hi ? 1 : 0;
      slot[i] = hi ? hib : i - hib;
      before += (gt ? 1ull : 0ull) | ((eq ? 1ull : 0ull) << 32);
    }
    run += total;
  }
}

// ---- long sequences on a thread-block cluster -----------------------------------
// The same selection and sweep with one sequence spread over a cluster of kCluster
// CTAs: CTA r keeps the keys of tokens [r chunk, (r+1) chunk) in its shared memory and
// counts them into its own histograms; each pass every CTA sums the cluster's 256-bin
// histograms through distributed shared memory and takes the same bin (the choice is
// deterministic); for the sweep each CTA adds the (greater, equal) totals of the CTAs
// before it, so every token sees the counts of all earlier tokens of the sequence.
constexpr int kCluster = 8;

__global__ void __cluster_dims__(kCluster, 1, 1) __launch_bounds__(kThreads)
    rank_cluster_kernel(RankArgs a) {
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  extern __shared__ uint32_t ckeys[];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t whist[kThreads / 32][256];
  __shared__ uint32_t sel_bin, sel_above;
  __shared__ uint64_t warp_sums[32];
  __shared__ uint64_t chunk_total;
  const int rank_in = (int)cluster.block_rank();
  const int b = blockIdx.x / kCluster;
  const float* s = a.scores + (int64_t)b * a.ld;
  uint8_t* is_high = a.is_high + (int64_t)b * a.T;
  uint32_t* slot = a.slot + (int64_t)b * a.T;
  const uint32_t T = (uint32_t)a.T;
  const uint32_t chunk = (T + kCluster - 1) / kCluster;
  const uint32_t c_begin = min(T, (uint32_t)rank_in * chunk);
  const uint32_t c_end = min(T, c_begin + chunk);
  const uint32_t nloc = c_end - c_begin;
  const int tid = threadIdx.x;

  if (a.n_high == 0 || a.n_high == T) {  // the same branch in every CTA of the cluster
    const uint8_t all = a.n_high == T ? 1 : 0;
    for (uint32_t i = c_begin + tid; i < c_end; i += kThreads) {
      is_high[i] = all;
      slot[i] = i;
    }
    return;
  }
  for (uint32_t i = tid; i < nloc; i += kThreads) ckeys[i] = order_key(s[c_begin + i]);

  uint32_t prefix = 0, mask = 0, k = a.n_high;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    uint32_t* wh = whist[tid >> 5];
    for (int i = tid; i < (kThreads / 32) * 256; i += kThreads) (&whist[0][0])[i] = 0;
    __syncthreads();
    for (uint32_t i0 = 0; i0 < nloc; i0 += kThreads * kSelItems) {
      uint32_t key[kSelItems];
#pragma unroll
      for (int j = 0; j < kSelItems; ++j) {
        const uint32_t i = i0 + j * kThreads + tid;
        key[j] = i < nloc ? ckeys[i] : 0u;
      }
#pragma unroll
      for (int j = 0; j < kSelItems; ++j) {
        const uint32_t i = i0 + j * kThreads + tid;
        if (i < nloc && (key[j] & mask) == prefix) atomicAdd(&wh[(key[j] >> shift) & 0xFFu], 1u);
      }
    }
    __syncthreads();
    for (int i = tid; i < 256; i += kThreads) {
      uint32_t c = 0;
#pragma unroll 8
      for (int w = 0; w < kThreads / 32; ++w) c += whist[w][i];
      hist[i] = c;
    }
    cluster.sync();  // every CTA's histogram is complete
    if (tid < 32) {
      // the cluster's counts, summed in CTA order (each CTA reaches the same totals)
      uint32_t tot[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) tot[e] = 0;
      for (int r = 0; r < kCluster; ++r) {
        const uint32_t* rh = cluster.map_shared_rank(hist, r);
#pragma unroll
        for (int e = 0; e < 8; ++e) tot[e] += rh[255 - 8 * tid - e];
      }
      // select_bin over the summed counts (lane l holds bins 255 - 8l .. 248 - 8l)
      uint32_t sum = 0;
#pragma unroll
      for (int e = 0; e < 8; ++e) sum += tot[e];
      uint32_t incl = sum;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
        if (tid >= off) incl += y;
      }
      const uint32_t excl = incl - sum;
      if (excl < k && incl >= k) {
        uint32_t cum = excl;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          if (cum + tot[e] >= k) {
            sel_bin = 255u - 8u * tid - (uint32_t)e;
            sel_above = cum;
            break;
          }
          cum += tot[e];
        }
      }
    }
    cluster.sync();  // every CTA has read the others' histograms: they may be reset
    prefix |= sel_bin << shift;
    k -= sel_above;
    mask |= 0xFFu << shift;
  }
  const uint32_t theta = prefix, need = k;

  // ---- this CTA's (greater, equal) totals, then the totals of the CTAs before it
  {
    uint64_t local = 0;
    for (uint32_t i = tid; i < nloc; i += kThreads)
      local += (ckeys[i] > theta ? 1ull : 0ull) | ((ckeys[i] == theta ? 1ull : 0ull) << 32);
    uint64_t total;
    (void)block_exclusive_scan(local, warp_sums, &total);
    if (tid == 0) chunk_total = total;
  }
  cluster.sync();
  uint64_t run = 0;
  for (int r = 0; r < rank_in; ++r) run += *cluster.map_shared_rank(&chunk_total, r);
  cluster.sync();  // no CTA leaves while another still reads its shared memory

  for (uint32_t c0 = 0; c0 < nloc; c0 += kThreads * kItems) {
    uint32_t keys[kItems];
    uint64_t local = 0;
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      const uint32_t i = c0 + tid * kItems + j;
      keys[j] = i < nloc ? ckeys[i] : 0u;
      if (i < nloc) local += (keys[j] > theta ? 1ull : 0ull) | ((keys[j] == theta ? 1ull : 0ull) << 32);
    }
    uint64_t total;
    uint64_t before = run + block_exclusive_scan(local, warp_sums, &total);
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      const uint32_t il = c0 + tid * kItems + j;
      if (il >= nloc) break;
      const uint32_t i = c_begin + il;
      const uint32_t gt_b = (uint32_t)(before & 0xFFFFFFFFu);
      const uint32_t eq_b = (uint32_t)(before >> 32);
      const bool gt = keys[j] > theta, eq = keys[j] == theta;
      const bool hi = gt || (eq && eq_b < need);
      const uint32_t hib = gt_b + min(eq_b, need);
      is_high[i] = hi ? 1 : 0;
      slot[i] = hi ? hib : i - hib;
      before += (gt ? 1ull : 0ull) | ((eq ? 1ull : 0ull) << 32);
    }
    run += total;
  }
}

// ---- full ranks (optional output): a stable LSD radix sort of the inverted keys
// (ascending inverted key = descending score; a stable pass keeps equal keys in index
// order, which is the tie rule), 4-bit digits in 8 passes, one CTA per sequence,
// 1024 keys per step.  Within a step a key's place among the equal digits before it
// comes from match_any inside its warp plus a scan of the per-warp digit counts.
// Then rank[index at sorted position p] = p.  Workspace per sequence: keys and
// indices, double-buffered (4 T words).
constexpr int kSortBins = 16;

__global__ void __launch_bounds__(kThreads) rank_sort_kernel(RankArgs a, uint32_t* ws) {
  __shared__ uint32_t wcount[32][kSortBins];  // per-warp digit counts, then offsets
  __shared__ uint32_t base[kSortBins];        // first output position of each digit
  __shared__ uint32_t total[kSortBins];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t T = (uint32_t)a.T;
  const float* s = a.scores + (int64_t)b * a.ld;
  uint32_t* kb[2] = {ws + (size_t)b * 4 * T, ws + (size_t)b * 4 * T + 2 * (size_t)T};
  uint32_t* ib[2] = {kb[0] + T, kb[1] + T};
  for (uint32_t i = tid; i < T; i += kThreads) {
    kb[0][i] = ~order_key(s[i]);
    ib[0][i] = i;
  }
  __syncthreads();
  const uint32_t lt_mask = (1u << lane) - 1u;
  for (int pass = 0; pass < 8; ++pass) {
    const int sh = 4 * pass;
    const uint32_t* ksrc = kb[pass & 1];
    const uint32_t* isrc = ib[pass & 1];
    uint32_t* kdst = kb[(pass + 1) & 1];
    uint32_t* idst = ib[(pass + 1) & 1];
    // digit histogram of the whole sequence -> first position of each digit
    if (tid < kSortBins) total[tid] = 0;
    __syncthreads();
    for (uint32_t i0 = 0; i0 < T; i0 += kThreads) {
      const uint32_t i = i0 + tid;
      const bool ok = i < T;
      const uint32_t d = ok ? (ksrc[i] >> sh) & (kSortBins - 1) : 0u;
      const uint32_t act = __ballot_sync(0xffffffffu, ok);
      if (ok) {
        const uint32_t peers = __match_any_sync(act, d);
        if ((peers & lt_mask) == 0) atomicAdd(&total[d], (uint32_t)__popc(peers));
      }
    }
    __syncthreads();
    if (tid == 0) {
      uint32_t run = 0;
      for (int d = 0; d < kSortBins; ++d) {
        base[d] = run;
        run += total[d];
      }
    }
    __syncthreads();
    // stable scatter, 1024 keys at a time in index order
    for (uint32_t i0 = 0; i0 < T; i0 += kThreads) {
      const uint32_t i = i0 + tid;
      const bool ok = i < T;
      uint32_t key = 0, idx = 0, d = 0;
      if (ok) {
        key = ksrc[i];
        idx = isrc[i];
        d = (key >> sh) & (kSortBins - 1);
      }
      if (lane < kSortBins) wcount[warp][lane] = 0;
      __syncwarp();
      const uint32_t act = __ballot_sync(0xffffffffu, ok);
      uint32_t before = 0;
      if (ok) {
        const uint32_t peers = __match_any_sync(act, d);
        before = __popc(peers & lt_mask);
        if (before == 0) wcount[warp][d] = (uint32_t)__popc(peers);
      }
      __syncthreads();
      if (tid < kSortBins) {  // exclusive scan over the warps, per digit
        uint32_t run = 0;
        for (int w = 0; w < 32; ++w) {
          const uint32_t c = wcount[w][tid];
          wcount[w][tid] = run;
          run += c;
        }
        total[tid] = run;
      }
      __syncthreads();
      if (ok) {
        const uint32_t pos = base[d] + wcount[warp][d] + before;
        kdst[pos] = key;
        idst[pos] = idx;
      }
      __syncthreads();
      if (tid < kSortBins) base[tid] += total[tid];
      __syncthreads();
    }
  }
  // after an even number of passes the sorted order is back in buffer 0
  uint32_t* rank = a.rank + (int64_t)b * a.T;
  for (uint32_t p = tid; p < T; p += kThreads) rank[ib[0][p]] = p;
}

}  // namespace

size_t rank_workspace_words(int B, int T) { return (size_t)B * 4 * (size_t)T; }

cudaError_t launch_rank_assign(const RankArgs& a, cudaStream_t stream) {
  if (a.B == 0 || a.T == 0) return cudaSuccess;
  const uint32_t chunk = ((uint32_t)a.T + kCluster - 1) / kCluster;
  if (a.T <= kThreads) {
    const cudaError_t e = launch_pdl(rank_small_kernel, dim3(a.B), dim3(kThreads), 0, stream, a);
    if (e != cudaSuccess) return e;
  } else if (a.T >= 8192 && chunk <= kSmemKeys) {
    static bool cattr_set[kAttrDevices] = {};
    const cudaError_t e = once_per_device(cattr_set, [] {
      return cudaFuncSetAttribute(rank_cluster_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)(kSmemKeys * sizeof(uint32_t)));
    });
    if (e != cudaSuccess) return e;
    rank_cluster_kernel<<<a.B * kCluster, kThreads, (size_t)chunk * sizeof(uint32_t), stream>>>(a);
  } else {
    static bool attr_set[kAttrDevices] = {};
    const cudaError_t e = once_per_device(attr_set, [] {
      return cudaFuncSetAttribute(rank_assign_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)(kSmemKeys * sizeof(uint32_t)));
    });
    if (e != cudaSuccess) return e;
    const size_t smem = (uint32_t)a.T <= kSmemKeys ? (size_t)a.T * sizeof(uint32_t) : 0;
    rank_assign_kernel<<<a.B, kThreads, smem, stream>>>(a);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || !a.rank) return e;
  rank_sort_kernel<<<a.B, kThreads, 0, stream>>>(a, a.ws);
  return cudaGetLastError();
}

}  // namespace semkv
