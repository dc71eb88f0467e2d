// Host-side check of the decode work plan (make_decode_plan in decode.cu), built by
// tests/test_decode_plan.py with nvcc and run on the CPU (no kernel is launched).
//
// For every (sequence, KV head) pair and pool the check recomputes, from the plan
// alone, the tile range each CTA of the balanced plan takes (the arithmetic of the
// affine pool kernels) and its partial slot, and requires: every tile of the pool in
// exactly one CTA's range, slots inside the pair's stride (the stage's slot after the
// pools'), the CTA count within one wave of resident CTAs (two 8-warp or one 16-warp CTA
// per SM), and the stride within the caller's limit.  Cases: the workloads' shapes, tiny and one-sided pools, staged tails,
// reduced strides (the no-allocation entry point), and seeded random shapes.
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "../paper_2608_28911_gb300/csrc/decode.cu"

using namespace semkv;

static int check(int L_hi, int L_lo, int B, int H, int Hq, long hi, long lo, int st, int sms,
                 int max_stride, bool verbose) {
  const DecodePlan P = make_decode_plan(SEMKV_BASE_AFFINE, L_hi, L_lo, B, H, Hq, hi, lo, st, sms,
                                        max_stride);
  if (P.stride > max_stride) return 0;  // reported to the caller as a short workspace
  const long pairs = (long)B * H;
  const long total = pairs * P.W;
  int bad = 0;
  if (P.ctas > 2L * sms) bad++;
  if (P.fast && P.warps == 16 && P.ctas > sms) bad++;   // one 16-warp CTA per SM
  for (long bh = 0; bh < pairs; ++bh) {
    int n_hi, n_lo;
    pair_slots(P, bh, n_hi, n_lo);
    if (n_hi + n_lo + st > P.stride) bad++;
    for (int src = 0; src < 2; ++src) {
      const int tiles = src ? P.tiles_lo : P.tiles_hi;
      const long w = src ? P.w_lo : P.w_hi;
      const long S = bh * P.W + (src ? (long)P.w_hi * P.tiles_hi : 0);
      const long E = S + w * tiles;
      std::vector<int> owners(tiles, 0);
      for (long c = 0; c < P.ctas; ++c) {
        const long start = c * P.per, end = start + P.per < total ? start + P.per : total;
        if (E <= S || E <= start || S >= end) continue;
        const long x0 = (start > S ? start : S) - S, x1 = (end < E ? end : E) - S;
        const long t0 = (x0 + w - 1) / w, t1l = (x1 + w - 1) / w;
        const long t1 = t1l < tiles ? t1l : tiles;
        for (long t = t0; t < t1; ++t) owners[t]++;
        const long slot = (c - S / P.per) + (src ? n_hi : 0);
        if (slot < 0 || slot >= (src ? n_hi + n_lo : n_hi)) bad++;
      }
      for (int t = 0; t < tiles; ++t)
        if (owners[t] != 1) bad++;
    }
  }
  if (verbose || bad)
    printf("L%d/%d B%d H%d hi %ld lo %ld stage %d sms %d max_stride %d: ctas %d stride %d "
           "per %lld w %d/%d warps %d: %s\n",
           L_hi, L_lo, B, H, hi, lo, st, sms, max_stride, P.ctas, P.stride, (long long)P.per,
           P.w_hi, P.w_lo, P.warps, bad ? "BAD" : "ok");
  return bad ? 1 : 0;
}

int main() {
  int bad = 0;
  // the workloads' shapes (counts after one appended 128-token block)
  bad += check(6, 5, 16, 8, 32, 17072 + 33, 48592 + 95, 0, 152, 65, true);   // 16 x 64K
  bad += check(6, 5, 4, 8, 32, 17072, 48592, 0, 152, 65, true);             // 4 x 64K
  bad += check(6, 5, 1, 8, 32, 8520 + 33, 24248 + 95, 0, 152, 65, true);     // 1 x 32K
  bad += check(6, 5, 1, 8, 32, 34079 + 33, 96993 + 95, 0, 152, 65, true);    // 128K layer
  bad += check(6, 5, 1, 8, 32, 1065, 3031, 1, 152, 65, true);                // block-wise
  bad += check(5, 5, 1, 1, 4, 0, 1024, 0, 152, 65, true);                    // uniform tiny
  // one-sided, single tiles, staged tails, reduced strides
  bad += check(6, 5, 1, 8, 32, 20, 0, 0, 152, 65, false);
  bad += check(6, 5, 1, 8, 32, 1, 1, 0, 152, 65, false);
  bad += check(6, 5, 2, 8, 32, 700, 2300, 1, 152, 65, false);
  bad += check(6, 5, 40, 8, 32, 312, 888, 1, 152, 6, false);
  bad += check(6, 5, 672, 1, 4, 12, 36, 0, 152, 3, false);
  bad += check(6, 5, 504, 1, 4, 12, 36, 1, 152, 4, false);
  srand(12345);
  for (int i = 0; i < 3000; ++i) {
    const int B = 1 + rand() % 24, H = 1 + rand() % 8;
    const long hi = rand() % 40000, lo = rand() % 90000;
    const int sms = 1 + rand() % 200;
    bad += check(rand() % 2 ? 6 : 5, 5, B, H, 4 * H, hi, lo, rand() % 2, sms,
                 rand() % 3 ? 65 : 3 + rand() % 30, false);
  }
  printf("%s\n", bad ? "FAILED" : "all plans ok");
  return bad != 0;
}
