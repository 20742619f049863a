// Per-token routing decisions (Eqs. 18-27) and the per-chunk (expert, block)
// pair counts, shared by the CUDA-core router and the tensor-core router.
#pragma once

#include "internal.cuh"

namespace unif {

// What the decision step reads and writes (device pointers, one entry per
// token unless stated).
struct DecideArgs {
  const uint8_t* mask;  // [T] or null (0 = padding)
  int T, K, B;
  const float* bias;    // [K+1] router bias (zero when the caller gave none)
  float tau, alpha_fixed, beta_fixed;
  int topk_fixed, prefix;
  float* alpha;
  int32_t* b;
  int32_t* k;
  uint64_t* shr;
  uint64_t* emask;
  float* s;             // [T][K] affinities by expert index
  int32_t* bcnt;        // caller's b(x) output or null
  int32_t* kcnt;        // caller's k(x) output or null
  int32_t* chunk_cnt;   // [G][n_chunks]: pairs per group and 32-token chunk
  int n_chunks;
};

// Blocks of expert e that a token with shared set `shr` and residual expert
// set `em` runs: the shared blocks for e = 0 (Eq. 28), the complementary
// blocks for a selected residual expert (Eqs. 23, 29).
__device__ __forceinline__ uint64_t expert_blocks(int e, uint64_t shr, uint64_t em,
                                                  uint64_t full) {
  if (e == 0) return shr;
  return ((em >> (e - 1)) & 1ull) ? (~shr & full) : 0ull;
}

// Decisions for token t, one thread. z points at the token's router outputs
// (z[0] shared logit, z[1..K] residual logits, z[K+1..K+B] block priorities),
// in shared memory; z[1..K] is overwritten with biased logits. sv is K floats
// of scratch. Returns the shared block set and the residual expert set.
__device__ __forceinline__ void decide_token(const DecideArgs& a, int t, bool valid, float* z,
                                             float* sv, uint64_t& shr_out, uint64_t& em_out) {
  const int K = a.K, B = a.B;
  uint64_t shr = 0ull, em = 0ull;
  if (valid) {
    // Eq. 18 (shared demand) and Eq. 19 (shared block count).
    const float z0 = z[0] + (a.bias ? a.bias[0] : 0.f);
    float alpha;
    if (isnan(a.alpha_fixed)) {
      const float sig = 1.0f / (1.0f + expf(-z0));
      alpha = a.tau + (1.0f - 2.0f * a.tau) * sig;
    } else {
      alpha = a.alpha_fixed;
    }
    const int bcount = min(max(__float2int_rn((float)B * alpha), 0), B);
    // Eqs. 21-23: the bcount blocks of largest priority (ties: lower index).
    if (a.prefix) {
      shr = (bcount >= 64) ? ~0ull : ((1ull << bcount) - 1ull);
    } else {
      const float* u = z + 1 + K;
      for (int r = 0; r < bcount; ++r) {
        int best = -1;
        for (int j = 0; j < B; ++j)
          if (!((shr >> j) & 1ull) && (best < 0 || u[j] > u[best])) best = j;
        shr |= 1ull << best;
      }
    }
    // Eq. 24: affinities over the K residual experts.
    float* l = z + 1;  // residual logits (bias added in place)
    float m = -INFINITY;
    for (int j = 0; j < K; ++j) {
      l[j] += a.bias ? a.bias[1 + j] : 0.f;
      m = fmaxf(m, l[j]);
    }
    float den = 0.f;
    for (int j = 0; j < K; ++j) {
      sv[j] = expf(l[j] - m);
      den += sv[j];
    }
    for (int j = 0; j < K; ++j) {
      sv[j] = sv[j] / den;
      a.s[(size_t)t * K + j] = sv[j];
    }
    // Eqs. 25-27: experts in decreasing affinity (decreasing logit, ties to
    // the lower index) until the cumulative mass reaches beta.
    const float beta = isnan(a.beta_fixed) ? 1.0f - alpha : a.beta_fixed;
    int kcount = 0;
    float P = 0.f;
    for (int n = 0; n < K; ++n) {
      int best = -1;
      for (int j = 0; j < K; ++j)
        if (!((em >> j) & 1ull) && (best < 0 || l[j] > l[best])) best = j;
      em |= 1ull << best;
      if (a.topk_fixed > 0) {
        if (n + 1 == a.topk_fixed) { kcount = n + 1; break; }
      } else {
        P += sv[best];
        if (P >= beta) { kcount = n + 1; break; }
      }
    }
    if (kcount == 0) kcount = K;  // rounding left every prefix below beta
    a.alpha[t] = alpha;
    a.b[t] = bcount;
    a.k[t] = kcount;
    a.shr[t] = shr;
    a.emask[t] = em;
    if (a.bcnt) a.bcnt[t] = bcount;
    if (a.kcnt) a.kcnt[t] = kcount;
  } else if (t < a.T) {
    a.alpha[t] = 0.f; a.b[t] = 0; a.k[t] = 0; a.shr[t] = 0ull; a.emask[t] = 0ull;
    for (int j = 0; j < K; ++j) a.s[(size_t)t * K + j] = 0.f;
    if (a.bcnt) a.bcnt[t] = 0;
    if (a.kcnt) a.kcnt[t] = 0;
  }

  shr_out = shr;
  em_out = em;
}

// The (expert, block) pairs of one 32-token chunk (this warp's tokens), per
// group g = e*B + blk, written to chunk_cnt[g][chunk]. All 32 lanes call it.
__device__ __forceinline__ void count_chunk_pairs(const DecideArgs& a, int chunk, int lane,
                                                  uint64_t shr, uint64_t em) {
  const int K = a.K, B = a.B;
  const uint64_t full = (B == 64) ? ~0ull : ((1ull << B) - 1ull);
  for (int e = 0; e <= K; ++e) {
    const uint64_t mb = expert_blocks(e, shr, em, full);
    const bool any = __ballot_sync(0xffffffffu, mb != 0ull) != 0u;
    for (int blk = 0; blk < B; ++blk) {
      const int g = e * B + blk;
      const int c = any ? __popc(__ballot_sync(0xffffffffu, (mb >> blk) & 1ull)) : 0;
      if (lane == (g & 31)) a.chunk_cnt[(size_t)g * a.n_chunks + chunk] = c;
    }
  }
}

DecideArgs decide_args(unif_moe_layer* L, const uint8_t* mask, int T, int32_t* b_out,
                       int32_t* k_out);

}  // namespace unif
