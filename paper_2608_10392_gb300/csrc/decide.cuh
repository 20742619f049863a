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
// in shared memory; z[1..K] is overwritten with biased logits. sv is 2K
// floats of shared-memory scratch. Returns the shared block set and the
// residual expert set. Orders are taken as ranks (how many entries precede
// an entry: larger value first, ties to the lower index), whose comparisons
// are independent of one another.
__device__ __forceinline__ void decide_token(const DecideArgs& a, int t, bool valid, float* z,
                                             float* sv, uint64_t& shr_out, uint64_t& em_out) {
  const int K = a.K, B = a.B;
  uint64_t shr = 0ull, em = 0ull;
  if (valid) {
    // Eq. 18 (shared demand) and Eq. 19 (shared block count).
    const float z0 = z[0] + a.bias[0];
    float alpha;
    if (isnan(a.alpha_fixed)) {
      const float sig = 1.0f / (1.0f + expf(-z0));
      alpha = a.tau + (1.0f - 2.0f * a.tau) * sig;
    } else {
      alpha = a.alpha_fixed;
    }
    const int bcount = min(max(__float2int_rn((float)B * alpha), 0), B);
    // Eqs. 21-23: block j is shared iff its priority rank is below b.
    if (a.prefix) {
      shr = (bcount >= 64) ? ~0ull : ((1ull << bcount) - 1ull);
    } else if (bcount > 0) {
      const float* u = z + 1 + K;
      for (int j = 0; j < B; ++j) {
        const float uj = u[j];
        int rank = 0;
        for (int i = 0; i < B; ++i) {
          const float ui = u[i];
          rank += (ui > uj) || (ui == uj && i < j);
        }
        if (rank < bcount) shr |= 1ull << j;
      }
    }
    // Eq. 24: affinities over the K residual experts.
    float* l = z + 1;  // residual logits (bias added in place)
    float m = -INFINITY;
    for (int j = 0; j < K; ++j) {
      l[j] += a.bias[1 + j];
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
    // Eqs. 25-27: rank the experts by affinity (by logit, which orders them
    // the same way exactly); P at expert j's rank is the mass of the experts
    // ranked up to and including it. k is the smallest rank + 1 whose mass
    // reaches beta; the selected experts are those ranked below k.
    const float beta = isnan(a.beta_fixed) ? 1.0f - alpha : a.beta_fixed;
    int* rk = reinterpret_cast<int*>(sv + K);
    int kcount = K;  // K if rounding left every prefix below beta
    for (int j = 0; j < K; ++j) {
      const float lj = l[j];
      int rank = 0;
      float mass = 0.f;
      for (int i = 0; i < K; ++i) {
        const float li = l[i];
        const bool before = (li > lj) || (li == lj && i < j);
        rank += before;
        mass += (before || i == j) ? sv[i] : 0.f;
      }
      rk[j] = rank;
      if (a.topk_fixed == 0 && mass >= beta) kcount = min(kcount, rank + 1);
    }
    if (a.topk_fixed > 0) kcount = a.topk_fixed;
    for (int j = 0; j < K; ++j)
      if (rk[j] < kcount) em |= 1ull << j;
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
// group g = e*B + blk, written to chunk_cnt[g][chunk]. All 32 lanes call it;
// scratch is 128 words of this warp's shared memory. One ballot per block
// (lanes sharing it) and per residual expert (lanes selecting it); a group's
// count is then a population count of their intersection.
__device__ __forceinline__ void count_chunk_pairs(const DecideArgs& a, int chunk, int lane,
                                                  uint64_t shr, uint64_t em, uint32_t* scratch) {
  const int K = a.K, B = a.B;
  for (int blk = 0; blk < B; ++blk) {
    const uint32_t m = __ballot_sync(0xffffffffu, (shr >> blk) & 1ull);
    if (lane == 0) scratch[blk] = m;
  }
  for (int e = 0; e < K; ++e) {
    const uint32_t m = __ballot_sync(0xffffffffu, (em >> e) & 1ull);
    if (lane == 0) scratch[64 + e] = m;
  }
  __syncwarp();
  const int G = (K + 1) * B;
  for (int g = lane; g < G; g += 32) {
    const int e = g / B, blk = g % B;
    const uint32_t shared_lanes = scratch[blk];
    const int c = (e == 0) ? __popc(shared_lanes) : __popc(scratch[64 + e - 1] & ~shared_lanes);
    a.chunk_cnt[(size_t)g * a.n_chunks + chunk] = c;
  }
  __syncwarp();
}

DecideArgs decide_args(unif_moe_layer* L, const uint8_t* mask, int T, int32_t* b_out,
                       int32_t* k_out);

}  // namespace unif
