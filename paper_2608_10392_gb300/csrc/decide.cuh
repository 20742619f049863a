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
__device__ __forceinline__ void decide_token_rt(const DecideArgs& a, int t, bool valid, float* z,
                                                float* sv, uint64_t& shr_out, uint64_t& em_out,
                                                float& alpha_out) {
  const int K = a.K, B = a.B;
  uint64_t shr = 0ull, em = 0ull;
  alpha_out = 0.f;
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
    alpha_out = alpha;
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

// The same decisions with K and B known at compile time: the priorities,
// logits and affinities stay in registers and every loop unrolls. The
// arithmetic and its order are those of decide_token_rt.
template <int KC, int BC>
__device__ __forceinline__ void decide_token_ct(const DecideArgs& a, int t, bool valid, float* z,
                                                float* sv, uint64_t& shr_out, uint64_t& em_out,
                                                float& alpha_out) {
  uint64_t shr = 0ull, em = 0ull;
  alpha_out = 0.f;
  if (valid) {
    const float z0 = z[0] + a.bias[0];
    float alpha;
    if (isnan(a.alpha_fixed)) {
      const float sig = 1.0f / (1.0f + expf(-z0));
      alpha = a.tau + (1.0f - 2.0f * a.tau) * sig;
    } else {
      alpha = a.alpha_fixed;
    }
    const int bcount = min(max(__float2int_rn((float)BC * alpha), 0), BC);
    if (a.prefix) {
      shr = (bcount >= 64) ? ~0ull : ((1ull << bcount) - 1ull);
    } else if (bcount > 0) {
      float u[BC];
#pragma unroll
      for (int j = 0; j < BC; ++j) u[j] = z[1 + KC + j];
#pragma unroll
      for (int j = 0; j < BC; ++j) {
        int rank = 0;
#pragma unroll
        for (int i = 0; i < BC; ++i) rank += (u[i] > u[j]) || (u[i] == u[j] && i < j);
        if (rank < bcount) shr |= 1ull << j;
      }
    }
    float l[KC], e[KC];
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      l[j] = z[1 + j] + a.bias[1 + j];
      m = fmaxf(m, l[j]);
    }
    float den = 0.f;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      e[j] = expf(l[j] - m);
      den += e[j];
    }
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      e[j] = e[j] / den;
      sv[j] = e[j];
      a.s[(size_t)t * KC + j] = e[j];
    }
    const float beta = isnan(a.beta_fixed) ? 1.0f - alpha : a.beta_fixed;
    int rk[KC];
    int kcount = KC;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      int rank = 0;
      float mass = 0.f;
#pragma unroll
      for (int i = 0; i < KC; ++i) {
        const bool before = (l[i] > l[j]) || (l[i] == l[j] && i < j);
        rank += before;
        mass += (before || i == j) ? e[i] : 0.f;
      }
      rk[j] = rank;
      if (a.topk_fixed == 0 && mass >= beta) kcount = min(kcount, rank + 1);
    }
    if (a.topk_fixed > 0) kcount = a.topk_fixed;
#pragma unroll
    for (int j = 0; j < KC; ++j)
      if (rk[j] < kcount) em |= 1ull << j;
    a.alpha[t] = alpha;
    alpha_out = alpha;
    a.b[t] = bcount;
    a.k[t] = kcount;
    a.shr[t] = shr;
    a.emask[t] = em;
    if (a.bcnt) a.bcnt[t] = bcount;
    if (a.kcnt) a.kcnt[t] = kcount;
  } else if (t < a.T) {
    a.alpha[t] = 0.f; a.b[t] = 0; a.k[t] = 0; a.shr[t] = 0ull; a.emask[t] = 0ull;
#pragma unroll
    for (int j = 0; j < KC; ++j) a.s[(size_t)t * KC + j] = 0.f;
    if (a.bcnt) a.bcnt[t] = 0;
    if (a.kcnt) a.kcnt[t] = 0;
  }
  shr_out = shr;
  em_out = em;
}

// Decisions for token t (dispatch on the layer's K and B).
__device__ __forceinline__ void decide_token(const DecideArgs& a, int t, bool valid, float* z,
                                             float* sv, uint64_t& shr_out, uint64_t& em_out,
                                             float& alpha_out) {
  if (a.K == 8 && a.B == 8)
    decide_token_ct<8, 8>(a, t, valid, z, sv, shr_out, em_out, alpha_out);
  else if (a.K == 16 && a.B == 16)
    decide_token_ct<16, 16>(a, t, valid, z, sv, shr_out, em_out, alpha_out);
  else
    decide_token_rt(a, t, valid, z, sv, shr_out, em_out, alpha_out);
}

// The (expert, block) pairs of one 32-token chunk (this warp's tokens), per
// group g = e*B + blk, written to out[g * stride]. All 32 lanes call it;
// scratch is 128 words of this warp's shared memory. One ballot per block
// (lanes sharing it) and per residual expert (lanes selecting it); a group's
// count is then a population count of their intersection.
__device__ __forceinline__ void count_chunk_pairs(const DecideArgs& a, int lane, uint64_t shr,
                                                  uint64_t em, uint32_t* scratch, int32_t* out,
                                                  int stride) {
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
    out[(size_t)g * stride] = c;
  }
  __syncwarp();
}

// ---------------------------------------------------------------------------
// Grouping inside the router (Eq. 35's pairs laid out per group)
// ---------------------------------------------------------------------------
// Each group g owns a region of `region` rows (at most one row per token) in
// row_tok / row_w, so a router CTA can place its tokens' rows as soon as it
// knows, per group, how many rows the CTAs before it produced: a single-pass
// scan with decoupled look-back over per-CTA aggregates. The last CTA to
// finish numbers the tiles (128 rows) of every group into the tile list,
// with each tile's count of real rows (the rest of a group's last tile is
// padding, which the GEMM kernels skip).
struct GroupArgs {
  int G, K, B;
  int n_ctas;
  int region;
  uint32_t epoch;          // this forward's tag in the look-back flags
  int32_t* lb_agg;         // [n_ctas][G] rows per CTA and group
  int32_t* lb_incl;        // [n_ctas][G] rows of CTAs 0..c per group
  uint32_t* lb_flag;       // [n_ctas] (epoch << 2) | 1 aggregate, | 2 inclusive
  int32_t* ticket;         // CTAs done; the last resets it
  int32_t* row_tok;
  float* row_w;
  int32_t* grp_cnt;
  int32_t* grp_off;        // padded offsets as if the groups were contiguous
  int32_t* n_tiles;
  int32_t* tile_group;
  int32_t* tile_row0;
  int32_t* tile_rows;
  int* status;
  long long wait_limit;
};
constexpr int kMaxGroupsPerThread = 8;

__device__ __forceinline__ void named_bar(uint32_t id, uint32_t n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Runs in the NW decision warps of router CTA `cta` (threads tid = 0 ..
// NW*32-1, named barrier `bar`), after warp w's count_chunk_pairs wrote its
// 32-token chunk's per-group pair counts to cnt_s[w][g] and its lane masks
// to `masks`. Lane `lane` of warp w holds token t
// (valid or not) with its shared block set, residual expert set, alpha and
// affinities s_tok[0..K-1]. base_s is [NW][G] ints of shared memory, misc_s
// NW + 3 ints.
template <int NW>
__device__ void group_rows(const GroupArgs& a, int cta, int tid, int w, int lane, int t,
                           uint64_t shr, uint64_t em, float alpha, const float* s_tok,
                           const uint32_t* masks, const int32_t* cnt_s, int32_t* base_s,
                           int32_t* misc_s, uint32_t bar) {
  constexpr int NT = NW * 32;
  const int G = a.G;
  const uint32_t tag = a.epoch << 2;
  // 1. this CTA's rows per group, published
  int gl[kMaxGroupsPerThread], agg[kMaxGroupsPerThread], excl[kMaxGroupsPerThread];
  int ng = 0;
  for (int g = tid; g < G && ng < kMaxGroupsPerThread; g += NT) {
    int sum = 0;
    for (int v = 0; v < NW; ++v) sum += cnt_s[v * G + g];
    gl[ng] = g;
    agg[ng] = sum;
    excl[ng] = 0;
    a.lb_agg[(size_t)cta * G + g] = sum;
    ++ng;
  }
  __threadfence();
  named_bar(bar, NT);
  if (tid == 0) st_release_u32(a.lb_flag + cta, tag | 1u);
  // 2. rows of all CTAs before this one: walk back 32 CTAs at a time (warp
  // 0 reads their flags together), summing aggregates up to the nearest CTA
  // whose inclusive count is published
  for (int top = cta - 1; top >= 0;) {
    if (w == 0) {
      const int j = top - lane;
      uint32_t st = 0u;
      if (j >= 0) {
        const long long t0 = clock64();
        for (;;) {
          const uint32_t f = ld_acquire_u32(a.lb_flag + j);
          if ((f & ~3u) == tag && (f & 3u) != 0u) { st = f & 3u; break; }
          if (clock64() - t0 > a.wait_limit) {
            atomicOr(a.status, kStatusTimeout);
            st = 2u;  // give up: treat as published (the result is invalid anyway)
            break;
          }
        }
      }
      const unsigned incl_lanes = __ballot_sync(0xffffffffu, st == 2u);
      // nearest inclusive CTA in this window, or none (-1)
      const int k = incl_lanes ? __ffs(incl_lanes) - 1 : -1;
      if (lane == 0) {
        misc_s[NW + 1] = k;
        misc_s[NW + 2] = min(32, top + 1);  // CTAs in this window
      }
    }
    named_bar(bar, NT);
    const int k = misc_s[NW + 1], n = misc_s[NW + 2];
    named_bar(bar, NT);  // misc_s is rewritten by the next window
    const int n_agg = k >= 0 ? k : n;
    for (int i = 0; i < ng; ++i) {
      int sum = 0;
      for (int v = 0; v < n_agg; ++v) sum += __ldcg(a.lb_agg + (size_t)(top - v) * G + gl[i]);
      if (k >= 0) sum += __ldcg(a.lb_incl + (size_t)(top - k) * G + gl[i]);
      excl[i] += sum;
    }
    if (k >= 0) break;
    top -= n;
  }
  // 3. inclusive counts published; each warp's first row per group
  for (int i = 0; i < ng; ++i) {
    const int g = gl[i];
    a.lb_incl[(size_t)cta * G + g] = excl[i] + agg[i];
    int b = excl[i];
    for (int v = 0; v < NW; ++v) {
      base_s[v * G + g] = b;
      b += cnt_s[v * G + g];
    }
  }
  __threadfence();
  named_bar(bar, NT);
  if (tid == 0) st_release_u32(a.lb_flag + cta, tag | 2u);
  // 4. this lane's rows, one per (expert, block) pair of its token: the
  // row's rank among the chunk's tokens in the group (tokens stay in index
  // order) comes from the lane masks count_chunk_pairs left in `masks`
  // (masks[blk]: lanes sharing block blk, masks[64 + j]: lanes selecting
  // residual expert j)
  {
    const uint64_t full = (a.B == 64) ? ~0ull : ((1ull << a.B) - 1ull);
    const unsigned lt_mask = (1u << lane) - 1u;
    const int32_t* base = base_s + w * G;
    for (uint64_t m = shr; m != 0ull; m &= m - 1ull) {
      const int blk = __ffsll((long long)m) - 1;
      const size_t pos = (size_t)blk * a.region + base[blk] + __popc(masks[blk] & lt_mask);
      a.row_tok[pos] = t;
      a.row_w[pos] = alpha;
    }
    const uint64_t comp = ~shr & full;
    for (uint64_t ee = em; ee != 0ull; ee &= ee - 1ull) {
      const int j = __ffsll((long long)ee) - 1;
      const float wt = s_tok[j];
      const uint32_t ej = masks[64 + j];
      for (uint64_t m = comp; m != 0ull; m &= m - 1ull) {
        const int blk = __ffsll((long long)m) - 1;
        const int g = (j + 1) * a.B + blk;
        const size_t pos = (size_t)g * a.region + base[g] + __popc(ej & ~masks[blk] & lt_mask);
        a.row_tok[pos] = t;
        a.row_w[pos] = wt;
      }
    }
  }
  // 5. the last CTA to finish builds the tile list
  if (tid == 0) {
    int old;
    asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], 1;" : "=r"(old) : "l"(a.ticket) : "memory");
    misc_s[NW] = old;
  }
  named_bar(bar, NT);
  if (misc_s[NW] != a.n_ctas - 1) return;
  if (tid == 0) *a.ticket = 0;  // every CTA has taken its ticket
  // group totals into shared memory first (one round of loads), then the
  // groups in contiguous runs per thread, so that a block scan numbers the
  // tiles in group order
  int32_t* tot = base_s;  // no longer needed for row offsets
  for (int g = tid; g < G; g += NT) tot[g] = __ldcg(a.lb_incl + (size_t)(a.n_ctas - 1) * G + g);
  named_bar(bar, NT);
  const int per = (G + NT - 1) / NT;
  const int g0 = min(G, tid * per), g1 = min(G, g0 + per);
  int my_tiles = 0;
  for (int g = g0; g < g1; ++g) my_tiles += (tot[g] + 127) / 128;
  int inc = my_tiles;
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += n;
  }
  if (lane == 31) misc_s[w] = inc;
  named_bar(bar, NT);
  int first_tile = inc - my_tiles;
  for (int v = 0; v < w; ++v) first_tile += misc_s[v];
  for (int g = g0; g < g1; ++g) {
    const int cnt = tot[g];
    const int tiles = (cnt + 127) / 128;
    a.grp_cnt[g] = cnt;
    a.grp_off[g] = first_tile * 128;
    for (int i = 0; i < tiles; ++i) {
      a.tile_group[first_tile + i] = g;
      a.tile_row0[first_tile + i] = g * a.region + 128 * i;
      a.tile_rows[first_tile + i] = min(128, cnt - 128 * i);
    }
    first_tile += tiles;
  }
  if (tid == NT - 1) {
    a.n_tiles[0] = first_tile;
    a.grp_off[G] = first_tile * 128;
  }
}

DecideArgs decide_args(unif_moe_layer* L, const uint8_t* mask, int T, int32_t* b_out,
                       int32_t* k_out);

}  // namespace unif
