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
    const float inv_den = 1.0f / den;
    for (int j = 0; j < K; ++j) {
      sv[j] = sv[j] * inv_den;
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

// A token's KC affinities (KC a multiple of 8, dst 32-byte aligned): one
// 32-byte store per 8, so that each store fills a whole sector instead of a
// warp's store instruction touching 32 sectors partially.
template <int KC>
__device__ __forceinline__ void store_affinities(float* dst, const float (&e)[KC]) {
  static_assert(KC % 8 == 0, "whole 32-byte sectors");
#pragma unroll
  for (int j = 0; j < KC; j += 8)
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(dst + j),
                 "r"(__float_as_uint(e[j])), "r"(__float_as_uint(e[j + 1])),
                 "r"(__float_as_uint(e[j + 2])), "r"(__float_as_uint(e[j + 3])),
                 "r"(__float_as_uint(e[j + 4])), "r"(__float_as_uint(e[j + 5])),
                 "r"(__float_as_uint(e[j + 6])), "r"(__float_as_uint(e[j + 7]))
                 : "memory");
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
    const float inv_den = 1.0f / den;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      e[j] = e[j] * inv_den;
      sv[j] = e[j];
    }
    store_affinities<KC>(a.s + (size_t)t * KC, e);
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
    for (int j = 0; j < KC; j += 4)
      *reinterpret_cast<float4*>(a.s + (size_t)t * KC + j) = make_float4(0.f, 0.f, 0.f, 0.f);
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
__device__ __forceinline__ void count_chunk_pairs_rt(const DecideArgs& a, int lane, uint64_t shr,
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

// The same counts with K and B known at compile time: the ballots issue
// back to back, lane 0 stores all masks at once, and the group loop unrolls
// with shifts for the divisions, so its shared-memory reads are all in
// flight together.
template <int KC, int BC>
__device__ __forceinline__ void count_chunk_pairs_ct(int lane, uint64_t shr, uint64_t em,
                                                     uint32_t* scratch, int32_t* out, int stride) {
  uint32_t mb[BC], me[KC];
#pragma unroll
  for (int blk = 0; blk < BC; ++blk) mb[blk] = __ballot_sync(0xffffffffu, (shr >> blk) & 1ull);
#pragma unroll
  for (int e = 0; e < KC; ++e) me[e] = __ballot_sync(0xffffffffu, (em >> e) & 1ull);
  if (lane == 0) {
#pragma unroll
    for (int blk = 0; blk < BC; ++blk) scratch[blk] = mb[blk];
#pragma unroll
    for (int e = 0; e < KC; ++e) scratch[64 + e] = me[e];
  }
  __syncwarp();
  constexpr int G = (KC + 1) * BC;
#pragma unroll
  for (int g0 = 0; g0 < G; g0 += 32) {
    const int g = g0 + lane;
    if (g < G) {
      const int e = g / BC, blk = g % BC;
      const uint32_t sh = scratch[blk];
      out[(size_t)g * stride] = e == 0 ? __popc(sh) : __popc(scratch[64 + e - 1] & ~sh);
    }
  }
  __syncwarp();
}

__device__ __forceinline__ void count_chunk_pairs(const DecideArgs& a, int lane, uint64_t shr,
                                                  uint64_t em, uint32_t* scratch, int32_t* out,
                                                  int stride) {
  if (a.K == 8 && a.B == 8)
    count_chunk_pairs_ct<8, 8>(lane, shr, em, scratch, out, stride);
  else if (a.K == 16 && a.B == 16)
    count_chunk_pairs_ct<16, 16>(lane, shr, em, scratch, out, stride);
  else
    count_chunk_pairs_rt(a, lane, shr, em, scratch, out, stride);
}

// ---------------------------------------------------------------------------
// Grouping inside the router (Eq. 35's pairs laid out per group)
// ---------------------------------------------------------------------------
// Each group g owns a region of `region` rows (at most one row per token) in
// row_tok / row_w. A router CTA reserves its rows of every group with one
// atomic add on the group's fill counter, so rows of different CTAs land in
// arrival order (within a CTA, in token order); nothing downstream depends
// on the order of a group's rows. Once the router grid has completed, the
// fill counters are the group sizes: the GEMM kernels number the 128-row
// tiles of every group from them (tile_table below), each tile with its
// count of real rows (the rest of a group's last tile is padding, which
// they skip). The combine kernel copies the sizes out for the group table
// and zeroes the counters for the next forward, also after a forward whose
// router gave up a wait.
struct GroupArgs {
  int G, K, B;
  int region;
  int32_t* fill;           // [G] rows reserved so far (0 at the start of a forward)
  int32_t* row_tok;
  float* row_w;
  int* status;
};

__device__ __forceinline__ void named_bar(uint32_t id, uint32_t n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// Shared-memory ints group_rows needs.
__host__ __device__ constexpr int group_rows_smem_ints(int NW, int G) {
  return NW * G + 8;  // per-chunk counts (then first rows), misc
}

// Runs in the NW decision warps of a router CTA (threads tid = 0 .. NW*32-1,
// named barrier `bar`; thread tid holds token t0 + tid, with shared block set
// `shr` and residual expert set `em`), after warp w's count_chunk_pairs
// wrote its 32-token chunk's per-group pair counts to sm[w * G + g] and its
// lane masks to masks[w * 128 ...] (masks[blk] = lanes sharing block blk,
// masks[64 + j] = lanes selecting residual expert j). Token i of the CTA has
// alpha at dec_s[i * dec_stride + 2K] and its affinities s_1..s_K at
// dec_s[i * dec_stride + j]. `sm` has group_rows_smem_ints(NW, G) ints.
//
// Each thread writes its own token's rows: with one warp per scheduler the
// phase is bound by the length of each thread's chain of index arithmetic,
// and a token's rows (b + k (B - b) of them) make a shorter chain than the
// rows of one (group, chunk) pair walked by one thread.
template <int NW>
__device__ void group_rows(const GroupArgs& a, int tid, int t0, uint64_t shr, uint64_t em,
                           const uint32_t* masks, const float* dec_s, int dec_stride,
                           int32_t* sm, uint32_t bar) {
  constexpr int NT = NW * 32;
  const int G = a.G, B = a.B;
  int32_t* first = sm;  // [NW][G] chunk counts, then each chunk's first row
  // 1. this CTA's rows of each group, reserved in the group's region; the
  // rows of chunk v follow those of chunks 0 .. v-1 (token order). A group
  // whose rows were not reserved gets a negative first row in every chunk.
  for (int g = tid; g < G; g += NT) {
    int n = 0;
#pragma unroll
    for (int v = 0; v < NW; ++v) n += first[v * G + g];
    int base = -1;
    if (n > 0) {
      base = atomicAdd(a.fill + g, n);
      if (base + n > a.region) {  // stale counters: keep the writes inside the region
        atomicOr(a.status, kStatusBadIndex);
        base = -1;
      }
    }
    int o = base < 0 ? -(1 << 30) : base;
#pragma unroll
    for (int v = 0; v < NW; ++v) {
      const int c = first[v * G + g];
      first[v * G + g] = o;
      o += c;
    }
  }
  named_bar(bar, NT);
  // 2. the token's rows: its row in group g is the chunk's first row of g
  // plus the number of lower lanes of the chunk that are also in g
  const int c = tid >> 5;
  const uint32_t lt = (1u << (tid & 31)) - 1u;
  const int32_t* fc = first + c * G;
  const uint32_t* mk = masks + c * 128;
  const float* ds = dec_s + tid * dec_stride;
  const int tok = t0 + tid;
  const float alpha = ds[2 * a.K];
  for (uint64_t rem = shr; rem != 0ull; rem &= rem - 1ull) {  // shared blocks (e = 0)
    const int blk = __ffsll((long long)rem) - 1;
    const int r = fc[blk] + __popc(mk[blk] & lt);
    if (r >= 0) {
      a.row_tok[(size_t)blk * a.region + r] = tok;
      a.row_w[(size_t)blk * a.region + r] = alpha;
    }
  }
  const uint64_t comp = ~shr & (B >= 64 ? ~0ull : ((1ull << B) - 1ull));
  for (uint64_t rj = em; rj != 0ull; rj &= rj - 1ull) {  // residual experts
    const int j = __ffsll((long long)rj) - 1;
    const uint32_t mj = mk[64 + j];
    const float w = ds[j];
    for (uint64_t rb = comp; rb != 0ull; rb &= rb - 1ull) {  // their complementary blocks
      const int blk = __ffsll((long long)rb) - 1, g = (j + 1) * B + blk;
      const int r = fc[g] + __popc(mj & ~mk[blk] & lt);
      if (r >= 0) {
        a.row_tok[(size_t)g * a.region + r] = tok;
        a.row_w[(size_t)g * a.region + r] = w;
      }
    }
  }
}

// Expert-major grouping (the fused expert-tile FFN): group e = expert e
// (G = K + 1), one row per (token, expert) the token runs: the shared expert
// for every token with b > 0 (weight alpha, Eq. 28), each selected residual
// expert j (weight s_j, Eq. 29). The blocks a row runs follow from the
// token's shared block set (expert_blocks). Lane masks: masks[0] = lanes
// with b > 0, masks[64 + j] = lanes selecting residual expert j; counts
// out[e * stride] per expert.
__device__ __forceinline__ void count_chunk_experts(int K, int lane, uint64_t shr, uint64_t em,
                                                    uint32_t* scratch, int32_t* out, int stride) {
  const uint32_t m0 = __ballot_sync(0xffffffffu, shr != 0ull);
  if (lane == 0) scratch[0] = m0;
  for (int e = 0; e < K; ++e) {
    const uint32_t m = __ballot_sync(0xffffffffu, (em >> e) & 1ull);
    if (lane == 0) scratch[64 + e] = m;
  }
  __syncwarp();
  for (int g = lane; g <= K; g += 32)
    out[(size_t)g * stride] = __popc(g == 0 ? scratch[0] : scratch[64 + g - 1]);
  __syncwarp();
}

// group_rows for the expert-major grouping (the same reservation, then each
// thread writes its token's 1 + k rows; arguments as group_rows, G = K + 1).
template <int NW>
__device__ void group_rows_expert(const GroupArgs& a, int tid, int t0, uint64_t shr, uint64_t em,
                                  const uint32_t* masks, const float* dec_s, int dec_stride,
                                  int32_t* sm, uint32_t bar) {
  constexpr int NT = NW * 32;
  const int G = a.G;
  int32_t* first = sm;
  for (int g = tid; g < G; g += NT) {
    int n = 0;
#pragma unroll
    for (int v = 0; v < NW; ++v) n += first[v * G + g];
    int base = -1;
    if (n > 0) {
      base = atomicAdd(a.fill + g, n);
      if (base + n > a.region) {
        atomicOr(a.status, kStatusBadIndex);
        base = -1;
      }
    }
    int o = base < 0 ? -(1 << 30) : base;
#pragma unroll
    for (int v = 0; v < NW; ++v) {
      const int c = first[v * G + g];
      first[v * G + g] = o;
      o += c;
    }
  }
  named_bar(bar, NT);
  const int c = tid >> 5;
  const uint32_t lt = (1u << (tid & 31)) - 1u;
  const int32_t* fc = first + c * G;
  const uint32_t* mk = masks + c * 128;
  const float* ds = dec_s + tid * dec_stride;
  const int tok = t0 + tid;
  if (shr != 0ull) {
    const int r = fc[0] + __popc(mk[0] & lt);
    if (r >= 0) {
      a.row_tok[r] = tok;
      a.row_w[r] = ds[2 * a.K];
    }
  }
  for (uint64_t rj = em; rj != 0ull; rj &= rj - 1ull) {
    const int j = __ffsll((long long)rj) - 1;
    const int r = fc[j + 1] + __popc(mk[64 + j] & lt);
    if (r >= 0) {
      a.row_tok[(size_t)(j + 1) * a.region + r] = tok;
      a.row_w[(size_t)(j + 1) * a.region + r] = ds[j];
    }
  }
}

// The tiles of the groups whose sizes are fill[0..G) (each clamped to the
// region): first_s[g] = first tile of group g (first_s[G] = all tiles),
// cnt_s[g] = its size. Run by one warp; shared arrays of G + 1 and G ints.
__device__ __forceinline__ void tile_table(const int32_t* fill, int G, int region, int lane,
                                           int32_t* first_s, int32_t* cnt_s) {
  int carry = 0;
  for (int g0 = 0; g0 < G; g0 += 32) {
    const int g = g0 + lane;
    const int c = g < G ? min(__ldcg(fill + g), region) : 0;
    const int nt = (c + 127) / 128;
    int inc = nt;
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += v;
    }
    if (g < G) {
      first_s[g] = carry + inc - nt;
      cnt_s[g] = c;
    }
    carry += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (lane == 0) first_s[G] = carry;
}

// Group, first row and real rows of tile k, from tile_table's arrays.
__device__ __forceinline__ void tile_lookup(int k, const int32_t* first_s, const int32_t* cnt_s,
                                            int G, int region, int& g, int& row0, int& rows) {
  int lo = 0, hi = G - 1;  // the last group whose first tile is <= k
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (first_s[mid] <= k) lo = mid; else hi = mid - 1;
  }
  const int i = k - first_s[lo];
  g = lo;
  row0 = lo * region + 128 * i;
  rows = min(128, cnt_s[lo] - 128 * i);
}

DecideArgs decide_args(unif_moe_layer* L, const uint8_t* mask, int T, int32_t* b_out,
                       int32_t* k_out);

}  // namespace unif
