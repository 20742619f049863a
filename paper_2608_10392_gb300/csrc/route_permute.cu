// Router, permute and combine kernels of the UniF-MoE forward pass, plus the
// load-time prototype kernel.
//
//   router  : z = x [W_shr | W_g | mu_1..mu_B] (Eqs. 17, 21) on CUDA cores in
//             fp32, then per token (one warp each) the shared demand and
//             block count (Eqs. 18-19), prototype TopK (Eqs. 22-23), softmax,
//             sort and cumulative cutoff (Eqs. 24-27).
//   permute : groups the (expert, block) pairs of Eqs. 28-29 by pair with a
//             per-chunk ballot histogram, a scan, and a stable scatter, so
//             every group's rows are contiguous and in token order.
//   combine : casts the fp32 accumulator of Eq. 30 to the layer dtype.
#include <math.h>

#include "internal.cuh"

namespace unif {
namespace {

__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }

// fp64 -> bf16 with one round-to-nearest-even step (bf16 keeps 8 significant
// bits): round the fp64 significand at bit 45, which leaves a value that bf16
// holds exactly.
__device__ __forceinline__ float round_f64_to_bf16(double v) {
  if (v == 0.0 || !isfinite(v)) return (float)v;
  if (fabs(v) < 0x1p-126) return (float)(rint(v * 0x1p133) * 0x1p-133);
  unsigned long long u = (unsigned long long)__double_as_longlong(v);
  const unsigned long long lsb = (u >> 45) & 1ull;
  u += 0x0FFFFFFFFFFFull + lsb;  // 2^44 - 1 + lsb: ties to even
  u &= ~((1ull << 45) - 1ull);
  return (float)__longlong_as_double((long long)u);
}

// Eq. 20: mu_b = (1/M) sum_{h in H_b} K_shr[:, h]. The sum of stored
// (fp32/bf16) keys is exact in fp64 for these magnitudes, so the single
// rounding below gives the same value on any summation order.
template <typename Tin>
__global__ void prototypes_kernel(const Tin* __restrict__ w_up0, int d, int H, int B,
                                  int round_bf16, float* __restrict__ mu_rows) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= B * d) return;
  const int b = idx / d, i = idx % d, M = H / B;
  double sum = 0.0;
  for (int h = b * M; h < (b + 1) * M; ++h) sum += (double)to_f32(w_up0[(size_t)h * d + i]);
  const double m = sum / (double)M;
  mu_rows[(size_t)b * d + i] = round_bf16 ? round_f64_to_bf16(m) : __double2float_rn(m);
}

// Router columns 0..K (Eq. 17) transposed to [column][d] in fp32.
template <typename Tin>
__global__ void router_transpose_kernel(const Tin* __restrict__ w_router, int d, int C1,
                                        float* __restrict__ wr_t) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= d * C1) return;
  const int i = idx / C1, c = idx % C1;
  wr_t[(size_t)c * d + i] = to_f32(w_router[idx]);
}

// ---------------------------------------------------------------------------
// Router
// ---------------------------------------------------------------------------

constexpr int kRouterThreads = 256;
constexpr int kKc = 32;  // d-chunk of the router GEMM

struct RouterArgs {
  const uint8_t* mask;
  int T, d, K, B, C, Cpad;
  const float* wr_t;
  const float* bias;
  float tau, alpha_fixed, beta_fixed;
  int topk_fixed, prefix;
  float* alpha;
  int32_t* b;
  int32_t* k;
  uint64_t* shr;
  uint64_t* emask;
  int32_t* q;
  float* p;
  float* s;
  int32_t* bcnt;
  int32_t* kcnt;
};

__device__ __forceinline__ float warp_sum_ordered(float v) {
  // Tree to lane 0, then broadcast: every lane sees the same value.
  for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  return __shfl_sync(0xffffffffu, v, 0);
}

__device__ __forceinline__ float warp_max(float v) {
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

template <typename Tin>
__global__ void __launch_bounds__(kRouterThreads)
router_kernel(const Tin* __restrict__ x, RouterArgs a) {
  extern __shared__ float sm[];
  const int Cp = a.Cpad;
  float* xs = sm;                           // [kKc][64]
  float* ws = xs + kKc * kRouterTokens;     // [kKc][Cp]
  float* zs = ws + kKc * Cp;                // [64][Cp + 1]
  float* wscr = zs + kRouterTokens * (Cp + 1);  // per warp: s[64], psort[64], qsort[64]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t0 = blockIdx.x * kRouterTokens;

  // ---- z = x W^T for 64 tokens x Cp columns (fp32 accumulate) ----
  const int ty = tid >> 4, tx = tid & 15;  // 16 x 16 threads: 4 tokens x (Cp/16) cols
  const int ncol = Cp / 16;
  float acc[4][9];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 9; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < a.d; k0 += kKc) {
    // x chunk: 64 tokens x 32 dims, 8 consecutive dims per thread.
    {
      const int tok = tid >> 2, dd = (tid & 3) * 8;
      const int t = t0 + tok;
      float v[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = 0.f;
      if (t < a.T && k0 + dd < a.d) {
        const Tin* src = x + (size_t)t * a.d + k0 + dd;
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = to_f32(src[e]);
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) xs[(dd + e) * kRouterTokens + tok] = v[e];
    }
    for (int idx = tid; idx < kKc * Cp; idx += kRouterThreads) {
      const int c = idx / kKc, kk = idx % kKc;
      ws[kk * Cp + c] = (k0 + kk < a.d) ? a.wr_t[(size_t)c * a.d + k0 + kk] : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < kKc; ++kk) {
      const float4 xv = *reinterpret_cast<const float4*>(&xs[kk * kRouterTokens + ty * 4]);
      const float xa[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
      for (int j = 0; j < 9; ++j) {
        if (j < ncol) {
          const float w = ws[kk * Cp + tx + 16 * j];
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[i][j] = fmaf(xa[i], w, acc[i][j]);
        }
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 9; ++j)
      if (j < ncol) zs[(ty * 4 + i) * (Cp + 1) + tx + 16 * j] = acc[i][j];
  __syncthreads();

  // ---- decisions: one warp per token ----
  float* s_w = wscr + warp * 192;
  float* ps_w = s_w + 64;
  int* qs_w = reinterpret_cast<int*>(ps_w + 64);
  const int K = a.K, B = a.B;
  for (int lt = warp; lt < kRouterTokens; lt += kRouterThreads / 32) {
    const int t = t0 + lt;
    if (t >= a.T) break;
    const bool valid = (a.mask == nullptr) || a.mask[t] != 0;
    const float* z = zs + lt * (Cp + 1);
    if (!valid) {
      if (lane == 0) {
        a.alpha[t] = 0.f; a.b[t] = 0; a.k[t] = 0; a.shr[t] = 0ull; a.emask[t] = 0ull;
        if (a.bcnt) a.bcnt[t] = 0;
        if (a.kcnt) a.kcnt[t] = 0;
      }
      for (int j = lane; j < K; j += 32) {
        a.q[(size_t)t * K + j] = j; a.p[(size_t)t * K + j] = 0.f; a.s[(size_t)t * K + j] = 0.f;
      }
      continue;
    }
    // Eq. 18, Eq. 19.
    const float z0 = z[0] + (a.bias ? a.bias[0] : 0.f);
    float alpha;
    if (isnan(a.alpha_fixed)) {
      const float sig = 1.0f / (1.0f + expf(-z0));
      alpha = a.tau + (1.0f - 2.0f * a.tau) * sig;
    } else {
      alpha = a.alpha_fixed;
    }
    int bcount = __float2int_rn((float)B * alpha);
    bcount = min(max(bcount, 0), B);
    // Eqs. 21-23: rank of each block's priority (ties to the lower index).
    uint64_t shr = 0ull;
    for (int base = 0; base < B; base += 32) {
      const int blk = base + lane;
      bool in = false;
      if (blk < B) {
        if (a.prefix) {
          in = blk < bcount;
        } else {
          const float ub = z[1 + K + blk];
          int rank = 0;
          for (int i = 0; i < B; ++i) {
            const float ui = z[1 + K + i];
            rank += (ui > ub) || (ui == ub && i < blk);
          }
          in = rank < bcount;
        }
      }
      shr |= (uint64_t)__ballot_sync(0xffffffffu, in) << base;
    }
    // Eq. 24: softmax over the K residual logits.
    float zl[2], el[2];
    float m = -INFINITY;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int j = lane + 32 * r;
      zl[r] = (j < K) ? z[1 + j] + (a.bias ? a.bias[1 + j] : 0.f) : -INFINITY;
      m = fmaxf(m, zl[r]);
    }
    m = warp_max(m);
    float part = 0.f;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int j = lane + 32 * r;
      el[r] = (j < K) ? expf(zl[r] - m) : 0.f;
      part += el[r];
    }
    const float den = warp_sum_ordered(part);
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int j = lane + 32 * r;
      if (j < K) s_w[j] = el[r] / den;
    }
    __syncwarp();
    // Eq. 25: rank by decreasing affinity (ties to the lower index). The
    // identity fill keeps the sorted lists a permutation even for NaN logits.
    for (int r = lane; r < K; r += 32) { ps_w[r] = 0.f; qs_w[r] = r; }
    __syncwarp();
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int j = lane + 32 * r;
      if (j < K) {
        const float sj = s_w[j];
        int rank = 0;
        for (int i = 0; i < K; ++i) {
          const float si = s_w[i];
          rank += (si > sj) || (si == sj && i < j);
        }
        ps_w[rank] = sj;
        qs_w[rank] = j;
        a.s[(size_t)t * K + j] = sj;
      }
    }
    __syncwarp();
    // Eqs. 26-27: smallest prefix whose cumulative mass reaches beta.
    const float beta = isnan(a.beta_fixed) ? 1.0f - alpha : a.beta_fixed;
    int kcount = K;
    if (a.topk_fixed > 0) {
      kcount = a.topk_fixed;
    } else {
      int first = K;
      for (int base = 0; base < K; base += 32) {
        const int r = base + lane;
        bool hit = false;
        if (r < K) {
          float P = 0.f;
          for (int i = 0; i <= r; ++i) P += ps_w[i];
          hit = P >= beta;
        }
        const unsigned bal = __ballot_sync(0xffffffffu, hit);
        if (bal && first == K) first = base + __ffs(bal) - 1;
      }
      kcount = min(first + 1, K);
    }
    uint64_t em = 0ull;
    for (int i = 0; i < kcount; ++i) em |= 1ull << qs_w[i];
    for (int r = lane; r < K; r += 32) {
      a.q[(size_t)t * K + r] = qs_w[r];
      a.p[(size_t)t * K + r] = ps_w[r];
    }
    if (lane == 0) {
      a.alpha[t] = alpha;
      a.b[t] = bcount;
      a.k[t] = kcount;
      a.shr[t] = shr;
      a.emask[t] = em;
      if (a.bcnt) a.bcnt[t] = bcount;
      if (a.kcnt) a.kcnt[t] = kcount;
    }
    __syncwarp();
  }
}

// ---------------------------------------------------------------------------
// Permute: (expert, block) group table
// ---------------------------------------------------------------------------

constexpr int kPermThreads = kChunkTokens;  // one token per thread
constexpr int kPermWarps = kPermThreads / 32;
constexpr int kGroupBatch = 1024;           // groups per shared-memory pass

// Blocks of expert e that token (shr, em) runs: the shared blocks for e = 0,
// the complementary blocks for a selected residual expert (Eqs. 22-23, 28-29).
__device__ __forceinline__ uint64_t expert_blocks(int e, uint64_t shr, uint64_t em,
                                                  uint64_t full) {
  if (e == 0) return shr;
  return ((em >> (e - 1)) & 1ull) ? (~shr & full) : 0ull;
}

__global__ void __launch_bounds__(kPermThreads)
count_kernel(const uint64_t* __restrict__ shr_o, const uint64_t* __restrict__ em_o, int T,
             int K, int B, int n_chunks, int32_t* __restrict__ chunk_cnt) {
  __shared__ int wcnt[kPermWarps][kGroupBatch];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int chunk = blockIdx.x;
  const int t = chunk * kChunkTokens + tid;
  const uint64_t full = (B == 64) ? ~0ull : ((1ull << B) - 1ull);
  const uint64_t shr = (t < T) ? shr_o[t] : 0ull;
  const uint64_t em = (t < T) ? em_o[t] : 0ull;
  const int G = (K + 1) * B;
  for (int g0 = 0; g0 < G; g0 += kGroupBatch) {
    const int g1 = min(G, g0 + kGroupBatch);
    for (int e = g0 / B; e * B < g1; ++e) {
      const uint64_t m = expert_blocks(e, shr, em, full);
      const bool any = __ballot_sync(0xffffffffu, m != 0ull) != 0u;
      for (int blk = 0; blk < B; ++blk) {
        const int g = e * B + blk;
        if (g < g0 || g >= g1) continue;
        const unsigned bal = any ? __ballot_sync(0xffffffffu, (m >> blk) & 1ull) : 0u;
        if (lane == 0) wcnt[warp][g - g0] = __popc(bal);
      }
    }
    __syncthreads();
    for (int g = g0 + tid; g < g1; g += kPermThreads) {
      int sum = 0;
#pragma unroll
      for (int w = 0; w < kPermWarps; ++w) sum += wcnt[w][g - g0];
      chunk_cnt[(size_t)g * n_chunks + chunk] = sum;
    }
    __syncthreads();
  }
}

__device__ __forceinline__ int warp_incl_scan(int v, int lane) {
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  return v;
}

// Exclusive scans: per group over chunks, then over groups (rows padded to
// the tile height) -> group offsets, the tile list and the padding rows.
__global__ void __launch_bounds__(1024)
scan_kernel(int G, int n_chunks, int32_t* __restrict__ chunk_cnt, int32_t* __restrict__ grp_cnt,
            int32_t* __restrict__ grp_off, int32_t* __restrict__ n_tiles,
            int32_t* __restrict__ tile_group, int32_t* __restrict__ tile_row0,
            int32_t* __restrict__ row_tok, float* __restrict__ row_w) {
  __shared__ int wsum_rows[32], wsum_tiles[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int g = warp; g < G; g += 32) {
    int carry = 0;
    int32_t* col = chunk_cnt + (size_t)g * n_chunks;
    for (int c0 = 0; c0 < n_chunks; c0 += 32) {
      const int c = c0 + lane;
      const int v = (c < n_chunks) ? col[c] : 0;
      const int inc = warp_incl_scan(v, lane);
      if (c < n_chunks) col[c] = carry + inc - v;
      carry += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (lane == 0) grp_cnt[g] = carry;
  }
  __syncthreads();
  const int per = (G + 1023) / 1024;
  const int ga = min(G, tid * per), gb = min(G, ga + per);
  int my_rows = 0, my_tiles = 0;
  for (int g = ga; g < gb; ++g) {
    const int padded = (grp_cnt[g] + kTileRows - 1) / kTileRows * kTileRows;
    my_rows += padded;
    my_tiles += padded / kTileRows;
  }
  const int inc_r = warp_incl_scan(my_rows, lane);
  const int inc_t = warp_incl_scan(my_tiles, lane);
  if (lane == 31) { wsum_rows[warp] = inc_r; wsum_tiles[warp] = inc_t; }
  __syncthreads();
  if (warp == 0) {
    const int vr = wsum_rows[lane], vt = wsum_tiles[lane];
    const int ir = warp_incl_scan(vr, lane), it = warp_incl_scan(vt, lane);
    wsum_rows[lane] = ir - vr;
    wsum_tiles[lane] = it - vt;
    if (lane == 31) { grp_off[G] = ir; n_tiles[0] = it; }
  }
  __syncthreads();
  int row = wsum_rows[warp] + inc_r - my_rows;
  int tile = wsum_tiles[warp] + inc_t - my_tiles;
  for (int g = ga; g < gb; ++g) {
    const int cnt = grp_cnt[g];
    const int padded = (cnt + kTileRows - 1) / kTileRows * kTileRows;
    grp_off[g] = row;
    for (int i = 0; i < padded / kTileRows; ++i) {
      tile_group[tile + i] = g;
      tile_row0[tile + i] = row + i * kTileRows;
    }
    for (int r = row + cnt; r < row + padded; ++r) { row_tok[r] = -1; row_w[r] = 0.f; }
    row += padded;
    tile += padded / kTileRows;
  }
}

// Stable scatter: row position = group offset + rows of earlier chunks +
// rows of earlier warps in this chunk + earlier lanes of this warp.
__global__ void __launch_bounds__(kPermThreads)
scatter_kernel(const uint64_t* __restrict__ shr_o, const uint64_t* __restrict__ em_o,
               const float* __restrict__ alpha_o, const float* __restrict__ s_o, int T, int K,
               int B, int n_chunks, const int32_t* __restrict__ chunk_off,
               const int32_t* __restrict__ grp_off, int32_t* __restrict__ row_tok,
               float* __restrict__ row_w) {
  __shared__ int wbase[kPermWarps][kGroupBatch];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int chunk = blockIdx.x;
  const int t = chunk * kChunkTokens + tid;
  const uint64_t full = (B == 64) ? ~0ull : ((1ull << B) - 1ull);
  const uint64_t shr = (t < T) ? shr_o[t] : 0ull;
  const uint64_t em = (t < T) ? em_o[t] : 0ull;
  const unsigned lt_mask = (1u << lane) - 1u;
  const int G = (K + 1) * B;
  for (int g0 = 0; g0 < G; g0 += kGroupBatch) {
    const int g1 = min(G, g0 + kGroupBatch);
    for (int e = g0 / B; e * B < g1; ++e) {
      const uint64_t m = expert_blocks(e, shr, em, full);
      const bool any = __ballot_sync(0xffffffffu, m != 0ull) != 0u;
      for (int blk = 0; blk < B; ++blk) {
        const int g = e * B + blk;
        if (g < g0 || g >= g1) continue;
        const unsigned bal = any ? __ballot_sync(0xffffffffu, (m >> blk) & 1ull) : 0u;
        if (lane == 0) wbase[warp][g - g0] = __popc(bal);
      }
    }
    __syncthreads();
    for (int g = g0 + tid; g < g1; g += kPermThreads) {
      int run = grp_off[g] + chunk_off[(size_t)g * n_chunks + chunk];
#pragma unroll
      for (int w = 0; w < kPermWarps; ++w) {
        const int c = wbase[w][g - g0];
        wbase[w][g - g0] = run;
        run += c;
      }
    }
    __syncthreads();
    for (int e = g0 / B; e * B < g1; ++e) {
      const uint64_t m = expert_blocks(e, shr, em, full);
      if (__ballot_sync(0xffffffffu, m != 0ull) == 0u) continue;
      const float w = (m == 0ull) ? 0.f : (e == 0 ? alpha_o[t] : s_o[(size_t)t * K + e - 1]);
      for (int blk = 0; blk < B; ++blk) {
        const int g = e * B + blk;
        if (g < g0 || g >= g1) continue;
        const bool f = (m >> blk) & 1ull;
        const unsigned bal = __ballot_sync(0xffffffffu, f);
        if (f) {
          const int pos = wbase[warp][g - g0] + __popc(bal & lt_mask);
          row_tok[pos] = t;
          row_w[pos] = w;
        }
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Combine: y (fp32 accumulator) -> output dtype
// ---------------------------------------------------------------------------

__global__ void cast_out_bf16(const float4* __restrict__ y, uint2* __restrict__ out, size_t n4) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4;
       i += (size_t)gridDim.x * blockDim.x) {
    const float4 v = y[i];
    __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y);
    __nv_bfloat162 hi = __floats2bfloat162_rn(v.z, v.w);
    uint2 o;
    o.x = *reinterpret_cast<unsigned*>(&lo);
    o.y = *reinterpret_cast<unsigned*>(&hi);
    out[i] = o;
  }
}

__global__ void copy_out_f32(const float4* __restrict__ y, float4* __restrict__ out, size_t n4) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4;
       i += (size_t)gridDim.x * blockDim.x)
    out[i] = y[i];
}

}  // namespace

cudaError_t launch_prototypes(unif_moe_layer* L, const void* w_router, const float* bias,
                              cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(L->wr_t, 0, sizeof(float) * L->router_cols_pad * L->d, s);
  if (e != cudaSuccess) return e;
  const int C1 = L->K + 1;
  const int n1 = L->d * C1;
  if (L->dtype == UNIF_MOE_BF16)
    router_transpose_kernel<<<(n1 + 255) / 256, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(w_router), L->d, C1, L->wr_t);
  else
    router_transpose_kernel<<<(n1 + 255) / 256, 256, 0, s>>>(static_cast<const float*>(w_router),
                                                             L->d, C1, L->wr_t);
  const int n2 = L->B * L->d;
  float* mu_rows = L->wr_t + (size_t)C1 * L->d;
  if (L->dtype == UNIF_MOE_BF16)
    prototypes_kernel<<<(n2 + 255) / 256, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(L->w_up), L->d, L->H, L->B, 1, mu_rows);
  else
    prototypes_kernel<<<(n2 + 255) / 256, 256, 0, s>>>(static_cast<const float*>(L->w_up), L->d,
                                                       L->H, L->B, 0, mu_rows);
  if (bias)
    e = cudaMemcpyAsync(L->bias, bias, sizeof(float) * C1, cudaMemcpyDeviceToDevice, s);
  else
    e = cudaMemsetAsync(L->bias, 0, sizeof(float) * C1, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

static size_t router_smem(const unif_moe_layer* L) {
  const int Cp = L->router_cols_pad;
  return sizeof(float) * ((size_t)kKc * kRouterTokens + (size_t)kKc * Cp +
                          (size_t)kRouterTokens * (Cp + 1) + 8 * 192);
}

cudaError_t launch_router(unif_moe_layer* L, const void* x, const uint8_t* mask, int T,
                          int32_t* b_out, int32_t* k_out, cudaStream_t s) {
  RouterArgs a;
  a.mask = mask; a.T = T; a.d = L->d; a.K = L->K; a.B = L->B;
  a.C = L->router_cols; a.Cpad = L->router_cols_pad;
  a.wr_t = L->wr_t; a.bias = L->bias;
  a.tau = L->tau; a.alpha_fixed = L->th.alpha_fixed; a.beta_fixed = L->th.beta_fixed;
  a.topk_fixed = L->th.topk_fixed; a.prefix = L->th.prefix_blocks;
  a.alpha = L->ws.alpha; a.b = L->ws.b; a.k = L->ws.k; a.shr = L->ws.shr_mask;
  a.emask = L->ws.exp_mask; a.q = L->ws.q; a.p = L->ws.p; a.s = L->ws.s;
  a.bcnt = b_out; a.kcnt = k_out;
  const size_t smem = router_smem(L);
  const int grid = (T + kRouterTokens - 1) / kRouterTokens;
  if (L->dtype == UNIF_MOE_BF16)
    router_kernel<__nv_bfloat16><<<grid, kRouterThreads, smem, s>>>(
        static_cast<const __nv_bfloat16*>(x), a);
  else
    router_kernel<float><<<grid, kRouterThreads, smem, s>>>(static_cast<const float*>(x), a);
  return cudaGetLastError();
}

cudaError_t router_setup(unif_moe_layer* L) {
  const int smem = (int)router_smem(L);
  cudaError_t e = cudaFuncSetAttribute(router_kernel<__nv_bfloat16>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(router_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              smem);
}

cudaError_t launch_permute(unif_moe_layer* L, int T, cudaStream_t s) {
  const int n_chunks = (T + kChunkTokens - 1) / kChunkTokens;
  Workspace& w = L->ws;
  count_kernel<<<n_chunks, kPermThreads, 0, s>>>(w.shr_mask, w.exp_mask, T, L->K, L->B, n_chunks,
                                                 w.chunk_cnt);
  scan_kernel<<<1, 1024, 0, s>>>(L->G, n_chunks, w.chunk_cnt, w.grp_cnt, w.grp_off, w.n_tiles,
                                 w.tile_group, w.tile_row0, w.row_tok, w.row_w);
  scatter_kernel<<<n_chunks, kPermThreads, 0, s>>>(w.shr_mask, w.exp_mask, w.alpha, w.s, T, L->K,
                                                   L->B, n_chunks, w.chunk_cnt, w.grp_off,
                                                   w.row_tok, w.row_w);
  return cudaGetLastError();
}

cudaError_t launch_combine(unif_moe_layer* L, void* out, int T, cudaStream_t s) {
  const size_t n4 = (size_t)T * L->d / 4;
  const int grid = L->n_sm * 8;
  if (L->dtype == UNIF_MOE_BF16)
    cast_out_bf16<<<grid, 256, 0, s>>>(reinterpret_cast<const float4*>(L->ws.y32),
                                       static_cast<uint2*>(out), n4);
  else
    copy_out_f32<<<grid, 256, 0, s>>>(reinterpret_cast<const float4*>(L->ws.y32),
                                      static_cast<float4*>(out), n4);
  return cudaGetLastError();
}

}  // namespace unif

// ---------------------------------------------------------------------------
// Grouping without allocation (unif_moe_group_noalloc)
// ---------------------------------------------------------------------------
// Some callers cannot call cudaMalloc: inference engines that plan all
// device memory up front and give plugins no allocator after setup, and
// latency-critical paths that must not pay cudaMalloc's implicit device
// synchronisation. For them the grouping step's only scratch, the per-chunk
// group counts, lives in this file-scope device array, which every GPU that
// loads the library holds (1 MiB) until the process exits. Its contents
// persist between calls; the count kernel overwrites every entry a call
// reads, so nothing needs clearing. Calls that overlap on the GPU share the
// array and race.
#include <mutex>

namespace unif {

constexpr int kNoAllocScratchInts = 1 << 18;  // 1 MiB of int32
static __device__ __align__(256) int32_t g_group_scratch[kNoAllocScratchInts];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
int32_t* g_scratch_dev_ptr[kMaxDevices] = {};

// The device address of g_group_scratch on the current device. In host code
// the array's name is only a host-side stand-in, so the address is looked up
// once per device (first call with that device current) and cached.
int32_t* group_scratch_on_current_device(cudaError_t* err) {
  int dev = -1;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= kMaxDevices) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_dev_ptr[dev]) {
    void* p = nullptr;
    *err = cudaGetSymbolAddress(&p, g_group_scratch);
    if (*err != cudaSuccess) return nullptr;
    g_scratch_dev_ptr[dev] = static_cast<int32_t*>(p);
  }
  return g_scratch_dev_ptr[dev];
}

}  // namespace
}  // namespace unif

extern "C" UNIF_MOE_API int unif_moe_group_noalloc(
    int T, int n_experts, int n_blocks, const uint64_t* shared_mask, const uint64_t* expert_mask,
    const float* alpha, const float* affinity, int32_t* counts, int32_t* offsets,
    int32_t* n_tiles, int32_t* tile_group, int32_t* tile_row0, int32_t* row_token,
    float* row_weight, int64_t row_capacity, void* stream) {
  using namespace unif;
  if (T < 0 || n_experts < 1 || n_experts > 64 || n_blocks < 2 || n_blocks > 64) {
    set_error("group_noalloc: bad sizes T=%d K=%d B=%d", T, n_experts, n_blocks);
    return UNIF_MOE_ERR_ARG;
  }
  if (!counts || !offsets || !n_tiles || !tile_group || !tile_row0 || !row_token || !row_weight ||
      (T > 0 && (!shared_mask || !expert_mask || !alpha || !affinity))) {
    set_error("group_noalloc: NULL pointer");
    return UNIF_MOE_ERR_ARG;
  }
  const int G = (n_experts + 1) * n_blocks;
  const int n_chunks = (T + kChunkTokens - 1) / kChunkTokens;
  if ((int64_t)G * n_chunks > kNoAllocScratchInts) {
    set_error("group_noalloc: (K+1)*B*ceil(T/256) = %lld exceeds the built-in scratch of %d "
              "entries; reduce T", (long long)G * n_chunks, kNoAllocScratchInts);
    return UNIF_MOE_ERR_CAPACITY;
  }
  const int64_t need = (int64_t)T * n_experts * n_blocks + (int64_t)G * (kTileRows - 1);
  if (row_capacity < need) {
    set_error("group_noalloc: row_capacity %lld below the bound T*K*B + G*127 = %lld",
              (long long)row_capacity, (long long)need);
    return UNIF_MOE_ERR_CAPACITY;
  }
  cudaError_t e;
  int32_t* scratch = group_scratch_on_current_device(&e);
  if (!scratch) {
    set_error("group_noalloc: scratch address lookup failed: %s", cudaGetErrorString(e));
    return UNIF_MOE_ERR_CUDA;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (n_chunks > 0)
    count_kernel<<<n_chunks, kPermThreads, 0, s>>>(shared_mask, expert_mask, T, n_experts,
                                                   n_blocks, n_chunks, scratch);
  scan_kernel<<<1, 1024, 0, s>>>(G, n_chunks, scratch, counts, offsets, n_tiles, tile_group,
                                 tile_row0, row_token, row_weight);
  if (n_chunks > 0)
    scatter_kernel<<<n_chunks, kPermThreads, 0, s>>>(shared_mask, expert_mask, alpha, affinity, T,
                                                     n_experts, n_blocks, n_chunks, scratch,
                                                     offsets, row_token, row_weight);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error("group_noalloc: launch failed: %s", cudaGetErrorString(e));
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}
