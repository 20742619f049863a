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

#include <algorithm>

#include "decide.cuh"
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
// The router matrix is kept as [d][Cp] fp32: row i holds x_i's weights for
// W_shr, W_g (columns 0..K) and mu_1..mu_B (columns K+1..K+B), zero padded.
template <typename Tin>
__global__ void prototypes_kernel(const Tin* __restrict__ w_up0, int d, int H, int B,
                                  int round_bf16, int Cp, int col0, float* __restrict__ wr) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= B * d) return;
  const int b = idx / d, i = idx % d, M = H / B;
  double sum = 0.0;
  for (int h = b * M; h < (b + 1) * M; ++h) sum += (double)to_f32(w_up0[(size_t)h * d + i]);
  const double m = sum / (double)M;
  wr[(size_t)i * Cp + col0 + b] = round_bf16 ? round_f64_to_bf16(m) : __double2float_rn(m);
}

// The router matrix as bf16 [Cp][d] (K-major operand of the tensor-core
// router). Every entry is a bf16 value already (bf16 weights, prototypes
// rounded to bf16, zero padding), so the conversion is exact.
__global__ void router_to_bf16_kernel(const float* __restrict__ wr, int d, int Cp,
                                      __nv_bfloat16* __restrict__ wr_bf) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= d * Cp) return;
  const int c = idx / d, i = idx % d;
  wr_bf[idx] = __float2bfloat16_rn(wr[(size_t)i * Cp + c]);
}

// Router columns 0..K (Eq. 17) into the [d][Cp] fp32 router matrix.
template <typename Tin>
__global__ void router_copy_kernel(const Tin* __restrict__ w_router, int d, int C1, int Cp,
                                   float* __restrict__ wr) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= d * C1) return;
  const int i = idx / C1, c = idx % C1;
  wr[(size_t)i * Cp + c] = to_f32(w_router[idx]);
}

// ---------------------------------------------------------------------------
// Router
// ---------------------------------------------------------------------------

constexpr int kRouterThreads = 256;
constexpr int kKc = 32;          // d-chunk of the router GEMM
constexpr int kWarpChunk = 32;   // tokens per permute chunk on the forward path (one warp)

struct RouterArgs {
  DecideArgs dec;
  int d;
  const float* wr;  // [d][Cp] router matrix
};

__device__ __forceinline__ void load8(const float* src, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 b = *reinterpret_cast<const float4*>(src + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void load8(const __nv_bfloat16* src, float (&v)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(src);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(w[i] << 16);
    v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

// One CTA: 64 tokens. z = x W on CUDA cores (fp32 accumulate), then one
// thread per token takes the decisions of Eqs. 18-27, then each of the two
// deciding warps counts its 32 tokens' (expert, block) pairs per group.
// NCB = Cp / 32 column blocks (each thread: 4 tokens x 2 NCB columns).
template <typename Tin, int NCB>
__global__ void __launch_bounds__(kRouterThreads)
router_kernel(const Tin* __restrict__ x, RouterArgs a) {
  extern __shared__ float sm[];
  constexpr int Cp = 32 * NCB;
  const int K = a.dec.K;
  float* xs = sm;                               // [kKc][64]
  float* ws = xs + kKc * kRouterTokens;         // [kKc][Cp]
  float* zs = ws + kKc * Cp;                    // [64][Cp + 1] logits
  float* ss = zs + kRouterTokens * (Cp + 1);    // [64][2K + 1] decision scratch
  uint32_t* cscr = reinterpret_cast<uint32_t*>(ss + kRouterTokens * (2 * K + 1));  // [2][128]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t0 = blockIdx.x * kRouterTokens;

  // ---- z = x W for 64 tokens x Cp columns (Eqs. 17, 21) ----
  const int ty = tid >> 4, tx = tid & 15;  // tokens 4ty..4ty+3, columns tx + 16 j
  float acc[4][2 * NCB];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 2 * NCB; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < a.d; k0 += kKc) {
    {
      const int tok = tid >> 2, dd = (tid & 3) * 8;
      const int t = t0 + tok;
      float v[8];
      if (t < a.dec.T && k0 + dd < a.d) {
        load8(x + (size_t)t * a.d + k0 + dd, v);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = 0.f;
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) xs[(dd + e) * kRouterTokens + tok] = v[e];
    }
    // weight rows k0..k0+31 are contiguous in the [d][Cp] router matrix
    for (int idx = tid; idx < kKc * Cp / 4; idx += kRouterThreads) {
      const int kk = (idx * 4) / Cp;
      float4 w4 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (k0 + kk < a.d) w4 = reinterpret_cast<const float4*>(a.wr + (size_t)k0 * Cp)[idx];
      reinterpret_cast<float4*>(ws)[idx] = w4;
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < kKc; ++kk) {
      const float4 xv = *reinterpret_cast<const float4*>(&xs[kk * kRouterTokens + ty * 4]);
      const float xa[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
      for (int j = 0; j < 2 * NCB; ++j) {
        const float w = ws[kk * Cp + tx + 16 * j];
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i][j] = fmaf(xa[i], w, acc[i][j]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 2 * NCB; ++j) zs[(ty * 4 + i) * (Cp + 1) + tx + 16 * j] = acc[i][j];
  __syncthreads();
  if (tid >= kRouterTokens) return;

  // ---- decisions: one thread per token ----
  const int t = t0 + tid;
  const bool valid = t < a.dec.T && (a.dec.mask == nullptr || a.dec.mask[t] != 0);
  uint64_t shr, em;
  float alpha;
  decide_token(a.dec, t, valid, zs + tid * (Cp + 1), ss + tid * (2 * K + 1), shr, em, alpha);

  // ---- (expert, block) pairs per group for this warp's 32 tokens ----
  const int chunk = blockIdx.x * (kRouterTokens / kWarpChunk) + warp;
  if (chunk < a.dec.n_chunks)
    count_chunk_pairs(a.dec, lane, shr, em, cscr + warp * 128, a.dec.chunk_cnt + chunk,
                      a.dec.n_chunks);
}

// get_routing helper: experts by decreasing affinity (ties to the lower
// index) and their affinities, one thread per token.
__global__ void sort_affinities_kernel(const float* __restrict__ s, int T, int K,
                                       int32_t* __restrict__ q, float* __restrict__ p) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  const float* st = s + (size_t)t * K;
  uint64_t used = 0ull;
  for (int n = 0; n < K; ++n) {
    int best = -1;
    for (int j = 0; j < K; ++j)
      if (!((used >> j) & 1ull) && (best < 0 || st[j] > st[best])) best = j;
    used |= 1ull << best;
    if (q) q[(size_t)t * K + n] = best;
    if (p) p[(size_t)t * K + n] = st[best];
  }
}

// Per group: exclusive scan over the 32-token chunks (in place) and the
// group's row count. One warp per group.
__global__ void __launch_bounds__(256)
chunk_scan_kernel(int G, int n_chunks, int32_t* __restrict__ chunk_cnt,
                  int32_t* __restrict__ grp_cnt) {
  const int lane = threadIdx.x & 31;
  const int g = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (g >= G) return;
  int32_t* col = chunk_cnt + (size_t)g * n_chunks;
  int carry = 0;
  for (int c0 = 0; c0 < n_chunks; c0 += 32) {
    const int c = c0 + lane;
    const int v = (c < n_chunks) ? col[c] : 0;
    int inc = v;
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += n;
    }
    if (c < n_chunks) col[c] = carry + inc - v;
    carry += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (lane == 0) grp_cnt[g] = carry;
}

// Stable scatter of the (token, weight) rows into their groups, four 32-token
// chunks per CTA (one per warp). Every CTA first scans the groups' padded
// sizes into offsets (shared memory); CTA c also writes the tile list and the
// padding rows of groups g = c, c + gridDim.x, ...
__global__ void __launch_bounds__(128)
group_scatter_kernel(const uint64_t* __restrict__ shr_o, const uint64_t* __restrict__ em_o,
                     const float* __restrict__ alpha_o, const float* __restrict__ s_o, int T,
                     int K, int B, int n_chunks, const int32_t* __restrict__ chunk_off,
                     const int32_t* __restrict__ grp_cnt, int32_t* __restrict__ grp_off,
                     int32_t* __restrict__ n_tiles, int32_t* __restrict__ tile_group,
                     int32_t* __restrict__ tile_row0, int32_t* __restrict__ tile_rows,
                     int32_t* __restrict__ row_tok, float* __restrict__ row_w) {
  extern __shared__ int goff[];  // [G + 1]
  __shared__ int wsum[4];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G = (K + 1) * B;
  const int per = (G + 127) / 128;
  const int ga = min(G, tid * per), gb = min(G, ga + per);
  int mine = 0;
  for (int g = ga; g < gb; ++g) mine += (grp_cnt[g] + kTileRows - 1) / kTileRows * kTileRows;
  int inc = mine;
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += n;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  int base = inc - mine;
  for (int w = 0; w < warp; ++w) base += wsum[w];
  for (int g = ga; g < gb; ++g) {
    goff[g] = base;
    base += (grp_cnt[g] + kTileRows - 1) / kTileRows * kTileRows;
  }
  if (tid == 127) goff[G] = base;
  __syncthreads();
  // side outputs: offsets, tile list, padding rows
  for (int g = blockIdx.x; g < G; g += gridDim.x) {
    const int cnt = grp_cnt[g], off = goff[g];
    const int padded = (cnt + kTileRows - 1) / kTileRows * kTileRows;
    if (tid == 0) grp_off[g] = off;
    for (int i = tid; i < padded / kTileRows; i += 128) {
      tile_group[off / kTileRows + i] = g;
      tile_row0[off / kTileRows + i] = off + i * kTileRows;
      tile_rows[off / kTileRows + i] = min(kTileRows, cnt - i * kTileRows);
    }
    for (int r = off + cnt + tid; r < off + padded; r += 128) { row_tok[r] = -1; row_w[r] = 0.f; }
  }
  if (blockIdx.x == 0 && tid == 0) {
    grp_off[G] = goff[G];
    n_tiles[0] = goff[G] / kTileRows;
  }
  // scatter: each warp first stages its chunk's per-group offsets and its
  // tokens' affinities in shared memory, so the loop below only waits on
  // shared-memory reads
  const int chunk = blockIdx.x * 4 + warp;
  if (chunk >= n_chunks) return;
  int* coff = goff + (G + 1) + warp * G;
  float* sw = reinterpret_cast<float*>(goff + (G + 1) + 4 * G) + warp * 32 * K;
  for (int g = lane; g < G; g += 32) coff[g] = goff[g] + chunk_off[(size_t)g * n_chunks + chunk];
  const int t = chunk * kWarpChunk + lane;
  const int tfirst = chunk * kWarpChunk;
  const int nvalid = min(kWarpChunk, T - tfirst);
  for (int i = lane; i < nvalid * K; i += 32) sw[i] = s_o[(size_t)tfirst * K + i];
  __syncwarp();
  const uint64_t full = (B == 64) ? ~0ull : ((1ull << B) - 1ull);
  const uint64_t shr = (t < T) ? shr_o[t] : 0ull;
  const uint64_t em = (t < T) ? em_o[t] : 0ull;
  const float alpha = (t < T) ? alpha_o[t] : 0.f;
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int e = 0; e <= K; ++e) {
    const uint64_t mb = expert_blocks(e, shr, em, full);
    if (__ballot_sync(0xffffffffu, mb != 0ull) == 0u) continue;
    const float w = (mb == 0ull) ? 0.f : (e == 0 ? alpha : sw[lane * K + e - 1]);
    for (int blk = 0; blk < B; ++blk) {
      const int g = e * B + blk;
      const bool f = (mb >> blk) & 1ull;
      const unsigned bal = __ballot_sync(0xffffffffu, f);
      if (f) {
        const int pos = coff[g] + __popc(bal & lt_mask);
        row_tok[pos] = t;
        row_w[pos] = w;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Permute with 256-token chunks and its own counting pass (used by the
// allocation-free grouping entry point below)
// ---------------------------------------------------------------------------

constexpr int kPermThreads = kChunkTokens;  // one token per thread
constexpr int kPermWarps = kPermThreads / 32;
constexpr int kGroupBatch = 1024;           // groups per shared-memory pass


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
// Tile list from the router's group sizes (bf16 layers that group inside the
// router, when a streaming grouped GEMM reads the list; the weight-stationary
// kernels number their tiles themselves)
// ---------------------------------------------------------------------------
__global__ void tile_list_kernel(const int32_t* __restrict__ fill, int G, int region,
                                 int32_t* __restrict__ n_tiles, int32_t* __restrict__ tile_group,
                                 int32_t* __restrict__ tile_row0, int32_t* __restrict__ tile_rows) {
  extern __shared__ int32_t tl_s[];  // [G + 1] first tiles, [G] sizes
  if (threadIdx.x < 32) tile_table(fill, G, region, threadIdx.x, tl_s, tl_s + G + 1);
  __syncthreads();
  const int nt = tl_s[G];
  if (threadIdx.x == 0) n_tiles[0] = nt;
  for (int k = threadIdx.x; k < nt; k += blockDim.x) {
    int g, r0, rows;
    tile_lookup(k, tl_s, tl_s + G + 1, G, region, g, r0, rows);
    tile_group[k] = g;
    tile_row0[k] = r0;
    tile_rows[k] = rows;
  }
}

// ---------------------------------------------------------------------------
// Combine: y (fp32 accumulator) -> output dtype
// ---------------------------------------------------------------------------

// The fp32 accumulator is all zero between forwards: each combine zeroes
// the rows it reads (zero != 0; the down projection of the next forward
// adds into them), or the expert-tile FFN zeroed the other of its two
// accumulators for the next pass (zero == 0). Also copies the router's
// group fill counters (n_fill ints, the group sizes) to the group table's
// counts and zeroes them for the next forward: every kernel that reads
// them has finished.
__global__ void cast_out_bf16(float4* __restrict__ y, uint2* __restrict__ out, size_t n4,
                              int32_t* fill, int32_t* counts, int n_fill, int region, int zero) {
  grid_dep_wait();  // the down projection's sums are complete
  if (blockIdx.x == 0)
    for (int i = threadIdx.x; i < n_fill; i += blockDim.x) {
      counts[i] = min(fill[i], region);
      fill[i] = 0;
    }
  // four elements per thread and round: all loads first, then the stores
  constexpr int kU = 4;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  for (size_t i0 = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i0 < n4; i0 += kU * stride) {
    float4 v[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const size_t i = i0 + u * stride;
      v[u] = i < n4 ? y[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const size_t i = i0 + u * stride;
      if (i >= n4) break;
      __nv_bfloat162 lo = __floats2bfloat162_rn(v[u].x, v[u].y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(v[u].z, v[u].w);
      uint2 o;
      o.x = *reinterpret_cast<unsigned*>(&lo);
      o.y = *reinterpret_cast<unsigned*>(&hi);
      out[i] = o;
      if (zero) y[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

// ---------------------------------------------------------------------------
// The layer as a Transformer sublayer (converted FFN layers of the paper's
// DeiT-S and BERT backbones, Appendix A, Architecture details): layer
// normalisation LN(v) = gamma (v - mean) / sqrt(var + eps) + beta over each
// token's d features (fp32 statistics: the mean, then the biased variance of
// the centred values), and the residual sum. One warp per token row; lane l
// keeps the row's 8-feature groups l, l + 32, ... (d a multiple of 8, at
// most 1024) in registers and moves each group with 16-byte accesses.
// ---------------------------------------------------------------------------
constexpr int kGroups = 4;  // 8-feature groups per lane: d <= 32 * 8 * kGroups

template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// (load8, the router's 8-value loader, reads the groups)
__device__ __forceinline__ void store8(float* p, const float (&v)[8]) {
  reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}
__device__ __forceinline__ void store8(__nv_bfloat16* p, const float (&v)[8]) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    w[i] = *reinterpret_cast<uint32_t*>(&h);
  }
  *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
}

// In place: this lane's groups of v (features 8 (32 j + lane) ..) -> LN(v);
// the whole warp calls.
template <typename T>
__device__ __forceinline__ void layernorm_warp(float (&v)[kGroups][8], int d, int lane,
                                               const T* __restrict__ gamma,
                                               const T* __restrict__ beta, float eps) {
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < kGroups; ++j)
    if (8 * (32 * j + lane) < d)
#pragma unroll
      for (int i = 0; i < 8; ++i) sum += v[j][i];
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  const float mean = sum / (float)d;
  float sq = 0.f;
#pragma unroll
  for (int j = 0; j < kGroups; ++j)
    if (8 * (32 * j + lane) < d)
#pragma unroll
      for (int i = 0; i < 8; ++i) sq += (v[j][i] - mean) * (v[j][i] - mean);
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  const float inv = 1.0f / sqrtf(sq / (float)d + eps);
#pragma unroll
  for (int j = 0; j < kGroups; ++j) {
    const int f = 8 * (32 * j + lane);
    if (f < d) {
      float g[8], b[8];
      load8(gamma + f, g);
      load8(beta + f, b);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[j][i] = g[i] * ((v[j][i] - mean) * inv) + b[i];
    }
  }
}

// out = LN(x), rows of padding (mask 0) give 0.
template <typename T>
__global__ void __launch_bounds__(256)
layernorm_rows(const T* __restrict__ x, T* __restrict__ out, const uint8_t* __restrict__ mask,
               const T* __restrict__ gamma, const T* __restrict__ beta, float eps, int n_rows,
               int d) {
  const int lane = threadIdx.x & 31;
  const int warps = gridDim.x * (blockDim.x >> 5);
  for (int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < n_rows; r += warps) {
    const size_t base = (size_t)r * d;
    const bool pad = mask != nullptr && mask[r] == 0;
    float v[kGroups][8];
#pragma unroll
    for (int j = 0; j < kGroups; ++j) {
      const int f = 8 * (32 * j + lane);
      if (f < d && !pad) {
        load8(x + base + f, v[j]);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) v[j][i] = 0.f;
      }
    }
    if (!pad) layernorm_warp<T>(v, d, lane, gamma, beta, eps);
#pragma unroll
    for (int j = 0; j < kGroups; ++j) {
      const int f = 8 * (32 * j + lane);
      if (f < d) store8(out + base + f, v[j]);
    }
  }
}

// The sublayer's combine: v = y + x (accumulator row plus the residual
// input), out = LN(v) (NORM) or v; padding rows give 0. Zeroes the
// accumulator rows (zero != 0) and, in block 0, hands the group sizes on
// and zeroes the grouping counters, as cast_out_bf16 does.
template <typename T, bool NORM>
__global__ void __launch_bounds__(256)
combine_residual(float* __restrict__ y, const T* __restrict__ x, T* __restrict__ out,
                 const uint8_t* __restrict__ mask, const T* __restrict__ gamma,
                 const T* __restrict__ beta, float eps, int n_rows, int d, int32_t* fill,
                 int32_t* counts, int n_fill, int region, int zero) {
  grid_dep_wait();  // the down projection's sums are complete
  if (blockIdx.x == 0)
    for (int i = threadIdx.x; i < n_fill; i += blockDim.x) {
      counts[i] = min(fill[i], region);
      fill[i] = 0;
    }
  const int lane = threadIdx.x & 31;
  const int warps = gridDim.x * (blockDim.x >> 5);
  const float zeros[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < n_rows; r += warps) {
    const size_t base = (size_t)r * d;
    const bool pad = mask != nullptr && mask[r] == 0;
    float v[kGroups][8];
#pragma unroll
    for (int j = 0; j < kGroups; ++j) {
      const int f = 8 * (32 * j + lane);
      if (f < d && !pad) {
        float a[8];
        load8(y + base + f, v[j]);
        load8(x + base + f, a);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[j][i] += a[i];
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) v[j][i] = 0.f;
      }
    }
    if (NORM && !pad) layernorm_warp<T>(v, d, lane, gamma, beta, eps);
#pragma unroll
    for (int j = 0; j < kGroups; ++j) {
      const int f = 8 * (32 * j + lane);
      if (f < d) {
        store8(out + base + f, v[j]);
        if (zero) store8(y + base + f, zeros);
      }
    }
  }
}

__global__ void copy_out_f32(float4* __restrict__ y, float4* __restrict__ out, size_t n4) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4;
       i += (size_t)gridDim.x * blockDim.x) {
    out[i] = y[i];
    y[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

}  // namespace

cudaError_t launch_prototypes(unif_moe_layer* L, const void* w_router, const float* bias,
                              cudaStream_t s) {
  const int Cp = L->router_cols_pad;
  cudaError_t e = cudaMemsetAsync(L->wr, 0, sizeof(float) * Cp * L->d, s);
  if (e != cudaSuccess) return e;
  const int C1 = L->K + 1;
  const int n1 = L->d * C1;
  if (L->dtype == UNIF_MOE_BF16)
    router_copy_kernel<<<(n1 + 255) / 256, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(w_router), L->d, C1, Cp, L->wr);
  else
    router_copy_kernel<<<(n1 + 255) / 256, 256, 0, s>>>(static_cast<const float*>(w_router),
                                                        L->d, C1, Cp, L->wr);
  const int n2 = L->B * L->d;
  if (L->dtype == UNIF_MOE_BF16)
    prototypes_kernel<<<(n2 + 255) / 256, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(L->w_up), L->d, L->H, L->B, 1, Cp, C1, L->wr);
  else
    prototypes_kernel<<<(n2 + 255) / 256, 256, 0, s>>>(static_cast<const float*>(L->w_up), L->d,
                                                       L->H, L->B, 0, Cp, C1, L->wr);
  if (L->dtype == UNIF_MOE_BF16)
    router_to_bf16_kernel<<<(L->d * Cp + 255) / 256, 256, 0, s>>>(L->wr, L->d, Cp, L->wr_bf);
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
                          (size_t)kRouterTokens * (Cp + 1) +
                          (size_t)kRouterTokens * (2 * L->K + 1) + 2 * 128);
}

int forward_chunks(int T) { return (T + kWarpChunk - 1) / kWarpChunk; }

DecideArgs decide_args(unif_moe_layer* L, const uint8_t* mask, int T, int32_t* b_out,
                       int32_t* k_out) {
  DecideArgs a;
  a.mask = mask; a.T = T; a.K = L->K; a.B = L->B;
  a.bias = L->bias;
  a.tau = L->tau; a.alpha_fixed = L->th.alpha_fixed; a.beta_fixed = L->th.beta_fixed;
  a.topk_fixed = L->th.topk_fixed; a.prefix = L->th.prefix_blocks;
  const size_t r0 = (size_t)L->rec0;  // the records of this pass's first token
  a.alpha = L->ws.alpha + r0; a.b = L->ws.b + r0; a.k = L->ws.k + r0;
  a.shr = L->ws.shr_mask + r0; a.emask = L->ws.exp_mask + r0; a.s = L->ws.s + r0 * L->K;
  a.bcnt = b_out; a.kcnt = k_out;
  a.chunk_cnt = L->ws.chunk_cnt; a.n_chunks = forward_chunks(T);
  return a;
}

template <typename Tin>
static void* router_fn(int ncb) {
  switch (ncb) {
    case 1: return reinterpret_cast<void*>(router_kernel<Tin, 1>);
    case 2: return reinterpret_cast<void*>(router_kernel<Tin, 2>);
    case 3: return reinterpret_cast<void*>(router_kernel<Tin, 3>);
    case 4: return reinterpret_cast<void*>(router_kernel<Tin, 4>);
    default: return reinterpret_cast<void*>(router_kernel<Tin, 5>);
  }
}

static void* router_entry(const unif_moe_layer* L) {
  const int ncb = L->router_cols_pad / 32;  // 1 + K + B <= 129 columns: ncb <= 5
  return L->dtype == UNIF_MOE_BF16 ? router_fn<__nv_bfloat16>(ncb) : router_fn<float>(ncb);
}

cudaError_t launch_router(unif_moe_layer* L, const void* x, const uint8_t* mask, int T,
                          int32_t* b_out, int32_t* k_out, cudaStream_t s) {
  RouterArgs a;
  a.dec = decide_args(L, mask, T, b_out, k_out);
  a.d = L->d;
  a.wr = L->wr;
  const void* xp = x;
  void* args[] = {const_cast<void**>(&xp), &a};
  const int grid = (T + kRouterTokens - 1) / kRouterTokens;
  return cudaLaunchKernel(router_entry(L), dim3(grid), dim3(kRouterThreads), args, router_smem(L),
                          s);
}

static size_t scatter_smem(const unif_moe_layer* L) {
  return sizeof(int) * ((size_t)L->G + 1 + 4 * (size_t)L->G) + sizeof(float) * 4 * 32 * L->K;
}

cudaError_t router_setup(unif_moe_layer* L) {
  cudaError_t e = cudaFuncSetAttribute(router_entry(L), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)router_smem(L));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(group_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)scatter_smem(L));
}

cudaError_t launch_permute(unif_moe_layer* L, int T, cudaStream_t s) {
  const int n_chunks = forward_chunks(T);
  Workspace& w = L->ws;
  const size_t r0 = (size_t)L->rec0;  // the records of this pass's first token
  chunk_scan_kernel<<<(L->G + 7) / 8, 256, 0, s>>>(L->G, n_chunks, w.chunk_cnt, w.grp_cnt);
  group_scatter_kernel<<<(n_chunks + 3) / 4, 128, scatter_smem(L), s>>>(
      w.shr_mask + r0, w.exp_mask + r0, w.alpha + r0, w.s + r0 * L->K, T, L->K, L->B, n_chunks,
      w.chunk_cnt, w.grp_cnt,
      w.grp_off, w.n_tiles, w.tile_group, w.tile_row0, w.tile_rows, w.row_tok, w.row_w);
  return cudaGetLastError();
}

cudaError_t launch_sort_affinities(unif_moe_layer* L, int T, int32_t* q, float* p,
                                   cudaStream_t s) {
  sort_affinities_kernel<<<(T + 127) / 128, 128, 0, s>>>(L->ws.s, T, L->K, q, p);
  return cudaGetLastError();
}

cudaError_t launch_tile_list(unif_moe_layer* L, cudaStream_t s) {
  return launch_tile_list_from(L, L->ws.grp_fill, s);
}

cudaError_t launch_tile_list_from(unif_moe_layer* L, const int32_t* sizes, cudaStream_t s) {
  Workspace& w = L->ws;
  tile_list_kernel<<<1, 256, sizeof(int32_t) * (2 * (size_t)L->G + 1), s>>>(
      sizes, L->G, L->region_rows, w.n_tiles, w.tile_group, w.tile_row0, w.tile_rows);
  return cudaGetLastError();
}

cudaError_t launch_layernorm(unif_moe_layer* L, const void* x, void* out, const uint8_t* mask,
                             const void* gamma, const void* beta, float eps, int T,
                             cudaStream_t s) {
  const int grid = std::min((T + 7) / 8, L->n_sm * 8);
  if (L->dtype == UNIF_MOE_BF16)
    layernorm_rows<__nv_bfloat16><<<grid, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(x), static_cast<__nv_bfloat16*>(out), mask,
        static_cast<const __nv_bfloat16*>(gamma), static_cast<const __nv_bfloat16*>(beta), eps, T,
        L->d);
  else
    layernorm_rows<float><<<grid, 256, 0, s>>>(
        static_cast<const float*>(x), static_cast<float*>(out), mask,
        static_cast<const float*>(gamma), static_cast<const float*>(beta), eps, T, L->d);
  return cudaGetLastError();
}

cudaError_t launch_combine_residual(unif_moe_layer* L, const void* x, void* out,
                                    const uint8_t* mask, const void* gamma, const void* beta,
                                    float eps, bool norm, int T, cudaStream_t s) {
  const int grid = std::min((T + 7) / 8, L->n_sm * 8);
  const int n_fill = L->fused_group ? L->G : 0;
  float* y = acc_cur(L);
  const int zero = L->ffn_fused ? 0 : 1;  // the expert-tile FFN zeroed the other accumulator
  if (L->dtype == UNIF_MOE_BF16) {
    using B = __nv_bfloat16;
    auto k = norm ? combine_residual<B, true> : combine_residual<B, false>;
    return launch_dependent(k, dim3(grid), dim3(256), 0, s, y, static_cast<const B*>(x),
                            static_cast<B*>(out), mask, static_cast<const B*>(gamma),
                            static_cast<const B*>(beta), eps, T, L->d, L->ws.grp_fill,
                            L->ws.grp_cnt, n_fill, L->region_rows, zero);
  }
  auto k = norm ? combine_residual<float, true> : combine_residual<float, false>;
  return launch_dependent(k, dim3(grid), dim3(256), 0, s, y, static_cast<const float*>(x),
                          static_cast<float*>(out), mask, static_cast<const float*>(gamma),
                          static_cast<const float*>(beta), eps, T, L->d, L->ws.grp_fill,
                          L->ws.grp_cnt, n_fill, L->region_rows, zero);
}

cudaError_t launch_combine(unif_moe_layer* L, void* out, int T, cudaStream_t s) {
  const size_t n4 = (size_t)T * L->d / 4;
  const int grid = L->n_sm * 8;
  if (L->dtype == UNIF_MOE_BF16)
    return launch_dependent(cast_out_bf16, dim3(grid), dim3(256), 0, s,
                            reinterpret_cast<float4*>(acc_cur(L)), static_cast<uint2*>(out),
                            n4, L->ws.grp_fill, L->ws.grp_cnt, L->fused_group ? L->G : 0,
                            L->region_rows, L->ffn_fused ? 0 : 1);
  else
    copy_out_f32<<<grid, 256, 0, s>>>(reinterpret_cast<float4*>(L->ws.y32),
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
