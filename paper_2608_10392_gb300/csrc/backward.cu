// Backward pass of the UniF-MoE layer (training, Sec. III-E) for bf16 layers,
// on the tensor cores, over the group table of the forward that preceded it.
//
// The discrete decisions (b, I_shr, k and the selected experts) are
// piecewise constant in the parameters, so gradients flow through the
// pathway weights alpha (Eq. 18) and s_j (Eq. 24) and through the experts
// (Eq. 16). For a group row (token t, expert e, block b) with weight w and
// pre-activations a = x K_e[:, H_b]:
//   g      = dy V_e[H_b, :]^T                 (the output gradient per channel)
//   dL/da  = w g GeLU'(a)                     -> DA row
//   w GeLU(a)                                 -> HW row
//   dL/dw += sum_h GeLU(a_h) g_h              -> dwt[t][e] (alpha for e = 0, s_j for e = 1+j)
// then, summed over rows:
//   dL/dx[t]          += DA row K_e[H_b, :]   (the streaming down kernel on K^T)
//   dL/dK_e[H_b, :]    = DA^T X[rows]         (weight-gradient kernel)
//   dL/dV_e[:, H_b]    = DY[rows]^T HW        (same kernel)
// and per token dL/dz from dL/dalpha and dL/ds (Eqs. 18, 24), dL/dW* = X^T dL/dz,
// dL/dbias = sum dL/dz, dL/dx += dL/dz W*^T; the Gram regulariser (Eq.
// diversity-loss) adds lambda_div dL_div/dW*.
//
// Kernels (in stream order): tile list from the forward's group sizes,
// bwd_hidden_kernel (two tcgen05 accumulators: x K and dy V^T over the same
// gathered rows), the down kernel for dL/dx, bwd_wgrad_kernel (tcgen05 with
// MN-major operands: the token rows are the reduction dimension), the
// router-gradient kernels and the Gram kernel. Every wait on an mbarrier is
// bounded; a wait that runs out records kStatusTimeout and the CTA unwinds.
#include <stdio.h>

#include "decide.cuh"
#include "internal.cuh"
#include "tc_common.cuh"

namespace unif {
namespace tc {
namespace bwd {

// GeLU (exact erf form, Sec. II-A) and its derivative Phi(a) + a phi(a),
// from one evaluation of Phi.
__device__ __forceinline__ void gelu_and_grad(float a, float& g, float& dg) {
  const float cdf = 0.5f * (1.0f + erff(a * 0.70710678118654752f));
  g = a * cdf;
  dg = cdf + a * 0.39894228040143268f * __expf(-0.5f * a * a);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Instruction descriptor of kind::f16 (bf16 in, fp32 accumulate) with both
// operands MN-major (transpose bits 15 and 16).
__device__ __forceinline__ uint32_t idesc_bf16_mn(int m, int n) {
  return idesc_bf16(m, n) | (1u << 15) | (1u << 16);
}

// Shared-memory descriptor of an MN-major operand with the 128-byte swizzle:
// each 128-byte row holds 64 consecutive MN elements of one K index, 8-row
// (K) groups are 1024 bytes apart (stride-dimension offset), and blocks of
// 64 MN elements are `lbo` bytes apart (leading-dimension offset).
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

constexpr int kThreads = 416;     // 13 warps
constexpr int kMmaWarp = 4;
constexpr int kFirstEpiWarp = 5;  // warps 5-12
constexpr int kEpiWarps = 8;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAcc2 = 256;   // TMEM column of the second accumulator

// ---------------------------------------------------------------------------
// bwd_hidden_kernel: per (tile, N sub-tile) item, over the forward's tile
// list, acc_a = X[rows] K_e[cols]^T and acc_g = DY[rows] V_e^T[cols]^T (both
// reductions over d), then the epilogue of the header comment.
// Roles: warps 0-3 fill a 4-deep ring of single-operand stages (even
// stages: 128 gathered x rows and the key tile; odd stages: dy rows and the
// value tile, so that each 64-deep k-block takes one stage of each; warp s
// owns stage s and its lane 0 brings the stage's weight tile by TMA); warp 4
// allocates TMEM and issues the MMAs; warps 5-12 run the epilogue (warp w
// reads TMEM lane quarter w % 4, one half of the columns).
// ---------------------------------------------------------------------------
struct HiddenParams {
  const int32_t* n_tiles;
  const int32_t* tile_group;
  const int32_t* tile_row0;
  const int32_t* tile_rows;
  const int32_t* row_tok;
  const float* row_w;
  const __nv_bfloat16* x;
  const __nv_bfloat16* dy;
  __nv_bfloat16* da;   // [rows][M]
  __nv_bfloat16* hw;   // [rows][M]
  float* dwt;          // [T][K+1]
  int n_sub, bn, num_kb, B, M, H, d, K1;
  int* status;
  long long wait_limit;
};

constexpr int kHStages = 4;

__host__ __device__ constexpr uint32_t hidden_stage_bytes(int bn) {
  return kStageA + (uint32_t)bn * kBK * 2u;
}

__global__ void __launch_bounds__(kThreads, 1)
bwd_hidden_kernel(const __grid_constant__ CUtensorMap tm_wk, const __grid_constant__ CUtensorMap tm_wv,
                  HiddenParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t stage_bytes = hidden_stage_bytes(p.bn);
  const uint32_t wtile = (uint32_t)p.bn * kBK * 2u;
  const uint32_t s0 = smem_u32(smem);
  // stage s: [128 rows x 64 (16 KB)][weight tile bn x 64]
  auto sa = [&](int s) { return s0 + s * stage_bytes; };
  auto sw = [&](int s) { return s0 + s * stage_bytes + kStageA; };
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kHStages * stage_bytes);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kHStages + s); };
  const uint32_t accf = bar0 + 8u * (2 * kHStages);
  const uint32_t acce = bar0 + 8u * (2 * kHStages + 1);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kHStages + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kHStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accf, 1);
    mbar_init(acce, kEpiWarps);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_items = p.n_tiles[0] * p.n_sub;

  if (warp < kHStages) {
    // ---- producers: warp s owns stage s (s even: x rows and key tiles, s
    // odd: dy rows and value tiles) ----
    const int my_stage = warp, kind = warp & 1;
    const __nv_bfloat16* src = kind == 0 ? p.x : p.dy;
    const CUtensorMap* tmw = kind == 0 ? &tm_wk : &tm_wv;
    const int j = lane & 7, rsub = lane >> 3;
    bool ok = true;
    int seq = 0;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const int tile = item / p.n_sub, ns = item % p.n_sub;
      const int g = p.tile_group[tile];
      const int e = g / p.B, blk = g % p.B;
      const int brow = e * p.H + blk * p.M + ns * p.bn;
      const int r0 = p.tile_row0[tile], nrow = p.tile_rows[tile];
      int tk[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        // padding rows gather token 0; their results are never kept
        const int t = 32 * i + lane < nrow ? p.row_tok[r0 + 32 * i + lane] : 0;
        tk[i] = t < 0 ? 0 : t;
      }
      // stage sequence: seq = 2 kb + kind over the item's k-blocks
      for (int ks = 0; ks < 2 * p.num_kb; ++ks, ++seq) {
        const int stage = seq % kHStages;
        if (stage != my_stage) continue;
        const int kb = ks >> 1;
        const uint32_t phase = (uint32_t)(seq / kHStages) & 1u;
        ok = wait_warp(empty_bar(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        if (lane == 0) {
          mbar_expect_tx_only(full_bar(stage), wtile);
          tma_load_2d(sw(stage), tmw, full_bar(stage), kb * kBK, brow);
        }
        const uint32_t dst = sa(stage);
        const __nv_bfloat16* sj = src + j * 8 + kb * kBK;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int r = 4 * i + rsub;
          const int t = __shfl_sync(0xffffffffu, tk[i >> 3], r & 31);
          cp_async16(dst + r * 128u + ((j ^ (r & 7)) << 4), sj + (size_t)t * p.d);
        }
        cp_async_commit();
        cp_async_wait<0>();
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(full_bar(stage));
      }
    }
  } else if (warp == kMmaWarp) {
    // ---- MMA issuer ----
    const uint32_t idesc = idesc_bf16(kBM, p.bn);
    int seq = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      ok = wait_warp(acce, acc_phase ^ 1u, abort_flag, p.status, p.wait_limit);
      if (!ok) break;
      tc_fence_after();
      for (int ks = 0; ks < 2 * p.num_kb; ++ks, ++seq) {
        const int stage = seq % kHStages;
        const uint32_t phase = (uint32_t)(seq / kHStages) & 1u;
        ok = wait_warp(full_bar(stage), phase, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        tc_fence_after();
        // even stages feed x K (acc_a), odd ones dy V^T (acc_g)
        const uint32_t d_tmem = tmem_base + ((ks & 1) ? kAcc2 : 0u);
        if (elect_one()) {
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16(d_tmem, sw128_desc(sa(stage) + k * 32), sw128_desc(sw(stage) + k * 32),
                      idesc, ((ks >> 1) | k) != 0 ? 1u : 0u);
          umma_commit(empty_bar(stage));
        }
        __syncwarp();
      }
      if (!ok) break;
      if (elect_one()) umma_commit(accf);
      __syncwarp();
      acc_phase ^= 1u;
    }
  } else if (warp >= kFirstEpiWarp) {
    // ---- epilogue ----
    const int q = warp & 3;
    const int half = (warp - kFirstEpiWarp) >> 2;
    const int cols = p.bn / 2;
    const int c_begin = half * cols;
    uint32_t acc_phase = 0;
    for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
      const int tile = item / p.n_sub, ns = item % p.n_sub;
      const int g = p.tile_group[tile];
      const int e = g / p.B;
      const int r = q * 32 + lane;
      const bool real = r < p.tile_rows[tile];
      const int tok = real ? p.row_tok[p.tile_row0[tile] + r] : -1;
      const float w = real ? p.row_w[p.tile_row0[tile] + r] : 0.f;
      if (!wait_warp(accf, acc_phase, abort_flag, p.status, p.wait_limit)) break;
      tc_fence_after();
      const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16);
      const size_t orow = ((size_t)tile * kBM + r) * p.M + ns * p.bn + c_begin;
      float dot = 0.f;
      for (int c = 0; c < cols; c += 16) {
        float a[16], gv[16];
        tmem_ld16(t_row + c_begin + c, a);
        tmem_ld16(t_row + kAcc2 + c_begin + c, gv);
        uint32_t od[8], oh[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float d0 = 0.f, d1 = 0.f, h0 = 0.f, h1 = 0.f;
          if (tok >= 0) {
            float g0, g1, dg0, dg1;
            gelu_and_grad(a[2 * i], g0, dg0);
            gelu_and_grad(a[2 * i + 1], g1, dg1);
            dot = fmaf(g0, gv[2 * i], dot);
            dot = fmaf(g1, gv[2 * i + 1], dot);
            d0 = w * gv[2 * i] * dg0;
            d1 = w * gv[2 * i + 1] * dg1;
            h0 = w * g0;
            h1 = w * g1;
          }
          od[i] = pack_bf16(d0, d1);
          oh[i] = pack_bf16(h0, h1);
        }
        // padding rows are written as zeros: the weight-gradient kernel sums
        // over whole tiles
        uint4* pd = reinterpret_cast<uint4*>(p.da + orow + c);
        uint4* ph = reinterpret_cast<uint4*>(p.hw + orow + c);
        pd[0] = make_uint4(od[0], od[1], od[2], od[3]);
        pd[1] = make_uint4(od[4], od[5], od[6], od[7]);
        ph[0] = make_uint4(oh[0], oh[1], oh[2], oh[3]);
        ph[1] = make_uint4(oh[4], oh[5], oh[6], oh[7]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce);
      if (tok >= 0) atomicAdd(p.dwt + (size_t)tok * p.K1 + e, dot);
      acc_phase ^= 1u;
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// bwd_wgrad_kernel: per item (group g, 128 features c of d, N chunk nc of the
// block's M channels) two accumulators over all rows of the group, 64 rows
// per stage:
//   acc1[i][h] = sum_r X[tok_r][c*128 + i] DA[r][nc*N + h]   -> dK_e (transposed)
//   acc2[i][h] = sum_r DY[tok_r][c*128 + i] HW[r][nc*N + h]  -> dV_e
// The token rows are the reduction dimension, so both operands are MN-major:
// the gathered rows (x, dy) and the TMA tiles (DA, HW) keep the 128-byte
// swizzled row layout, read with MN-major descriptors. A group's rows are
// split into chunks of kChunkTiles tiles, one work item each, whose partial
// sums are added into the (zeroed) outputs.
// Roles: warps 0-3 fill the 4-deep ring (warp s: the x and dy rows of stage
// s, and the DA/HW tiles by TMA), warp 4 MMAs, warps 5-12 epilogue.
// ---------------------------------------------------------------------------
struct WgradParams {
  const int32_t* counts;   // [G] group sizes (the forward's)
  const int32_t* row_tok;  // per-group regions of `region` rows
  const __nv_bfloat16* x;
  const __nv_bfloat16* dy;
  float* dw_up;    // [K+1][H][d]
  float* dw_down;  // [K+1][d][H]
  int G, region, B, M, H, d, N, n_nc, n_c;
  int* status;
  long long wait_limit;
};

constexpr uint32_t kRows = 32;                 // group rows per stage
constexpr uint32_t kPBytes = 2u * kRows * 128u;  // 128 features x 32 rows (two 64-column blocks)
constexpr int kWStages = 4;                      // one stage per producer warp
constexpr int kQuarters = kBM / (int)kRows;      // stages per 128-row tile
constexpr int kChunkTiles = 8;                   // tiles of a group per work item

__host__ __device__ constexpr uint32_t wgrad_stage_bytes(int N) {
  return 2u * kPBytes + 2u * (uint32_t)(N / 64) * kRows * 128u;
}

__global__ void __launch_bounds__(kThreads, 1)
bwd_wgrad_kernel(const __grid_constant__ CUtensorMap tm_da, const __grid_constant__ CUtensorMap tm_hw,
                 WgradParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t stage_bytes = wgrad_stage_bytes(p.N);
  const uint32_t qbytes = (uint32_t)(p.N / 64) * kRows * 128u;
  const uint32_t s0 = smem_u32(smem);
  // stage s: [x rows][dy rows][DA tile][HW tile]
  auto spx = [&](int s) { return s0 + s * stage_bytes; };
  auto spy = [&](int s) { return s0 + s * stage_bytes + kPBytes; };
  auto sqa = [&](int s) { return s0 + s * stage_bytes + 2 * kPBytes; };
  auto sqh = [&](int s) { return s0 + s * stage_bytes + 2 * kPBytes + qbytes; };
  uint8_t* gen_base = smem;  // generic pointer for zero-filling padding rows
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWStages * stage_bytes);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kWStages + s); };
  const uint32_t accf = bar0 + 8u * (2 * kWStages);
  const uint32_t acce = bar0 + 8u * (2 * kWStages + 1);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kWStages + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int32_t* first_s = reinterpret_cast<int32_t*>(tmem_slot + 4);  // [G + 1] first tiles
  int32_t* cnt_s = first_s + p.G + 1;                             // [G] sizes
  int32_t* chunk_s = cnt_s + p.G;                                 // [G + 1] first chunks

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kWStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accf, 1);
    mbar_init(acce, kEpiWarps);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  if (warp == kThreads / 32 - 1) {
    tile_table(p.counts, p.G, p.region, lane, first_s, cnt_s);
    __syncwarp();
    // each group's tiles in chunks of kChunkTiles: the first chunk of every
    // group (chunk_s[G] = all chunks)
    int carry = 0;
    for (int g0 = 0; g0 < p.G; g0 += 32) {
      const int g = g0 + lane;
      const int nch = g < p.G ? (first_s[g + 1] - first_s[g] + kChunkTiles - 1) / kChunkTiles : 0;
      int inc = nch;
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += v;
      }
      if (g < p.G) chunk_s[g] = carry + inc - nch;
      carry += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (lane == 0) chunk_s[p.G] = carry;
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_items = chunk_s[p.G] * p.n_c * p.n_nc;
  // item -> (group g, its tiles [t0, t0 + nt) of one chunk, feature chunk c,
  // N chunk nc); rows of the chunk start at row r0 of the group
  auto decode = [&](int item, int& g, int& t0, int& nt, int& r0, int& c, int& nc) {
    nc = item % p.n_nc;
    c = (item / p.n_nc) % p.n_c;
    const int q = item / (p.n_nc * p.n_c);
    int lo = 0, hi = p.G - 1;  // the last group whose first chunk is <= q
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (chunk_s[mid] <= q) lo = mid; else hi = mid - 1;
    }
    g = lo;
    const int k = q - chunk_s[g];
    t0 = first_s[g] + k * kChunkTiles;
    nt = min(kChunkTiles, first_s[g + 1] - t0);
    r0 = k * kChunkTiles * kBM;
  };

  if (warp < kWStages) {
    // ---- producers: warp w owns stage w: the x and dy rows of its 32 group
    // rows, and lane 0 brings the DA and HW tiles by TMA ----
    const int my_stage = warp;
    const int j = lane & 7, rsub = lane >> 3;
    bool ok = true;
    int seq = 0;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      int g, t_first, nt, r0, c, nc;
      decode(item, g, t_first, nt, r0, c, nc);
      const int size = cnt_s[g];
      for (int kt = 0; kt < nt * kQuarters && ok; ++kt, ++seq) {  // 32-row quarters of the tiles
        const int stage = seq % kWStages;
        if (stage != my_stage) continue;
        const uint32_t phase = (uint32_t)(seq / kWStages) & 1u;
        ok = wait_warp(empty_bar(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        const int row_in_group = r0 + kt * (int)kRows;  // first row of this quarter in the group
        const int crow = (t_first + kt / kQuarters) * kBM + (kt % kQuarters) * (int)kRows;
        if (lane == 0) {
          mbar_expect_tx_only(full_bar(stage), 2u * qbytes);
          for (int b = 0; b < p.N / 64; ++b) {
            tma_load_2d(sqa(stage) + b * kRows * 128u, &tm_da, full_bar(stage), nc * p.N + b * 64,
                        crow);
            tma_load_2d(sqh(stage) + b * kRows * 128u, &tm_hw, full_bar(stage), nc * p.N + b * 64,
                        crow);
          }
        }
        // this quarter's row tokens: lane l holds row l (-1: padding)
        const int rg = row_in_group + lane;
        const int tk = rg < size ? p.row_tok[(size_t)g * p.region + rg] : -1;
#pragma unroll
        for (int kind = 0; kind < 2; ++kind) {
          const uint32_t dst = kind == 0 ? spx(stage) : spy(stage);
          const __nv_bfloat16* sj = (kind == 0 ? p.x : p.dy) + (size_t)c * 128 + j * 8;
#pragma unroll
          for (int b = 0; b < 2; ++b) {
#pragma unroll
            for (int i = 0; i < (int)kRows / 4; ++i) {
              const int r = 4 * i + rsub;
              const int t = __shfl_sync(0xffffffffu, tk, r);
              const uint32_t off = b * kRows * 128u + r * 128u + ((j ^ (r & 7)) << 4);
              if (t >= 0)
                cp_async16(dst + off, sj + (size_t)t * p.d + b * 64);
              else  // padding rows contribute zeros to the row sums
                *reinterpret_cast<uint4*>(gen_base + (dst - s0) + off) = make_uint4(0u, 0u, 0u, 0u);
            }
          }
        }
        cp_async_commit();
        cp_async_wait<0>();
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(full_bar(stage));
      }
    }
  } else if (warp == kMmaWarp) {
    const uint32_t idesc = idesc_bf16_mn(kBM, p.N);
    const uint32_t lbo = kRows * 128u;  // 64-element MN blocks of kRows rows
    int seq = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      int g, t_first, nt, r0, c, nc;
      decode(item, g, t_first, nt, r0, c, nc);
      ok = wait_warp(acce, acc_phase ^ 1u, abort_flag, p.status, p.wait_limit);
      if (!ok) break;
      tc_fence_after();
      for (int kt = 0; kt < nt * kQuarters; ++kt, ++seq) {
        const int stage = seq % kWStages;
        const uint32_t phase = (uint32_t)(seq / kWStages) & 1u;
        ok = wait_warp(full_bar(stage), phase, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        tc_fence_after();
        if (elect_one()) {
#pragma unroll
          for (int k = 0; k < (int)kRows / 16; ++k) {  // 16 rows (two 8-row groups) per MMA
            const uint32_t acc = (kt | k) != 0 ? 1u : 0u;
            umma_bf16(tmem_base, sw128_mn_desc(spx(stage) + k * 2048u, lbo),
                      sw128_mn_desc(sqa(stage) + k * 2048u, lbo), idesc, acc);
            umma_bf16(tmem_base + kAcc2, sw128_mn_desc(spy(stage) + k * 2048u, lbo),
                      sw128_mn_desc(sqh(stage) + k * 2048u, lbo), idesc, acc);
          }
          umma_commit(empty_bar(stage));
        }
        __syncwarp();
      }
      if (!ok) break;
      if (elect_one()) umma_commit(accf);
      __syncwarp();
      acc_phase ^= 1u;
    }
  } else if (warp >= kFirstEpiWarp) {
    const int q = warp & 3;
    const int half = (warp - kFirstEpiWarp) >> 2;
    const int cols = p.N / 2;
    uint32_t acc_phase = 0;
    for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
      int g, t_first, nt, r0, c, nc;
      decode(item, g, t_first, nt, r0, c, nc);
      const int e = g / p.B, blk = g % p.B;
      const int i = c * 128 + q * 32 + lane;  // this thread's feature
      const int h0 = blk * p.M + nc * p.N + half * cols;  // first channel of its columns
      float* up_col = p.dw_up + ((size_t)e * p.H + h0) * p.d + i;   // dK_e[h][i], stride d per h
      float* dn_row = p.dw_down + ((size_t)e * p.d + i) * p.H + h0;  // dV_e[i][h], contiguous
      if (!wait_warp(accf, acc_phase, abort_flag, p.status, p.wait_limit)) break;
      tc_fence_after();
      const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) + half * cols;
      // the chunks of a group add their partial sums (the outputs start at zero)
      for (int cc = 0; cc < cols; cc += 32) {
        float v[32];
        tmem_ld32(t_row + cc, v);
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) atomicAdd(up_col + (size_t)(cc + jj) * p.d, v[jj]);
        tmem_ld32(t_row + kAcc2 + cc, v);
#pragma unroll
        for (int jj = 0; jj < 32; jj += 4)
          atomicAdd(reinterpret_cast<float4*>(dn_row + cc + jj),
                    make_float4(v[jj], v[jj + 1], v[jj + 2], v[jj + 3]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce);
      acc_phase ^= 1u;
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Router gradients (Eqs. 17, 18, 24)
// ---------------------------------------------------------------------------
// dL/dz of token t into z[0..KC) (K + 1 <= KC values, the rest and a padding
// token's all zero): dL/dz_0 = dL/dalpha (1 - 2 tau) sigma(z_0)(1 - sigma(z_0))
// (adaptive alpha; sigma(z_0) = (alpha - tau) / (1 - 2 tau) from the stored
// alpha), dL/dz_{1+j} = s_j (dL/ds_j - sum_l s_l dL/ds_l), from the pathway
// weights' gradients dL/dalpha, dL/ds_j that the hidden kernel accumulated.
// All of the token's loads go out before the arithmetic.
template <int KC>
__device__ __forceinline__ void router_token_dz(int t, int K, float tau, int adaptive,
                                                const uint8_t* __restrict__ mask,
                                                const float* __restrict__ alpha,
                                                const float* __restrict__ s,
                                                const float* __restrict__ dwt, float (&z)[KC]) {
  const int K1 = K + 1;
  const bool valid = !mask || mask[t];
  const float* st = s + (size_t)t * K;
  const float* gt = dwt + (size_t)t * K1;
  float sv[KC], gv[KC];
#pragma unroll
  for (int j = 0; j < KC; ++j) {
    sv[j] = valid && j < K ? st[j] : 0.f;
    gv[j] = valid && j < K1 ? gt[j] : 0.f;
  }
  const float al = valid ? alpha[t] : 0.f;
  float part = 0.f;
#pragma unroll
  for (int j = 0; j + 1 < KC; ++j) part += sv[j] * gv[1 + j];
  z[0] = 0.f;
  if (valid && adaptive && tau < 0.5f) {
    const float sg = (al - tau) / (1.0f - 2.0f * tau);
    z[0] = gv[0] * (1.0f - 2.0f * tau) * sg * (1.0f - sg);
  }
#pragma unroll
  for (int j = 0; j + 1 < KC; ++j) z[1 + j] = sv[j] * (gv[1 + j] - part);
}

// dL/dz of every token into dz [T][K+1] (a thread per token).
template <int KC>
__global__ void __launch_bounds__(256)
router_dz_kernel(int T, int K, float tau, int adaptive, const uint8_t* __restrict__ mask,
                 const float* __restrict__ alpha, const float* __restrict__ s,
                 const float* __restrict__ dwt, float* __restrict__ dz) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  float z[KC];
  router_token_dz<KC>(t, K, tau, adaptive, mask, alpha, s, dwt, z);
  float* o = dz + (size_t)t * (K + 1);
#pragma unroll
  for (int c = 0; c < KC; ++c)
    if (c <= K) o[c] = z[c];
}

// dx[t][8 f .. 8 f + 8) += sum_c dL/dz_c(t) W*^T[c][8 f .. 8 f + 8) for the
// two tokens t = 2 p, 2 p + 1: a thread per (token pair, 8 features), so that
// each W*^T load serves both tokens. W*^T is the router's first K+1 columns
// as fp32 [K+1][d]; d % 128 == 0; padding tokens have dL/dz = 0 and keep dx.
__global__ void __launch_bounds__(256)
router_dx_kernel(int T, int K1, int d, const float* __restrict__ dz,
                 const float* __restrict__ wrT, float* __restrict__ dx) {
  const int per = d / 8;
  const int n = ((T + 1) / 2) * per;
  for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < n; it += gridDim.x * blockDim.x) {
    const int p = it / per, f8 = it - p * per;
    const int ta = 2 * p, tb = min(2 * p + 1, T - 1);  // (tb == ta: the last odd token)
    float4* pa = reinterpret_cast<float4*>(dx + (size_t)ta * d + 8 * f8);
    float4* pb = reinterpret_cast<float4*>(dx + (size_t)tb * d + 8 * f8);
    const float4 xa0 = pa[0], xa1 = pa[1], xb0 = pb[0], xb1 = pb[1];  // added at the end
    const float* za = dz + (size_t)ta * K1;
    const float* zb = dz + (size_t)tb * K1;
    float4 a0 = make_float4(0.f, 0.f, 0.f, 0.f), a1 = a0, b0 = a0, b1 = a0;
    // four columns at a time: their loads go out together
    for (int cb = 0; cb < K1; cb += 4) {
      float4 w0[4], w1[4];
      float u[4], v[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int c = cb + k;
        if (c < K1) {
          const float4* wc = reinterpret_cast<const float4*>(wrT + (size_t)c * d + 8 * f8);
          w0[k] = wc[0];
          w1[k] = wc[1];
          u[k] = za[c];
          v[k] = zb[c];
        } else {
          w0[k] = w1[k] = make_float4(0.f, 0.f, 0.f, 0.f);
          u[k] = v[k] = 0.f;
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        a0.x = fmaf(u[k], w0[k].x, a0.x); a0.y = fmaf(u[k], w0[k].y, a0.y);
        a0.z = fmaf(u[k], w0[k].z, a0.z); a0.w = fmaf(u[k], w0[k].w, a0.w);
        a1.x = fmaf(u[k], w1[k].x, a1.x); a1.y = fmaf(u[k], w1[k].y, a1.y);
        a1.z = fmaf(u[k], w1[k].z, a1.z); a1.w = fmaf(u[k], w1[k].w, a1.w);
        b0.x = fmaf(v[k], w0[k].x, b0.x); b0.y = fmaf(v[k], w0[k].y, b0.y);
        b0.z = fmaf(v[k], w0[k].z, b0.z); b0.w = fmaf(v[k], w0[k].w, b0.w);
        b1.x = fmaf(v[k], w1[k].x, b1.x); b1.y = fmaf(v[k], w1[k].y, b1.y);
        b1.z = fmaf(v[k], w1[k].z, b1.z); b1.w = fmaf(v[k], w1[k].w, b1.w);
      }
    }
    a0.x += xa0.x; a0.y += xa0.y; a0.z += xa0.z; a0.w += xa0.w;
    a1.x += xa1.x; a1.y += xa1.y; a1.z += xa1.z; a1.w += xa1.w;
    b0.x += xb0.x; b0.y += xb0.y; b0.z += xb0.z; b0.w += xb0.w;
    b1.x += xb1.x; b1.y += xb1.y; b1.z += xb1.z; b1.w += xb1.w;
    pa[0] = a0;
    pa[1] = a1;
    if (tb != ta) {
      pb[0] = b0;
      pb[1] = b1;
    }
  }
}

// dL/dW*[i][c] = sum_t x[t][i] dL/dz_c(t) and dL/dbias[c] = sum_t dL/dz_c(t):
// block (fc, j, cc) takes features [128 fc, 128 fc + 128), the tokens of
// slice j (kRwSlice tokens) and columns [16 cc, 16 cc + 16); 32 tokens at a
// time, the tile of x (16-byte loads; zero rows for padding tokens, whose x
// may hold anything) and of dL/dz go to shared memory (the next tile's
// loads run while the current tile is summed), then thread (g, q)
// adds x[t][2 q .. 2 q + 2) times dL/dz_{16 cc + 4 g .. + 4}(t) into its
// 2 x 4 partial sums (one 4-byte and one 16-byte shared load per 8 FMAs),
// which go out with one atomic add each.
constexpr int kRwSlice = 128;
__global__ void __launch_bounds__(256)
router_dw_kernel(int T, int K1, int d, const uint8_t* __restrict__ mask,
                 const __nv_bfloat16* __restrict__ x, const float* __restrict__ dz,
                 float* __restrict__ dw_router, float* __restrict__ dbias) {
  __shared__ __align__(16) __nv_bfloat16 xs[32][128];
  __shared__ __align__(16) float zs[32][16];
  const int i0 = blockIdx.x * 128, c0 = blockIdx.z * 16;
  const int t_begin = blockIdx.y * kRwSlice, t_end = min(T, t_begin + kRwSlice);
  const int q = threadIdx.x & 63, g = threadIdx.x >> 6;
  const int lq = threadIdx.x & 15, lr = threadIdx.x >> 4;
  float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
  float bacc[4] = {0.f, 0.f, 0.f, 0.f};
  // this thread's share of a tile: 16-byte chunk lq of x rows lr, lr + 16
  // and column c0 + lq of dL/dz for the same two tokens; the next tile's
  // share is loaded into registers while the current one is summed
  uint4 xr[2];
  float zr[2];
  auto load = [&](int tt) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int t = tt + lr + 16 * k, c = c0 + lq;
      xr[k] = make_uint4(0u, 0u, 0u, 0u);
      if (t < t_end && (!mask || mask[t]))
        xr[k] = reinterpret_cast<const uint4*>(x + (size_t)t * d + i0)[lq];
      zr[k] = t < t_end && c < K1 ? dz[(size_t)t * K1 + c] : 0.f;
    }
  };
  load(t_begin);
  for (int tt = t_begin; tt < t_end; tt += 32) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      reinterpret_cast<uint4*>(&xs[lr + 16 * k][0])[lq] = xr[k];
      zs[lr + 16 * k][lq] = zr[k];
    }
    __syncthreads();
    if (tt + 32 < t_end) load(tt + 32);
    const int nr = min(32, t_end - tt);
    for (int r = 0; r < nr; ++r) {
      const float2 xv = __bfloat1622float2(reinterpret_cast<const __nv_bfloat162*>(&xs[r][0])[q]);
      const float4 z = reinterpret_cast<const float4*>(&zs[r][0])[g];
      acc[0][0] = fmaf(xv.x, z.x, acc[0][0]); acc[0][1] = fmaf(xv.x, z.y, acc[0][1]);
      acc[0][2] = fmaf(xv.x, z.z, acc[0][2]); acc[0][3] = fmaf(xv.x, z.w, acc[0][3]);
      acc[1][0] = fmaf(xv.y, z.x, acc[1][0]); acc[1][1] = fmaf(xv.y, z.y, acc[1][1]);
      acc[1][2] = fmaf(xv.y, z.z, acc[1][2]); acc[1][3] = fmaf(xv.y, z.w, acc[1][3]);
      if (q == 0) {
        bacc[0] += z.x; bacc[1] += z.y; bacc[2] += z.z; bacc[3] += z.w;
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int c = c0 + 4 * g + e;
    if (c < K1) {
      atomicAdd(dw_router + (size_t)(i0 + 2 * q) * K1 + c, acc[0][e]);
      atomicAdd(dw_router + (size_t)(i0 + 2 * q + 1) * K1 + c, acc[1][e]);
      if (dbias && blockIdx.x == 0 && q == 0) atomicAdd(dbias + c, bacc[e]);
    }
  }
}

// W*^T: the router's first K+1 columns (fp32 [d][Cp]) as [K+1][d].
__global__ void router_transpose_kernel(int K1, int d, int Cp, const float* __restrict__ wr,
                                        float* __restrict__ wrT) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k < K1 * d) {
    const int c = k / d, i = k % d;
    wrT[k] = wr[(size_t)i * Cp + c];
  }
}

// Gram regulariser (Eq. diversity-loss): A = W*^T W* - I over the K+1
// router columns (one block per entry, reduced over d), then L_div = ||A||_F
// and dW* += lambda 2 W* A / L_div (nothing where L_div = 0), W*^T as
// [K+1][d] fp32.
__global__ void __launch_bounds__(128)
gram_kernel(int K1, int d, const float* __restrict__ wrT, float* __restrict__ A) {
  __shared__ float red[4];
  const int a = blockIdx.x / K1, b = blockIdx.x % K1;
  float g = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x)
    g = fmaf(wrT[(size_t)a * d + i], wrT[(size_t)b * d + i], g);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = g;
  __syncthreads();
  if (threadIdx.x == 0) A[blockIdx.x] = red[0] + red[1] + red[2] + red[3] - (a == b ? 1.f : 0.f);
}

__global__ void __launch_bounds__(256)
diversity_grad_kernel(int K1, int d, const float* __restrict__ wrT, const float* __restrict__ A,
                      float lambda, float* __restrict__ dw_router, float* __restrict__ l_out) {
  __shared__ float red[8];
  float ss = 0.f;
  for (int k = threadIdx.x; k < K1 * K1; k += blockDim.x) ss = fmaf(A[k], A[k], ss);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += red[w];
  const float L = sqrtf(tot);
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k == 0 && l_out) *l_out = L;
  if (k >= d * K1 || !(L > 0.f) || lambda == 0.f || !dw_router) return;
  const int i = k / K1, b = k % K1;
  float g = 0.f;
  for (int a = 0; a < K1; ++a) g = fmaf(wrT[(size_t)a * d + i], A[a * K1 + b], g);
  dw_router[k] += 2.f * lambda / L * g;
}

// out[e][c][r] = in[e][r][c] for bf16 [E][R][C] (32 x 32 tiles through shared
// memory).
__global__ void transpose_bf16_kernel(const __nv_bfloat16* __restrict__ in,
                                      __nv_bfloat16* __restrict__ out, int R, int C) {
  __shared__ __nv_bfloat16 tile[32][33];
  const size_t base = (size_t)blockIdx.z * R * C;
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int k = threadIdx.y; k < 32; k += blockDim.y) {
    const int r = r0 + k, c = c0 + threadIdx.x;
    if (r < R && c < C) tile[k][threadIdx.x] = in[base + (size_t)r * C + c];
  }
  __syncthreads();
  for (int k = threadIdx.y; k < 32; k += blockDim.y) {
    const int c = c0 + k, r = r0 + threadIdx.x;
    if (r < R && c < C) out[base + (size_t)c * R + r] = tile[threadIdx.x][k];
  }
}

}  // namespace bwd
}  // namespace tc

// ---- host side ----

int backward_setup(unif_moe_layer* L) {
  using namespace tc::bwd;
  const uint64_t E = (uint64_t)L->K + 1;
  Workspace& w = L->ws;
  if (!encode_bf16_map(&L->tm_wdownT, w.w_downT, L->d, E * L->H, tc::kBK, L->up_bn, 128) ||
      !encode_bf16_map(&L->tm_wupT, w.w_upT, L->H, E * L->d, tc::kBK, L->down_bn, 128) ||
      !encode_bf16_map(&L->tm_da, w.da, L->M, (uint64_t)L->max_rows, tc::kBK, tc::kBM, 128) ||
      !encode_bf16_map(&L->tm_da_q, w.da, L->M, (uint64_t)L->max_rows, tc::kBK, kRows, 128) ||
      !encode_bf16_map(&L->tm_hw_q, w.hw, L->M, (uint64_t)L->max_rows, tc::kBK, kRows, 128)) {
    set_error("cuTensorMapEncodeTiled failed for the backward maps");
    return UNIF_MOE_ERR_CUDA;
  }
  L->bwd_hidden_smem = 1024 + kHStages * hidden_stage_bytes(L->up_bn) + 256;
  L->bwd_wgrad_smem =
      1024 + kWStages * wgrad_stage_bytes(L->up_bn) + 96 + 4 * (3 * (uint32_t)L->G + 2) + 16;
  if (L->bwd_hidden_smem > 232448 || L->bwd_wgrad_smem > 232448) {
    set_error("backward: shared memory for block width %d and %d groups exceeds 227 KB", L->M,
              L->G);
    return UNIF_MOE_ERR_SHAPE;
  }
  if (cudaFuncSetAttribute(bwd_hidden_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)L->bwd_hidden_smem) != cudaSuccess ||
      cudaFuncSetAttribute(bwd_wgrad_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)L->bwd_wgrad_smem) != cudaSuccess ) {
    set_error("cudaFuncSetAttribute failed for the backward kernels");
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

cudaError_t launch_transpose_weights(unif_moe_layer* L, cudaStream_t s) {
  using namespace tc::bwd;
  const int E = L->K + 1;
  dim3 blk(32, 8);
  // w_up [E][H][d] -> w_upT [E][d][H]; w_down [E][d][H] -> w_downT [E][H][d]
  transpose_bf16_kernel<<<dim3((L->d + 31) / 32, (L->H + 31) / 32, E), blk, 0, s>>>(
      static_cast<const __nv_bfloat16*>(L->w_up), static_cast<__nv_bfloat16*>(L->ws.w_upT), L->H,
      L->d);
  transpose_bf16_kernel<<<dim3((L->H + 31) / 32, (L->d + 31) / 32, E), blk, 0, s>>>(
      static_cast<const __nv_bfloat16*>(L->w_down), static_cast<__nv_bfloat16*>(L->ws.w_downT),
      L->d, L->H);
  return cudaGetLastError();
}

int backward_run(unif_moe_layer* L, const void* x, const void* dy, int T, const uint8_t* mask,
                 float* dx, float* dw_up, float* dw_down, float* dw_router, float* dbias,
                 float lambda_div, float* l_div, cudaStream_t s) {
  using namespace tc::bwd;
  Workspace& w = L->ws;
  const int K1 = L->K + 1;
#define CKB(call)                                                               \
  do {                                                                          \
    cudaError_t e_ = (call);                                                    \
    if (e_ != cudaSuccess) {                                                    \
      set_error("%s failed: %s", #call, cudaGetErrorString(e_));                \
      return UNIF_MOE_ERR_CUDA;                                                 \
    }                                                                           \
  } while (0)
  CKB(cudaMemsetAsync(dx, 0, sizeof(float) * (size_t)T * L->d, s));
  CKB(cudaMemsetAsync(w.dwt, 0, sizeof(float) * (size_t)T * K1, s));
  CKB(cudaMemsetAsync(dw_router, 0, sizeof(float) * (size_t)L->d * K1, s));
  if (dbias) CKB(cudaMemsetAsync(dbias, 0, sizeof(float) * K1, s));
  // tile list of the forward's groups (sizes in grp_cnt, rows in the regions)
  CKB(launch_tile_list_from(L, w.grp_cnt, s));
  // hidden gradients
  {
    HiddenParams p;
    p.n_tiles = w.n_tiles; p.tile_group = w.tile_group; p.tile_row0 = w.tile_row0;
    p.tile_rows = w.tile_rows; p.row_tok = w.row_tok; p.row_w = w.row_w;
    p.x = static_cast<const __nv_bfloat16*>(x);
    p.dy = static_cast<const __nv_bfloat16*>(dy);
    p.da = static_cast<__nv_bfloat16*>(w.da);
    p.hw = static_cast<__nv_bfloat16*>(w.hw);
    p.dwt = w.dwt;
    p.n_sub = L->up_nsub; p.bn = L->up_bn; p.num_kb = L->d / tc::kBK;
    p.B = L->B; p.M = L->M; p.H = L->H; p.d = L->d; p.K1 = K1;
    p.status = w.status;
    p.wait_limit = gemm_wait_limit();
    bwd_hidden_kernel<<<L->n_sm, kThreads, L->bwd_hidden_smem, s>>>(L->tm_wup, L->tm_wdownT, p);
    CKB(cudaGetLastError());
  }
  // dL/dx from the experts: DA K_e (the down kernel on the transposed keys)
  CKB(launch_down_streaming(L, L->tm_da, L->tm_wupT, nullptr, dx, s));
  // dL/dK_e and dL/dV_e (chunks of each group's rows add their parts)
  CKB(cudaMemsetAsync(dw_up, 0, sizeof(float) * (size_t)K1 * L->H * L->d, s));
  CKB(cudaMemsetAsync(dw_down, 0, sizeof(float) * (size_t)K1 * L->H * L->d, s));
  {
    WgradParams p;
    p.counts = w.grp_cnt; p.row_tok = w.row_tok;
    p.x = static_cast<const __nv_bfloat16*>(x);
    p.dy = static_cast<const __nv_bfloat16*>(dy);
    p.dw_up = dw_up; p.dw_down = dw_down;
    p.G = L->G; p.region = L->region_rows; p.B = L->B; p.M = L->M; p.H = L->H; p.d = L->d;
    p.N = L->up_bn; p.n_nc = L->up_nsub; p.n_c = L->d / 128;
    p.status = w.status;
    p.wait_limit = gemm_wait_limit();
    bwd_wgrad_kernel<<<L->n_sm, kThreads, L->bwd_wgrad_smem, s>>>(L->tm_da_q, L->tm_hw_q, p);
    CKB(cudaGetLastError());
  }
  // router: W*^T, then dL/dz, its share of dL/dx, dL/dW* and dL/dbias
  router_transpose_kernel<<<(K1 * L->d + 255) / 256, 256, 0, s>>>(K1, L->d, L->router_cols_pad,
                                                                   L->wr, w.wrT);
  CKB(cudaGetLastError());
  {
    const int adaptive = isnan(L->th.alpha_fixed) ? 1 : 0;
    const int dz_blocks = (T + 255) / 256;
    if (K1 <= 16)
      router_dz_kernel<16><<<dz_blocks, 256, 0, s>>>(T, L->K, L->tau, adaptive, mask, w.alpha,
                                                     w.s, w.dwt, w.dz);
    else if (K1 <= 32)
      router_dz_kernel<32><<<dz_blocks, 256, 0, s>>>(T, L->K, L->tau, adaptive, mask, w.alpha,
                                                     w.s, w.dwt, w.dz);
    else
      router_dz_kernel<65><<<dz_blocks, 256, 0, s>>>(T, L->K, L->tau, adaptive, mask, w.alpha,
                                                     w.s, w.dwt, w.dz);
    CKB(cudaGetLastError());
    const int items = (T + 1) / 2 * (L->d / 8);
    router_dx_kernel<<<std::min((items + 255) / 256, 8 * L->n_sm), 256, 0, s>>>(T, K1, L->d,
                                                                                 w.dz, w.wrT, dx);
    CKB(cudaGetLastError());
    router_dw_kernel<<<dim3(L->d / 128, (T + kRwSlice - 1) / kRwSlice, (K1 + 15) / 16), 256, 0,
                       s>>>(T, K1, L->d, mask, static_cast<const __nv_bfloat16*>(x), w.dz,
                            dw_router, dbias);
    CKB(cudaGetLastError());
  }
  if (lambda_div != 0.f || l_div) {
    gram_kernel<<<K1 * K1, 128, 0, s>>>(K1, L->d, w.wrT, w.gram);
    CKB(cudaGetLastError());
    diversity_grad_kernel<<<(L->d * K1 + 255) / 256, 256, 0, s>>>(K1, L->d, w.wrT, w.gram,
                                                                  lambda_div, dw_router, l_div);
    CKB(cudaGetLastError());
  }
#undef CKB
  return UNIF_MOE_OK;
}

}  // namespace unif
