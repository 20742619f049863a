// Grouped expert GEMMs on the sm_103a tensor cores (tcgen05 + TMEM, fed by
// TMA) for bf16 layers.
//
// Every (expert e, block b) pair of Eqs. 28-29 is one group; the permute step
// lists each group's rows (token, weight) contiguously, padded to 128-row
// tiles. Two persistent, warp-specialised kernels walk that tile list:
//   up   : h[row]  = GeLU(x[tok(row)] K_e[:, H_b])        128 x M  per tile
//   down : y[tok] += w(row) * h[row] V_e[H_b, :]          128 x d  per tile
// (Eq. 16 split at the activation; w = alpha for the shared expert and p_i
// for residual expert q_i, Eq. 30).
//
// Roles inside one CTA (one CTA per SM, 416 threads):
//   warps 0-3   up kernel: warp p owns the ring stages s = p (mod 4); it
//               gathers the stage's 128 token rows of x with 16-byte cp.async
//               into the swizzled operand layout, brings the weight tile with
//               TMA, and signals the stage as soon as its own copies landed
//   warp 0      down kernel: TMA of the h tile and the weight tile
//   warp 4      TMEM allocator and MMA issuer (one lane): 128 x BN x 16
//               kind::f16 MMAs, fp32 accumulators in TMEM
//   warps 5-12  epilogue: tcgen05.ld of the accumulator, GeLU -> bf16 h
//               (up), or weight-scale -> fp32 atomic add into y (down)
// Shared-memory stages are a 4-deep ring (full/empty mbarriers); the TMEM
// accumulator is double-buffered (2 x 256 columns) so the epilogue of one
// tile overlaps the MMAs of the next.
//
// Operands use the 128-byte-swizzled K-major layout: a stage row holds 64
// bf16 (128 bytes) of the reduction dimension, 8-row groups are 1024 bytes
// apart, and the MMA's 16-element K steps advance the descriptor start
// address by 32 bytes inside the swizzle atom.
//
// Every wait on an mbarrier is bounded; a wait that runs out records
// kStatusTimeout in the handle's status word and the CTA unwinds.
#include <stdio.h>

#include "decide.cuh"
#include "internal.cuh"
#include "tc_common.cuh"

namespace unif {
namespace tc {

constexpr int kThreads = 416;     // 13 warps
constexpr int kProducerWarps = 4;  // warps 0-3
constexpr int kMmaWarp = 4;        // TMEM allocation and MMA issue
constexpr int kEpiWarps = 8;
constexpr int kFirstEpiWarp = 5;   // warps 5-12 (warp % 4 covers every TMEM lane quarter twice)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccStride = 256;  // TMEM columns per accumulator buffer
constexpr int kMaxBN = 256;
constexpr uint32_t kStageB = kMaxBN * kBK * 2;   // 32 KB
constexpr int kStageRow = 36;                    // fp32 per staged row (32 + 4 pad, 16 B aligned)
constexpr uint32_t kHStageRow = 80;              // bytes per staged h row (64 + 16 pad)

// Per-kernel shared memory: the up kernel keeps 4 operand stages; the down
// kernel keeps 3 and a per-warp 32 x 32 fp32 staging tile that turns its
// row-per-thread accumulator into row-contiguous, coalesced atomic adds.
template <int MODE>
struct Cfg {
  static constexpr int kStages = MODE == 0 ? 4 : 3;
  // up: 32 rows x 32 bf16 per warp (80-byte rows); down: 32 rows x 32 fp32
  static constexpr uint32_t kStaging =
      MODE == 0 ? kEpiWarps * 32u * kHStageRow : kEpiWarps * 32u * kStageRow * 4u;
  static constexpr uint32_t kTokens = MODE == 0 ? kProducerWarps * kBM * 4u : 0u;
  static constexpr size_t kSmem = 1024 + kStages * (kStageA + kStageB) + kStaging + kTokens + 256;
};

struct Params {
  const int32_t* n_tiles;
  const int32_t* tile_group;
  const int32_t* tile_row0;
  const int32_t* tile_rows;  // rows of each tile that are not padding
  const int32_t* row_tok;
  const float* row_w;
  int n_sub;       // N sub-tiles per 128-row tile
  int bn;          // N per sub-tile (multiple of 64, <= 256)
  int num_kb;      // reduction steps of 64
  int B, M, H, d;
  const __nv_bfloat16* x;  // up: tokens [T][d] (rows gathered with cp.async)
  __nv_bfloat16* h;  // up: [rows][M]
  float* y32;        // down: [T][d]
  int* status;
  long long wait_limit;  // clock cycles before a wait gives up
};

// MODE 0 = up-projection (+GeLU), MODE 1 = down-projection (+weighted add).
template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    Params p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived from smem_raw by an offset so that the
  // compiler keeps every access through it in the shared state space
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  constexpr int kStages = Cfg<MODE>::kStages;
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + kStages * kStageA;
  float* staging = reinterpret_cast<float*>(smem + kStages * (kStageA + kStageB));
  int* tok_smem = reinterpret_cast<int*>(smem + kStages * (kStageA + kStageB) + Cfg<MODE>::kStaging);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * (kStageA + kStageB) +
                                               Cfg<MODE>::kStaging + Cfg<MODE>::kTokens);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
  auto accf_bar = [&](int a) { return bar0 + 8u * (2 * kStages + a); };
  auto acce_bar = [&](int a) { return bar0 + 8u * (2 * kStages + 2 + a); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(accf_bar(a), 1);
      mbar_init(acce_bar(a), kEpiWarps);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  __syncwarp();  // every warp converged before the CTA barrier
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_items = p.n_tiles[0] * p.n_sub;
  // Bytes the TMA brings per stage (the up kernel gathers A with cp.async).
  const uint32_t stage_bytes = (MODE == 0 ? 0u : kStageA) + (uint32_t)p.bn * kBK * 2;

  if (MODE == 0 && warp < kProducerWarps) {
    // ------------------- producers (up): stage owners ----------------------
    // Warp p handles the stages whose sequence number is p mod 4. For its
    // stage it copies the 128 token rows (instruction i covers rows
    // 4 i .. 4 i + 3, one 16-byte chunk per lane, so each instruction reads 4
    // whole 128-byte rows), waits for its own copies, fences them for the
    // tensor cores (async proxy) and signals the stage. Lane 0 also brings the
    // stage's weight tile with TMA.
    static_assert(Cfg<0>::kStages == kProducerWarps, "one ring stage per producer warp");
    const int j = lane & 7, rsub = lane >> 3;
    int seq = 0;  // stage sequence number over all items of this CTA
    bool ok = true;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const int tile = item / p.n_sub, ns = item % p.n_sub;
      // does this warp own any stage of this item?
      int first = (warp - seq % kProducerWarps + kProducerWarps) % kProducerWarps;
      if (first >= p.num_kb) { seq += p.num_kb; continue; }
      const int g = p.tile_group[tile];
      const int e = g / p.B, blk = g % p.B;
      const int brow = e * p.H + blk * p.M + ns * p.bn;
      // this tile's 128 row tokens, in the warp's own shared-memory slot
      int* tok = tok_smem + warp * kBM;
      const int r0 = p.tile_row0[tile], nrow = p.tile_rows[tile];
      __syncwarp();
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        // padding rows: token 0, unused
        const int t = 32 * i + lane < nrow ? p.row_tok[r0 + 32 * i + lane] : 0;
        tok[32 * i + lane] = t < 0 ? 0 : t;
      }
      __syncwarp();
      const __nv_bfloat16* xj = p.x + j * 8;
      for (int kb = first; kb < p.num_kb; kb += kProducerWarps) {
        const int sq = seq + kb;
        const int stage = sq % kProducerWarps;  // == warp
        const uint32_t phase = (uint32_t)(sq / kProducerWarps) & 1u;
        ok = wait_warp(empty_bar(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        if (lane == 0) {
          mbar_expect_tx_only(full_bar(stage), stage_bytes);
          tma_load_2d(sB + stage * kStageB, &tmB, full_bar(stage), kb * kBK, brow);
        }
        const uint32_t a_dst = sA + stage * kStageA;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int r = 4 * i + rsub;
          cp_async16(a_dst + r * 128u + ((j ^ (r & 7)) << 4), xj + (size_t)tok[r] * p.d + kb * kBK);
        }
        cp_async_commit();
        cp_async_wait<0>();
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(full_bar(stage));
      }
      seq += p.num_kb;
    }
  } else if (MODE == 1 && warp == 0) {
    // ------------------- producer (down): h tile and weight tile ------------
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    int g_nxt = (blockIdx.x < n_items) ? p.tile_group[blockIdx.x / p.n_sub] : 0;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const int tile = item / p.n_sub, ns = item % p.n_sub;
      const int g = g_nxt, row0 = tile * kBM;
      if (item + (int)gridDim.x < n_items) g_nxt = p.tile_group[(item + gridDim.x) / p.n_sub];
      const int e = g / p.B, blk = g % p.B;
      const int brow = e * p.d + ns * p.bn;  // w_down viewed [(K+1)d][H]
      for (int kb = 0; kb < p.num_kb; ++kb) {
        ok = wait_warp(empty_bar(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        if (lane == 0) {
          mbar_expect_tx(full_bar(stage), stage_bytes);
          tma_load_2d(sA + stage * kStageA, &tmA, full_bar(stage), kb * kBK, row0);
          tma_load_2d(sB + stage * kStageB, &tmB, full_bar(stage), blk * p.M + kb * kBK, brow);
        }
        __syncwarp();
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------ MMA issuer ----------------------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kBM, p.bn);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        if (!wait_bounded(acce_bar(acc), acc_phase ^ 1u, abort_flag, p.status, p.wait_limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)acc * kAccStride;
        for (int kb = 0; kb < p.num_kb; ++kb) {
          if (!wait_bounded(full_bar(stage), phase, abort_flag, p.status, p.wait_limit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = sA + stage * kStageA, b_base = sB + stage * kStageB;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16(d_tmem, sw128_desc(a_base + k * 32), sw128_desc(b_base + k * 32), idesc,
                      (kb | k) != 0 ? 1u : 0u);
          umma_commit(empty_bar(stage));
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit(accf_bar(acc));
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      }
    }
    __syncwarp();
  } else if (warp >= kFirstEpiWarp) {
    // ------------------------------ epilogue ------------------------------
    const int q = warp & 3;                        // TMEM lane quarter of this warp
    const int half = (warp - kFirstEpiWarp) >> 2;  // which half of the columns
    const int cols = p.bn / 2;
    int acc = 0;
    uint32_t acc_phase = 0;
    // down: this thread's row token and weight, fetched one tile ahead
    int t_nxt = -1;
    float w_nxt = 0.f;
    // (row_w == nullptr: every row's weight is 1)
    if (MODE == 1 && blockIdx.x < n_items &&
        q * 32 + lane < p.tile_rows[blockIdx.x / p.n_sub]) {
      const int r = p.tile_row0[blockIdx.x / p.n_sub] + q * 32 + lane;
      t_nxt = p.row_tok[r];
      w_nxt = p.row_w ? p.row_w[r] : 1.f;
    }
    for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
      const int tile = item / p.n_sub, ns = item % p.n_sub;
      const int row0 = tile * kBM;
      const int t_cur = t_nxt;
      const float w_cur = w_nxt;
      if (MODE == 1 && item + (int)gridDim.x < n_items) {
        const int nt = (item + gridDim.x) / p.n_sub;
        const int r = p.tile_row0[nt] + q * 32 + lane;
        const bool real = q * 32 + lane < p.tile_rows[nt];
        t_nxt = real ? p.row_tok[r] : -1;
        w_nxt = real ? (p.row_w ? p.row_w[r] : 1.f) : 0.f;
      }
      if (!wait_warp(accf_bar(acc), acc_phase, abort_flag, p.status, p.wait_limit)) break;
      tc_fence_after();
      const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)acc * kAccStride;
      const int c_begin = half * cols;
      if (MODE == 0) {
        // h = bf16(GeLU(acc)), 32 columns per TMEM load. Each thread stages its
        // row's 64 bytes; the warp then stores 8 rows x 64 contiguous bytes per
        // instruction.
        uint8_t* stg = reinterpret_cast<uint8_t*>(staging) +
                       (size_t)(warp - kFirstEpiWarp) * 32 * kHStageRow;
        __nv_bfloat16* hrow0 = p.h + (size_t)(row0 + q * 32) * p.M + ns * p.bn + c_begin;
        for (int c = 0; c < cols; c += 32) {
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {  // two 16-column TMEM loads keep register use low
            float v[16];
            tmem_ld16(t_row + c_begin + c + 16 * hh, v);
            uint32_t o[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) o[jj] = gelu2_bf16x2(v[2 * jj], v[2 * jj + 1]);
#pragma unroll
            for (int jj = 0; jj < 2; ++jj)
              *reinterpret_cast<uint4*>(stg + lane * kHStageRow + 32 * hh + 16 * jj) =
                  make_uint4(o[4 * jj], o[4 * jj + 1], o[4 * jj + 2], o[4 * jj + 3]);
          }
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int r = 8 * i + (lane >> 2), seg = lane & 3;
            *reinterpret_cast<uint4*>(hrow0 + (size_t)r * p.M + c + seg * 8) =
                *reinterpret_cast<const uint4*>(stg + r * kHStageRow + 16 * seg);
          }
          __syncwarp();
        }
      } else {
        // y[tok] += w * acc: each thread scales its row, the warp stages 32 rows x
        // 32 columns in shared memory and adds them back row-contiguously (8 lanes
        // x 16 B per row, 4 rows per instruction).
        float* stg = staging + (size_t)(warp - kFirstEpiWarp) * 32 * kStageRow;
        const int t = t_cur;
        const float wt = w_cur;
        const int r_sub = lane >> 3, c_sub = (lane & 7) * 4;
        for (int c = 0; c < cols; c += 32) {
          float v[32];
          tmem_ld32(t_row + c_begin + c, v);
#pragma unroll
          for (int j = 0; j < 32; j += 4)
            *reinterpret_cast<float4*>(stg + lane * kStageRow + j) =
                make_float4(wt * v[j], wt * v[j + 1], wt * v[j + 2], wt * v[j + 3]);
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int r = 4 * i + r_sub;
            const int tr = __shfl_sync(0xffffffffu, t, r);
            const float4 val = *reinterpret_cast<const float4*>(stg + r * kStageRow + c_sub);
            if (tr >= 0)
              atomicAdd(reinterpret_cast<float4*>(p.y32 + (size_t)tr * p.d + ns * p.bn + c_begin +
                                                  c + c_sub),
                        val);
          }
          __syncwarp();
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce_bar(acc));
      if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
    }
  }
  __syncwarp();  // every warp converged before the CTA barrier
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// A kernel that waits, with the same bounded wait, on a barrier that nothing
// completes: exercises the timeout path without hanging.
__global__ void timeout_probe_kernel(int* status, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(smem_u32(&bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    wait_bounded(smem_u32(&bar), 0u, &abort_flag, status, limit);
  }
}

// ---------------------------------------------------------------------------
// Router on the tensor cores (bf16 layers)
// ---------------------------------------------------------------------------
// One CTA per R tokens (R = 32, 64, 96 or 128, chosen per call so that the
// grid fits on the SMs in one wave): z = x [W_shr | W_g | mu] as a 128 x Cp
// x d MMA (Eqs. 17, 21; rows past R are computed and never read), TMA-fed,
// fp32 accumulator in TMEM. Each decision warp then owns 32 tokens = 32
// TMEM lanes: a thread reads its token's Cp logits, takes the decisions of
// Eqs. 18-27 and the warp counts its chunk's (expert, block) pairs.
constexpr int kRtThreads = 192;   // warp 0 TMA, warp 1 TMEM + MMA, warps 2-5 decisions
constexpr int kRtStages = 6;
constexpr uint32_t kRtStageB = 160u * kBK * 2;  // up to 160 router columns
constexpr size_t kRtSmem = 1024 + kRtStages * (kStageA + kRtStageB) + 256;
constexpr int kRtRingBytes = kRtStages * (kStageA + kRtStageB);

// Bytes of the operand ring that the decision warps reuse once the MMAs are
// done: logits [128][Cp + 1] and decision scratch [128][2K + 1] (fp32), lane
// masks [4][128], and (grouping) group_rows' counters.
__host__ __device__ constexpr int router_overlay_bytes(int Cp, int K, int G, bool fused) {
  return 4 * (kBM * (Cp + 1) + kBM * (2 * K + 1) + 4 * 128) +
         (fused ? 4 * group_rows_smem_ints(4, G) : 0);
}

struct RouterTcParams {
  DecideArgs dec;
  GroupArgs grp;
  int fused;     // 1: the router also lays out the group rows by (expert, block)
                 // (group_rows); 2: by expert (group_rows_expert)
  int d, Cp;
  int rows;      // tokens per CTA: 32, 64, 96 or 128 (the MMA always spans 128
                 // rows; the rows past the tile are never read back)
  uint32_t tmem_cols;
  int* status;
  long long wait_limit;
};

__global__ void __launch_bounds__(kRtThreads, 1)
router_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                 RouterTcParams p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived from smem_raw by an offset so that the
  // compiler keeps every access through it in the shared state space
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + kRtStages * kStageA;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kRtStages * (kStageA + kRtStageB));
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kRtStages + s); };
  const uint32_t accf = bar0 + 8u * (2 * kRtStages);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kRtStages + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int R = p.rows;
  const int t0 = blockIdx.x * R;
  const int Cp = p.Cp, K = p.dec.K;
  // the up projection may start its prologue on SMs this grid leaves free
  grid_dep_launch();

  if (threadIdx.x == 0) {
    for (int s = 0; s < kRtStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), p.tmem_cols);
    tmem_relinquish();
  }
  __syncwarp();  // every warp converged before the CTA barrier
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int num_kb = p.d / kBK;
  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      const uint32_t bytes = (uint32_t)(R + Cp) * kBK * 2;  // the x box (R rows) and the router box
      for (int kb = 0; kb < num_kb; ++kb) {
        if (!wait_bounded(empty_bar(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit)) break;
        mbar_expect_tx(full_bar(stage), bytes);
        tma_load_2d(sA + stage * kStageA, &tm_x, full_bar(stage), kb * kBK, t0);
        tma_load_2d(sB + stage * kRtStageB, &tm_w, full_bar(stage), kb * kBK, 0);
        if (++stage == kRtStages) { stage = 0; phase ^= 1u; }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kBM, Cp);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int kb = 0; kb < num_kb; ++kb) {
        if (!wait_bounded(full_bar(stage), phase, abort_flag, p.status, p.wait_limit)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = sA + stage * kStageA, b_base = sB + stage * kRtStageB;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          umma_bf16(tmem_base, sw128_desc(a_base + k * 32), sw128_desc(b_base + k * 32), idesc,
                    (kb | k) != 0 ? 1u : 0u);
        umma_commit(empty_bar(stage));
        if (++stage == kRtStages) { stage = 0; phase ^= 1u; }
      }
      if (ok) umma_commit(accf);
    }
    __syncwarp();
  } else {
    // decision warps: lane quarter q = warp % 4 holds tokens t0 + 32 q + lane.
    const int q = warp & 3;
    const int row = q * 32 + lane;
    // logits and affinities overlay the (now idle) operand ring
    float* zs = reinterpret_cast<float*>(smem);
    float* ss = zs + kBM * (Cp + 1);                                      // [128][2K + 1]
    uint32_t* cscr = reinterpret_cast<uint32_t*>(ss + kBM * (2 * K + 1));  // [4][128]
    float* sv = ss + row * (2 * K + 1);
    const int t = t0 + row;
    uint64_t shr = 0ull, em = 0ull;
    float alpha = 0.f;
    const int G = p.grp.G;
    int32_t* gsm = reinterpret_cast<int32_t*>(cscr + 4 * 128);  // group_rows' counters
    int32_t* misc_s = gsm + group_rows_smem_ints(4, G) - 8;
    // a warp whose quarter lies past the CTA's R tokens takes no decisions
    // (those token indices belong to the next CTA) and counts nothing
    const bool in_tile = q * 32 < R;
    if (wait_warp(accf, 0u, abort_flag, p.status, p.wait_limit)) {
      tc_fence_after();
      if (in_tile) {
        float* z = zs + row * (Cp + 1);
        for (int c = 0; c < Cp; c += 32) {
          float v[32];
          tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + c, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) z[c + i] = v[i];
        }
        const bool valid = t < p.dec.T && (p.dec.mask == nullptr || p.dec.mask[t] != 0);
        decide_token(p.dec, t, valid, z, sv, shr, em, alpha);
      }
      const int chunk = blockIdx.x * (R / 32) + q;
      if (!p.fused) {
        if (in_tile && chunk < p.dec.n_chunks)
          count_chunk_pairs(p.dec, lane, shr, em, cscr + q * 128,
                            p.dec.chunk_cnt + chunk, p.dec.n_chunks);
      } else {
        // per-chunk counts stay in shared memory (chunk q = tokens
        // 32 q .. 32 q + 31 of this CTA); alpha joins the affinities
        if (p.fused == 2)
          count_chunk_experts(K, lane, shr, em, cscr + q * 128, gsm + q * G, 1);
        else
          count_chunk_pairs(p.dec, lane, shr, em, cscr + q * 128, gsm + q * G, 1);
        sv[2 * K] = alpha;
      }
    }
    if (p.fused) {
      // all four decision warps meet here, also when a wait gave up (which
      // sets the abort flag for all of them), then place this CTA's rows
      named_bar(1, 128);
      if (row == 0) misc_s[7] = *abort_flag;  // one reading for all four warps
      named_bar(1, 128);
      if (!misc_s[7]) {
        if (p.fused == 2)
          group_rows_expert<4>(p.grp, row, t0, shr, em, cscr, ss, 2 * K + 1, gsm, 1);
        else
          group_rows<4>(p.grp, row, t0, shr, em, cscr, ss, 2 * K + 1, gsm, 1);
      }
    }
  }
  __syncwarp();  // every warp converged before the CTA barrier
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// ---- host side ----

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// 2-D bf16 tensor map [rows][cols] (cols contiguous), 128-byte swizzle.
bool encode_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows,
               uint32_t box_cols, uint32_t box_rows) {
  return encode_bf16_map(map, base, cols, rows, box_cols, box_rows, 128);
}

}  // namespace tc

// 2-D bf16 tensor map [rows][cols] (cols contiguous) with a 32-, 64- or
// 128-byte swizzle.
bool encode_bf16_map(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows,
                     uint32_t box_cols, uint32_t box_rows, int swizzle_bytes) {
  tc::EncodeTiledFn fn = tc::encode_fn();
  if (!fn) return false;
  const CUtensorMapSwizzle sw = swizzle_bytes == 32   ? CU_TENSOR_MAP_SWIZZLE_32B
                                : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                      : CU_TENSOR_MAP_SWIZZLE_128B;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace tc {

// N split into n_sub sub-tiles of bn columns: bn <= 256 and bn % 64 == 0, so
// that each of the two epilogue column halves is a whole number of 32-column
// TMEM loads.
bool pick_split(int n, int* bn, int* nsub) {
  for (int s = 1; s <= n / 64; ++s) {
    if (n % s) continue;
    const int b = n / s;
    if (b <= kMaxBN && b % 64 == 0) {
      *bn = b;
      *nsub = s;
      return true;
    }
  }
  return false;
}

long long g_wait_limit = 4000000000ll;  // ~2 s of SM clock

}  // namespace tc

long long gemm_wait_limit() { return tc::g_wait_limit; }

int gemm_tc_setup(unif_moe_layer* L) {
  if (!tc::pick_split(L->M, &L->up_bn, &L->up_nsub) ||
      !tc::pick_split(L->d, &L->down_bn, &L->down_nsub)) {
    set_error("no tensor-core tile split for M=%d or d=%d", L->M, L->d);
    return UNIF_MOE_ERR_SHAPE;
  }
  const uint64_t E = (uint64_t)L->K + 1;
  if (!tc::encode_2d(&L->tm_wup, L->w_up, L->d, E * L->H, tc::kBK, L->up_bn) ||
      !tc::encode_2d(&L->tm_wdown, L->w_down, L->H, E * L->d, tc::kBK, L->down_bn) ||
      !tc::encode_2d(&L->tm_h, L->ws.hbuf, L->M, (uint64_t)L->max_rows, tc::kBK, tc::kBM)) {
    set_error("cuTensorMapEncodeTiled failed for the weight or activation maps");
    return UNIF_MOE_ERR_CUDA;
  }
  cudaError_t e = cudaFuncSetAttribute(tc::grouped_gemm_kernel<0>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)tc::Cfg<0>::kSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc::grouped_gemm_kernel<1>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc::Cfg<1>::kSmem);
  if (e != cudaSuccess) {
    set_error("cudaFuncSetAttribute: %s", cudaGetErrorString(e));
    return UNIF_MOE_ERR_CUDA;
  }
  const int rc = gemm_ws_setup(L);
  L->tile_list = L->fused_group && !L->ffn_fused && !(L->up_ws && L->down_ws);
  return rc;
}

cudaError_t launch_gemms_tc(unif_moe_layer* L, const void* x, int T, cudaEvent_t mid,
                            cudaStream_t s) {
  (void)T;
  if (L->ffn_fused) {  // both projections in one kernel (the down stage takes no time)
    cudaError_t e = launch_ffn_fused(L, x, s);
    if (e == cudaSuccess && mid) e = cudaEventRecord(mid, s);
    return e;
  }
  tc::Params p;
  p.n_tiles = L->ws.n_tiles; p.tile_group = L->ws.tile_group; p.tile_row0 = L->ws.tile_row0;
  p.tile_rows = L->ws.tile_rows;
  p.row_tok = L->ws.row_tok; p.row_w = L->ws.row_w;
  p.B = L->B; p.M = L->M; p.H = L->H; p.d = L->d;
  p.x = static_cast<const __nv_bfloat16*>(x);
  p.h = static_cast<__nv_bfloat16*>(L->ws.hbuf);
  p.y32 = L->ws.y32;
  p.status = L->ws.status;
  p.wait_limit = tc::g_wait_limit;
  // up: N = M (block width), reduction over d
  p.n_sub = L->up_nsub; p.bn = L->up_bn; p.num_kb = L->d / tc::kBK;
  cudaError_t e;
  if (L->up_ws) {
    e = launch_up_ws(L, x, s);
  } else {
    tc::grouped_gemm_kernel<0><<<L->n_sm, tc::kThreads, tc::Cfg<0>::kSmem, s>>>(L->tm_h,
                                                                               L->tm_wup, p);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) return e;
  if (mid) cudaEventRecord(mid, s);
  // down: N = d, reduction over the block's M channels
  if (L->down_ws) return launch_down_ws(L, s);
  p.n_sub = L->down_nsub; p.bn = L->down_bn; p.num_kb = L->M / tc::kBK;
  tc::grouped_gemm_kernel<1><<<L->n_sm, tc::kThreads, tc::Cfg<1>::kSmem, s>>>(L->tm_h, L->tm_wdown,
                                                                             p);
  return cudaGetLastError();
}

// The streaming down-projection kernel on other operands: out[tok] +=
// w(row) * A[row] B_e[H_b, :] over the tile list, A an [rows][M] bf16 map
// like h's and B a [(K+1) d][H] bf16 map like w_down's; row_w == nullptr
// gives every row weight 1 (the backward's dL/dx = dL/da K_e^T).
cudaError_t launch_down_streaming(unif_moe_layer* L, const CUtensorMap& tmA,
                                  const CUtensorMap& tmB, const float* row_w, float* out,
                                  cudaStream_t s) {
  tc::Params p;
  p.n_tiles = L->ws.n_tiles; p.tile_group = L->ws.tile_group; p.tile_row0 = L->ws.tile_row0;
  p.tile_rows = L->ws.tile_rows;
  p.row_tok = L->ws.row_tok; p.row_w = row_w;
  p.B = L->B; p.M = L->M; p.H = L->H; p.d = L->d;
  p.x = nullptr;
  p.h = nullptr;
  p.y32 = out;
  p.status = L->ws.status;
  p.wait_limit = tc::g_wait_limit;
  p.n_sub = L->down_nsub; p.bn = L->down_bn; p.num_kb = L->M / tc::kBK;
  tc::grouped_gemm_kernel<1><<<L->n_sm, tc::kThreads, tc::Cfg<1>::kSmem, s>>>(tmA, tmB, p);
  return cudaGetLastError();
}

bool router_can_group(int Cp, int K, int G) {
  return tc::router_overlay_bytes(Cp, K, G, true) <= tc::kRtRingBytes;
}

int router_tc_setup(unif_moe_layer* L) {
  if (L->router_cols_pad > 160 || L->d % tc::kBK != 0) {
    set_error("tensor-core router needs 1+K+B <= 160 and d %% 64 == 0");
    return UNIF_MOE_ERR_SHAPE;
  }
  if (!tc::encode_2d(&L->tm_wr, L->wr_bf, L->d, L->router_cols_pad, tc::kBK,
                     L->router_cols_pad)) {
    set_error("cuTensorMapEncodeTiled failed for the router matrix");
    return UNIF_MOE_ERR_CUDA;
  }
  if (cudaFuncSetAttribute(tc::router_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)tc::kRtSmem) != cudaSuccess) {
    set_error("cudaFuncSetAttribute failed for the router kernel");
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

cudaError_t launch_router_tc(unif_moe_layer* L, const void* x, const uint8_t* mask, int T,
                             int32_t* b_out, int32_t* k_out, cudaStream_t s) {
  // Tokens per CTA: the smallest multiple of 32 whose grid still fits in one
  // wave on the SMs (the x load is bound per SM: spreading the tokens over
  // more SMs shortens it), else 128.
  int R = tc::kBM;
  for (int r = 32; r < tc::kBM; r += 32)
    if ((T + r - 1) / r <= L->n_sm) { R = r; break; }
  CUtensorMap tm_x;
  if (!tc::encode_2d(&tm_x, x, L->d, (uint64_t)T, tc::kBK, (uint32_t)R)) return cudaErrorInvalidValue;
  tc::RouterTcParams p;
  p.dec = decide_args(L, mask, T, b_out, k_out);
  p.fused = L->fused_group ? (L->ffn_fused ? 2 : 1) : 0;
  if (L->fused_group) {
    Workspace& w = L->ws;
    GroupArgs& g = p.grp;
    g.G = L->ffn_fused ? L->K + 1 : L->G; g.K = L->K; g.B = L->B;
    g.region = L->region_rows;
    g.fill = w.grp_fill;
    g.row_tok = w.row_tok; g.row_w = w.row_w;
    g.status = w.status;
  }
  p.d = L->d;
  p.Cp = L->router_cols_pad;
  p.rows = R;
  p.tmem_cols = p.Cp <= 32 ? 32u : (p.Cp <= 64 ? 64u : (p.Cp <= 128 ? 128u : 256u));
  p.status = L->ws.status;
  p.wait_limit = tc::g_wait_limit;
  tc::router_tc_kernel<<<(T + R - 1) / R, tc::kRtThreads, tc::kRtSmem, s>>>(
      tm_x, L->tm_wr, p);
  return cudaGetLastError();
}

cudaError_t launch_timeout_probe(unif_moe_layer* L, int timeout_us, cudaStream_t s) {
  int khz = 0;
  cudaError_t e = cudaDeviceGetAttribute(&khz, cudaDevAttrClockRate, L->device);
  if (e != cudaSuccess) return e;
  if (timeout_us > 1000000) timeout_us = 1000000;
  if (timeout_us < 1) timeout_us = 1;
  const long long limit = (long long)timeout_us * (long long)khz / 1000ll;
  tc::timeout_probe_kernel<<<1, 32, 0, s>>>(L->ws.status, limit);
  return cudaGetLastError();
}

}  // namespace unif
