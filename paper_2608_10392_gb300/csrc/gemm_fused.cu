// Expert-tile FFN (tcgen05 + TMEM) for bf16 layers with d <= 384: both
// projections of Eq. 16 for 128 rows of one expert's token list in one CTA,
// h kept on chip.
//
// The router groups the rows by expert (group e = expert e, one row per
// (token, expert) the token runs, weight alpha or s_j; Eqs. 28-30). A tile
// is 128 rows of one group. For each 128-channel chunk c of the expert's H
// channels the CTA computes
//   U = x K_e[c]^T                        (tcgen05, M=128, N=128, K=d; TMEM)
//   h = bf16(GeLU(U)), zero in the columns of blocks the row does not run
//   D += h V_e[:, c]^T                    (tcgen05, M=128, N=d, K=128; TMEM)
// and after the last chunk adds w D into the fp32 output accumulator, once
// per (token, expert) instead of once per (token, expert, block). Each
// token's x row is gathered once per expert it runs, and h never leaves
// the SM. The blocks a row does not run are computed and masked, so the
// tensor work is that of the whole expert: B (1 + k) blocks per token
// against the C_B = b + k (B - b) the method activates (Eq. 35).
//
// Shared memory: the x tile (128 x d bf16, resident for the tile), h of one
// chunk (128 x 128 bf16, two 64-column halves), a ring of 16 KB weight slabs
// (128 rows x 64 reduction elements: K_e rows of a chunk, or 128 output
// rows of V_e for 64 channels), and the drain warps' staging tiles. The
// weights are repacked at load time into those slabs, each 16 KB contiguous
// and already in the 128-byte-swizzled operand layout, so that a slab
// arrives as one bulk copy (a tensor-map load of the same slab from the
// [rows][d] weights moves 128 separate 128-byte rows).
// TMEM (512 columns): D in columns [0, d), U in [384, 512).
//
// Roles (one CTA per SM, 18 warps):
//   warps 0-3    gather the tile's x rows (16-byte cp.async, 32 rows each)
//   warp 4       weight slabs by TMA, in the order the MMAs consume them
//   warp 5       MMA issue (one elected lane) and the TMEM allocation
//   warps 6-13   chunk epilogue: U -> GeLU -> masked bf16 h in shared memory
//                (warp w: TMEM lane quarter w % 4, 64-column half (w-6)/4)
//   warps 14-17  drain: w D -> fp32 atomic adds into the accumulator
// Order of the MMAs in a tile: up(0), up(1), down(0), up(2), down(1), ...,
// up(n-1), down(n-2), down(n-1), so that the epilogue of chunk c runs while
// the tensor pipe computes down(c-1) and up(c+1). Every wait is bounded; a
// wait that runs out records kStatusTimeout in the status word and the CTA
// unwinds.
#include <stdio.h>

#include "decide.cuh"
#include "internal.cuh"
#include "tc_common.cuh"

namespace unif {
namespace tc {
namespace fused {

constexpr int kChunk = 128;           // H channels per chunk (the up MMA's N)
constexpr int kPiece = 128;           // output columns per down MMA (its N)
constexpr uint32_t kSlab = 16384;     // 128 rows x 64 bf16
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kUCol = 384;       // U's first TMEM column
constexpr int kMaxKb = 6;             // d <= 384
constexpr int kMaxSlots = 12;
constexpr int kGatherWarps = 4;
constexpr int kLoaderWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kFirstEpi = 6;
constexpr int kEpiWarps = 8;
constexpr int kFirstDrain = 14;
constexpr int kDrainWarps = 4;
constexpr int kThreads = 32 * (kFirstDrain + kDrainWarps);  // 576
constexpr uint32_t kStaging = kDrainWarps * 32u * 128u;       // 32 x 32 fp32 per drain warp
constexpr uint32_t kBarBytes = 512;
constexpr uint32_t kMaxSmem = 232448;

struct Params {
  const int32_t* fill;     // [G] rows per expert group (final once the router completed)
  int G, region, per_cta;  // G = K + 1 groups of `region` rows; tile run capacity
  const int32_t* row_tok;  // [G][region] pass-relative token of each row
  const float* row_w;      // [G][region] the row's pathway weight
  const uint64_t* shr;     // [T] shared block set of each token of the pass
  const uint8_t* wk;       // up slabs [K+1][H/128][d/64] (repack_up_kernel)
  const uint8_t* wv;       // down slabs [K+1][H/128][2][d/128] (repack_down_kernel)
  int d, H, M, B;
  int n_chunks, num_kb, n_pieces, slots;
  const __nv_bfloat16* x;  // [T][d] the pass's tokens
  float* y32;              // [T][d] fp32 output accumulator of the pass
  int* status;
  long long wait_limit;
};

// Bytes of dynamic shared memory for num_kb reduction blocks of x and
// `slots` weight slabs (plus the tile table of G groups and per_cta tiles).
__host__ __device__ constexpr uint32_t smem_bytes(int num_kb, int slots, int G, int per_cta) {
  return 1024u + (uint32_t)num_kb * kSlab + 2u * kSlab + (uint32_t)slots * kSlab + kStaging +
         kBarBytes + (uint32_t)((2 * G + 1 + 3 * per_cta) * 4 + 15) / 16u * 16u;
}

// cp.async.wait_group with a run-time count of groups allowed in flight.
__device__ __forceinline__ void cp_async_wait_n(int n) {
  switch (n) {
    case 0: cp_async_wait<0>(); break;
    case 1: cp_async_wait<1>(); break;
    case 2: cp_async_wait<2>(); break;
    case 3: cp_async_wait<3>(); break;
    case 4: cp_async_wait<4>(); break;
    default: cp_async_wait<5>(); break;
  }
}

// A bounded wait that ignores the abort flag: a role that gave up still
// lets the copies and MMAs it started land before the CTA exits.
__device__ __forceinline__ void wait_settle(uint32_t bar, uint32_t parity, long long limit) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > limit) return;
}

__global__ void __launch_bounds__(kThreads, 1)
ffn_fused_kernel(Params p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived from smem_raw by an offset so that the
  // compiler keeps every access through it in the shared state space
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int num_kb = p.num_kb, nch = p.n_chunks, npc = p.n_pieces;
  const uint32_t sX = smem_u32(smem);
  const uint32_t sH = sX + (uint32_t)num_kb * kSlab;
  const uint32_t sW = sH + 2u * kSlab;
  uint8_t* stg_base = smem + (size_t)(num_kb + 2 + p.slots) * kSlab;
  uint64_t* bars = reinterpret_cast<uint64_t*>(stg_base + kStaging);
  const uint32_t bar0 = smem_u32(bars);
  auto xfull = [&](int kb) { return bar0 + 8u * kb; };
  const uint32_t xempty = bar0 + 8u * 6;
  auto wfull = [&](int s) { return bar0 + 8u * (7 + s); };
  auto wempty = [&](int s) { return bar0 + 8u * (19 + s); };
  const uint32_t ufull = bar0 + 8u * 31, uempty = bar0 + 8u * 32;
  auto hsfull = [&](int h) { return bar0 + 8u * (33 + h); };
  auto hsempty = [&](int h) { return bar0 + 8u * (35 + h); };
  const uint32_t dfull = bar0 + 8u * 37, dempty = bar0 + 8u * 38;
  const uint32_t mma_done = bar0 + 8u * 39;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 40);
  static_assert(8 * 40 + 8 <= kBarBytes, "barrier region");
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // tile table: first tile and size of every group, then (group, first
  // row, real rows) of each tile of this CTA's run
  int32_t* first_s = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(bars) + kBarBytes);
  int32_t* gcnt_s = first_s + p.G + 1;
  int32_t* run_s = gcnt_s + p.G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int kb = 0; kb < kMaxKb; ++kb) mbar_init(xfull(kb), kGatherWarps);
    mbar_init(xempty, 1);
    for (int s = 0; s < kMaxSlots; ++s) {
      mbar_init(wfull(s), 1);
      mbar_init(wempty(s), 1);
    }
    mbar_init(ufull, 1);
    mbar_init(uempty, kEpiWarps);
    for (int h = 0; h < 2; ++h) {
      mbar_init(hsfull(h), kEpiWarps / 2);
      mbar_init(hsempty(h), 1);
    }
    mbar_init(dfull, 1);
    mbar_init(dempty, kDrainWarps);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  if (warp == kLoaderWarp) {
    // the group sizes are final once the router completed
    grid_dep_wait();
    tile_table(p.fill, p.G, p.region, lane, first_s, gcnt_s);
    __syncwarp();
    const int nt = first_s[p.G];
    const int tb = (int)(((long long)blockIdx.x * nt) / gridDim.x);
    const int te = (int)(((long long)(blockIdx.x + 1) * nt) / gridDim.x);
    for (int k = tb + lane; k < te; k += 32) {
      int g, r0, rows;
      tile_lookup(k, first_s, gcnt_s, p.G, p.region, g, r0, rows);
      run_s[k - tb] = g;
      run_s[p.per_cta + k - tb] = r0;
      run_s[2 * p.per_cta + k - tb] = rows;
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();
  grid_dep_launch();
  const int nt = first_s[p.G];
  const int t_begin = (int)(((long long)blockIdx.x * nt) / gridDim.x);
  const int n_run = (int)(((long long)(blockIdx.x + 1) * nt) / gridDim.x) - t_begin;
  const uint64_t full = p.B >= 64 ? ~0ull : ((1ull << p.B) - 1ull);
  // Each CTA walks the chunks of a tile from its own starting chunk: the
  // CTAs working on one expert at the same time then read different weight
  // slabs (reading the same 16 KB at once from many SMs concentrates the
  // requests on a few L2 slices). D's sum over the chunks is the same in
  // any order up to the order of the fp32 additions.
  const int rot = (int)(blockIdx.x % (unsigned)nch);
  auto chunk_of = [&](int c) { return c + rot < nch ? c + rot : c + rot - nch; };

  if (warp < kGatherWarps) {
    // ---------------- x rows of the tile ------------------------------------
    // warp w gathers rows 32 w .. 32 w + 31: lane (rsub, j) copies 16-byte
    // chunk j of rows 4 i + rsub into the 128-byte swizzled layout, one
    // commit group per 64-column block, so the first up MMAs can start on
    // the first block while the rest arrive
    const int j8 = lane & 7, rsub = lane >> 3;
    bool ok = true;
    for (int i = 0; i < n_run && ok; ++i) {
      const int r0 = run_s[p.per_cta + i], rows = run_s[2 * p.per_cta + i];
      const int r = 32 * warp + lane;
      // padding rows gather the tile's first token (their h is masked)
      const int tok = p.row_tok[r0 + (r < rows ? r : 0)];
      ok = wait_warp(xempty, ((uint32_t)i & 1u) ^ 1u, abort_flag, p.status, p.wait_limit);
      if (!ok) break;
      for (int kb = 0; kb < num_kb; ++kb) {
        const uint32_t dst = sX + (uint32_t)kb * kSlab;
#pragma unroll
        for (int ii = 0; ii < 8; ++ii) {
          const int rr = 4 * ii + rsub;
          const int t = __shfl_sync(0xffffffffu, tok, rr);
          const int row = 32 * warp + rr;
          cp_async16(dst + (uint32_t)row * 128u + ((uint32_t)(j8 ^ (row & 7)) << 4),
                     p.x + (size_t)t * p.d + kb * kBK + j8 * 8);
        }
        cp_async_commit();
      }
      for (int kb = 0; kb < num_kb; ++kb) {
        cp_async_wait_n(num_kb - 1 - kb);
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(xfull(kb));
      }
    }
  } else if (warp == kLoaderWarp) {
    // ---------------- weight slabs, in MMA order ----------------------------
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      long long issued = 0;
      bool ok = true;
      auto load = [&](const uint8_t* src) {
        if (!ok) return;
        if (!wait_bounded(wempty(s), ph ^ 1u, abort_flag, p.status, p.wait_limit)) {
          ok = false;
          return;
        }
        mbar_expect_tx(wfull(s), kSlab);
        bulk_load(sW + (uint32_t)s * kSlab, src, kSlab, wfull(s));
        ++issued;
        if (++s == p.slots) { s = 0; ph ^= 1u; }
      };
      auto load_down = [&](int e, int c) {
        const uint8_t* v = p.wv + (size_t)(e * nch + chunk_of(c)) * 2 * npc * kSlab;
        for (int j = 0; j < 2 * npc; ++j) load(v + (size_t)j * kSlab);
      };
      for (int i = 0; i < n_run && ok; ++i) {
        const int e = run_s[i];
        for (int c = 0; c < nch; ++c) {
          const uint8_t* k = p.wk + (size_t)(e * nch + chunk_of(c)) * num_kb * kSlab;
          for (int kb = 0; kb < num_kb; ++kb) load(k + (size_t)kb * kSlab);
          if (c > 0) load_down(e, c - 1);
        }
        load_down(e, nch - 1);
      }
      // the loads still in flight land before the CTA exits
      for (long long j = issued > p.slots ? issued - p.slots : 0; j < issued; ++j)
        wait_settle(wfull((int)(j % p.slots)), (uint32_t)((j / p.slots) & 1), p.wait_limit);
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issue ----------------------------------------------
    const uint32_t idesc = idesc_bf16(kBM, kChunk);
    const uint32_t tU = tmem_base + kUCol;
    int s = 0;
    uint32_t ph = 0, uc = 0, dc = 0;
    bool ok = true, any = false;
    auto next = [&]() {
      if (++s == p.slots) { s = 0; ph ^= 1u; }
    };
    auto up = [&](int i, int c) {
      if (!wait_warp(uempty, (uc & 1u) ^ 1u, abort_flag, p.status, p.wait_limit)) return false;
      tc_fence_after();
      for (int kb = 0; kb < num_kb; ++kb) {
        if (c == 0 && !wait_warp(xfull(kb), (uint32_t)i & 1u, abort_flag, p.status, p.wait_limit))
          return false;
        if (!wait_warp(wfull(s), ph, abort_flag, p.status, p.wait_limit)) return false;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t a = sw128_desc(sX + (uint32_t)kb * kSlab);
          const uint64_t b = sw128_desc(sW + (uint32_t)s * kSlab);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16(tU, a + 2 * k, b + 2 * k, idesc, (kb | k) != 0 ? 1u : 0u);
          umma_commit(wempty(s));
          if (c == nch - 1 && kb == num_kb - 1) umma_commit(xempty);
        }
        __syncwarp();
        any = true;
        next();
      }
      if (elect_one()) umma_commit(ufull);
      __syncwarp();
      ++uc;
      return true;
    };
    auto down = [&](int i, int c) {
      if (c == 0) {
        if (!wait_warp(dempty, ((uint32_t)i & 1u) ^ 1u, abort_flag, p.status, p.wait_limit))
          return false;
        tc_fence_after();
      }
      for (int hh = 0; hh < 2; ++hh) {
        if (!wait_warp(hsfull(hh), dc & 1u, abort_flag, p.status, p.wait_limit)) return false;
        tc_fence_after();
        for (int np = 0; np < npc; ++np) {
          if (!wait_warp(wfull(s), ph, abort_flag, p.status, p.wait_limit)) return false;
          tc_fence_after();
          if (elect_one()) {
            const uint64_t a = sw128_desc(sH + (uint32_t)hh * kSlab);
            const uint64_t b = sw128_desc(sW + (uint32_t)s * kSlab);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              umma_bf16(tmem_base + (uint32_t)(np * kPiece), a + 2 * k, b + 2 * k, idesc,
                        (c | hh | k) != 0 ? 1u : 0u);
            umma_commit(wempty(s));
          }
          __syncwarp();
          next();
        }
        if (elect_one()) umma_commit(hsempty(hh));
        __syncwarp();
      }
      ++dc;
      if (c == nch - 1) {
        if (elect_one()) umma_commit(dfull);
        __syncwarp();
      }
      return true;
    };
    for (int i = 0; i < n_run && ok; ++i) {
      for (int c = 0; c < nch && ok; ++c) {
        ok = up(i, c);
        if (ok && c > 0) ok = down(i, c - 1);
      }
      if (ok) ok = down(i, nch - 1);
    }
    // every MMA this warp issued has completed before TMEM is released
    if (any) {
      if (elect_one()) umma_commit(mma_done);
      __syncwarp();
      wait_settle(mma_done, 0u, p.wait_limit);
    }
    __syncwarp();
  } else if (warp < kFirstDrain) {
    // ---------------- chunk epilogue: U -> masked bf16 h ---------------------
    // Thread = row 32 q + lane of the tile, 64 columns (one half of the
    // chunk, one 64-column block of h in the down MMA's A operand).
    const int q = warp & 3, hh = (warp - kFirstEpi) >> 2;
    const int r = 32 * q + lane;
    const uint32_t t_row = tmem_base + ((uint32_t)(32 * q) << 16) + kUCol + (uint32_t)(hh * kBK);
    uint8_t* hrow = smem + (size_t)(num_kb + hh) * kSlab + (size_t)r * 128;
    uint32_t n = 0;  // chunks done by this CTA
    bool ok = true;
    for (int i = 0; i < n_run && ok; ++i) {
      const int e = run_s[i], r0 = run_s[p.per_cta + i], rows = run_s[2 * p.per_cta + i];
      // the blocks this row runs (none for a padding row)
      uint64_t bm = 0ull;
      if (r < rows) {
        const uint64_t sh = p.shr[p.row_tok[r0 + r]];
        bm = e == 0 ? sh : (~sh & full);
      }
      for (int c = 0; c < nch; ++c, ++n) {
        if (!wait_warp(ufull, n & 1u, abort_flag, p.status, p.wait_limit)) { ok = false; break; }
        tc_fence_after();
        const int blk = (chunk_of(c) * kChunk + hh * kBK) / p.M;
        // rows that do not run this block keep h = 0: GeLU is computed for
        // every row and masked (a per-row select compiles to a branch per
        // element, which serialises the GeLU chains: 4x slower)
        const uint32_t keep = ((bm >> blk) & 1ull) ? 0xffffffffu : 0u;
        uint32_t v0[32], v1[32], o[32];
        tmem_ld32_async(t_row, v0);
        tmem_ld32_async(t_row + 32u, v1);
        tmem_wait_ld();
        // U is in registers: the next chunk's up MMAs may overwrite it while
        // this warp applies GeLU
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(uempty);
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
          o[jj] = keep & gelu2_bf16x2(__uint_as_float(v0[2 * jj]), __uint_as_float(v0[2 * jj + 1]));
          o[16 + jj] =
              keep & gelu2_bf16x2(__uint_as_float(v1[2 * jj]), __uint_as_float(v1[2 * jj + 1]));
        }
        // h of this half is free once the previous chunk's down MMAs read it
        if (!wait_warp(hsempty(hh), (n & 1u) ^ 1u, abort_flag, p.status, p.wait_limit)) {
          ok = false;
          break;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j)
          *reinterpret_cast<uint4*>(hrow + ((j ^ (r & 7)) << 4)) =
              make_uint4(o[4 * j], o[4 * j + 1], o[4 * j + 2], o[4 * j + 3]);
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(hsfull(hh));
      }
    }
  } else {
    // ---------------- drain: y[tok] += w D -----------------------------------
    // Thread = row 32 q + lane; 32 columns per pass: the thread stages its
    // row's 128 scaled bytes (chunk c at c ^ (r & 7)), then 8 lanes per row
    // add 4 rows x 128 contiguous bytes per instruction.
    const int q = warp & 3;
    const int r = 32 * q + lane;
    float* stf = reinterpret_cast<float*>(stg_base + (size_t)(warp - kFirstDrain) * 32 * 128);
    const int r_sub = lane >> 3, c8 = lane & 7;
    bool ok = true;
    for (int i = 0; i < n_run && ok; ++i) {
      const int r0 = run_s[p.per_cta + i], rows = run_s[2 * p.per_cta + i];
      const int tok = r < rows ? p.row_tok[r0 + r] : -1;
      const float w = r < rows ? p.row_w[r0 + r] : 0.f;
      if (!wait_warp(dfull, (uint32_t)i & 1u, abort_flag, p.status, p.wait_limit)) break;
      tc_fence_after();
      const uint32_t t_row = tmem_base + ((uint32_t)(32 * q) << 16);
      for (int c = 0; c < p.d; c += 32) {
        float v[32];
        tmem_ld32(t_row + (uint32_t)c, v);
#pragma unroll
        for (int jj = 0; jj < 8; ++jj)
          *reinterpret_cast<float4*>(stf + lane * 32 + ((jj ^ (lane & 7)) << 2)) =
              make_float4(w * v[4 * jj], w * v[4 * jj + 1], w * v[4 * jj + 2], w * v[4 * jj + 3]);
        __syncwarp();
#pragma unroll
        for (int ii = 0; ii < 8; ++ii) {
          const int rr = 4 * ii + r_sub;
          const int tr = __shfl_sync(0xffffffffu, tok, rr);
          const float4 val =
              *reinterpret_cast<const float4*>(stf + rr * 32 + ((c8 ^ (rr & 7)) << 2));
          if (tr >= 0)
            atomicAdd(reinterpret_cast<float4*>(p.y32 + (size_t)tr * p.d + c + c8 * 4), val);
        }
        __syncwarp();
      }
      // D has been read: the next tile's down MMAs may overwrite it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(dempty);
    }
  }
  // every warp converged before the CTA barrier
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Load-time repacking into operand slabs: 16 KB each, [128 rows][64
// bf16], 16-byte chunk q of row i at chunk position q ^ (i & 7) (the
// 128-byte swizzle of sw128_desc). Up slab (e, c, kb): rows = channels
// 128 c + i of K_e, columns = features 64 kb + j. Down slab (e, c, hh, np):
// rows = output features 128 np + i of V_e, columns = channels
// 128 c + 64 hh + j. A thread moves one 16-byte chunk.
__global__ void repack_up_kernel(const __nv_bfloat16* __restrict__ w_up, uint8_t* __restrict__ out,
                                 int E, int H, int d) {
  const int nch = H / kChunk, nkb = d / kBK;
  const long long n = (long long)E * nch * nkb * 128 * 8;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < n;
       t += (long long)gridDim.x * blockDim.x) {
    const int q = (int)(t & 7), i = (int)((t >> 3) & 127);
    const long long slab = t >> 10;
    const int kb = (int)(slab % nkb);
    const long long ec = slab / nkb;
    const int c = (int)(ec % nch), e = (int)(ec / nch);
    const uint4 v = *reinterpret_cast<const uint4*>(
        w_up + ((size_t)e * H + (size_t)c * kChunk + i) * d + kb * kBK + q * 8);
    *reinterpret_cast<uint4*>(out + slab * kSlab + i * 128 + ((q ^ (i & 7)) << 4)) = v;
  }
}

__global__ void repack_down_kernel(const __nv_bfloat16* __restrict__ w_down,
                                   uint8_t* __restrict__ out, int E, int H, int d) {
  const int nch = H / kChunk, npc = d / kPiece;
  const long long n = (long long)E * nch * 2 * npc * 128 * 8;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < n;
       t += (long long)gridDim.x * blockDim.x) {
    const int q = (int)(t & 7), i = (int)((t >> 3) & 127);
    const long long slab = t >> 10;
    const int np = (int)(slab % npc);
    const long long r = slab / npc;
    const int hh = (int)(r % 2);
    const long long ec = r / 2;
    const int c = (int)(ec % nch), e = (int)(ec / nch);
    const uint4 v = *reinterpret_cast<const uint4*>(
        w_down + ((size_t)e * d + (size_t)np * kPiece + i) * H + c * kChunk + hh * kBK + q * 8);
    *reinterpret_cast<uint4*>(out + slab * kSlab + i * 128 + ((q ^ (i & 7)) << 4)) = v;
  }
}

}  // namespace fused
}  // namespace tc

// The expert-tile FFN where it applies: bf16 layers with d a multiple of
// 128 up to 384 (D and U share the 512 TMEM columns), H a multiple of the
// 128-channel chunk and blocks of whole 64-column halves (M % 64 == 0).
bool ffn_fused_fits(int d, int H, int M) {
  return d % 128 == 0 && d <= 384 && H % tc::fused::kChunk == 0 && M % tc::kBK == 0;
}

int gemm_fused_setup(unif_moe_layer* L) {
  using namespace tc::fused;
  // tiles of a pass: at most ceil(rows_e / 128) per expert, rows_e <= region
  const int G = L->K + 1;
  const int64_t max_tiles = (int64_t)G * (L->region_rows / tc::kBM);
  L->ffn_per_cta = (int)((max_tiles + L->n_sm - 1) / L->n_sm);
  const int num_kb = L->d / tc::kBK;
  const uint32_t fixed = smem_bytes(num_kb, 0, G, L->ffn_per_cta);
  int slots = fixed < kMaxSmem ? (int)((kMaxSmem - fixed) / kSlab) : 0;
  if (slots > kMaxSlots) slots = kMaxSlots;
  if (slots < 3) {
    set_error("expert-tile FFN: %d weight slots fit in shared memory (d=%d)", slots, L->d);
    return UNIF_MOE_ERR_SHAPE;
  }
  L->ffn_slots = slots;
  L->ffn_smem = smem_bytes(num_kb, slots, G, L->ffn_per_cta);
  if (cudaFuncSetAttribute(ffn_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)L->ffn_smem) != cudaSuccess) {
    set_error("cudaFuncSetAttribute failed for the expert-tile FFN kernel");
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

cudaError_t launch_ffn_fused(unif_moe_layer* L, const void* x, cudaStream_t s) {
  tc::fused::Params p;
  p.fill = L->ws.grp_fill;
  p.G = L->K + 1;
  p.region = L->region_rows;
  p.per_cta = L->ffn_per_cta;
  p.row_tok = L->ws.row_tok;
  p.row_w = L->ws.row_w;
  p.shr = L->ws.shr_mask + L->rec0;
  p.d = L->d; p.H = L->H; p.M = L->M; p.B = L->B;
  p.n_chunks = L->H / tc::fused::kChunk;
  p.num_kb = L->d / tc::kBK;
  p.n_pieces = L->d / tc::fused::kPiece;
  p.slots = L->ffn_slots;
  p.x = static_cast<const __nv_bfloat16*>(x);
  p.y32 = L->ws.y32;
  p.status = L->ws.status;
  p.wait_limit = gemm_wait_limit();
  p.wk = static_cast<const uint8_t*>(L->ws.wk_slabs);
  p.wv = static_cast<const uint8_t*>(L->ws.wv_slabs);
  return launch_dependent(tc::fused::ffn_fused_kernel, dim3(L->n_sm),
                          dim3(tc::fused::kThreads), L->ffn_smem, s, p);
}

cudaError_t launch_repack_slabs(unif_moe_layer* L, cudaStream_t s) {
  const int E = L->K + 1;
  const int blocks = 8 * L->n_sm;
  tc::fused::repack_up_kernel<<<blocks, 256, 0, s>>>(
      static_cast<const __nv_bfloat16*>(L->w_up), static_cast<uint8_t*>(L->ws.wk_slabs), E, L->H,
      L->d);
  tc::fused::repack_down_kernel<<<blocks, 256, 0, s>>>(
      static_cast<const __nv_bfloat16*>(L->w_down), static_cast<uint8_t*>(L->ws.wv_slabs), E,
      L->H, L->d);
  return cudaGetLastError();
}

}  // namespace unif
