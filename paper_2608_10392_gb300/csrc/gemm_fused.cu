// Expert-tile FFN (tcgen05 + TMEM, CTA pairs) for bf16 layers with d <= 384:
// both projections of Eq. 16 for 256 rows of one expert's token list in a
// pair of CTAs (a cluster of two, one per SM), h kept on chip.
//
// The router groups the rows by expert (group e = expert e, one row per
// (token, expert) the token runs, weight alpha or s_j; Eqs. 28-30). A pair
// tile is 256 rows of one group; CTA r of the pair owns rows 128 r ..
// 128 r + 127. For each 128-channel chunk c of the expert's H channels the
// pair computes
//   U = x K_e[c]^T                        (M=256, N=128, K=d; TMEM)
//   h = bf16(GeLU(U)), zero in the columns of blocks the row does not run
//   D += h V_e[:, c]^T                    (M=256, N=d: 256-column pieces,
//                                          then a 128-column remainder)
// with tcgen05.mma.cta_group::2 issued by the even CTA: each CTA holds the
// A rows of its own 128 rows (x, then h) and half of every B operand (64 of
// the 128 rows of each weight slab; for a 256-column piece, one whole slab
// each), and each CTA's TMEM the D and U rows of
// its own 128 rows. After the last chunk each CTA adds w D into the fp32
// output accumulator, once per (token, expert) instead of once per (token,
// expert, block). Each token's x row is gathered once per expert it runs,
// and h never leaves the SM. The blocks a row does not run are computed and
// masked, so the tensor work is that of the whole expert: B (1 + k) blocks
// per token against the C_B = b + k (B - b) the method activates (Eq. 35).
// Splitting every weight slab between the two SMs halves the bytes each SM
// streams per MMA (a single-CTA version of this kernel streamed 2.4 MB of
// weights per 128-row tile through a ring of five 16 KB slots).
//
// Shared memory (each CTA): the x tile (128 x d bf16, resident for the
// tile), h of one chunk (128 x 128 bf16, two 64-column halves), a ring of
// 8 KB weight half-slabs (64 rows x 64 reduction elements, loaded by TMA
// from the weights repacked at load time into [slab][128 rows][64] order,
// so that each half-slab is 8 KB contiguous), and the drain warps' staging
// tiles. TMEM (512 columns): D in columns [0, d), U in [384, 512).
//
// Roles (each CTA, 18 warps):
//   warps 0-3    gather this CTA's x rows (16-byte cp.async, 32 rows each),
//                then drain the previous tile's D columns [d/2, d)
//   warp 4       this CTA's weight half-slabs by TMA, in MMA order
//   warp 5       TMEM allocation (both CTAs); MMA issue (even CTA, one lane);
//                in the odd CTA, zeroing of the next pass's accumulator
//   warps 6-13   chunk epilogue: U -> GeLU -> masked bf16 h in shared memory
//                (warp w: TMEM lane quarter w % 4, 64-column half (w-6)/4)
//   warps 14-17  drain: w D columns [0, d/2) -> fp32 atomic adds into the
//                accumulator
// The even CTA's barriers collect both CTAs' arrivals (x rows, h, U and D
// read) and both halves of each slab (TMA with cta_group::2 completes on
// them); its MMA commits arrive on both CTAs' barriers (multicast). Order
// of the MMAs in a tile: up(0), up(1), down(0), up(2), down(1), ...,
// up(n-1), down(n-2), down(n-1), so that the epilogue of chunk c runs while
// the tensor pipe computes down(c-1) and up(c+1). Every wait is bounded; a
// wait that runs out records kStatusTimeout in the status word and the CTA
// unwinds, letting its copies and MMAs in flight land before the pair
// releases its TMEM.
#include <stdio.h>

#include "decide.cuh"
#include "internal.cuh"
#include "tc_common.cuh"

namespace unif {
namespace tc {
namespace fused {

constexpr int kChunk = 128;           // H channels per chunk (the up MMA's N)
constexpr int kPiece = 128;           // d rows per repacked V_e slab (an N = 128 MMA's B; N = 256 takes two)
constexpr uint32_t kSlab = 16384;     // a weight slab: 128 rows x 64 bf16
constexpr uint32_t kHalf = 8192;      // the half of a slab one CTA of the pair holds
constexpr uint32_t kXBlock = 16384;   // 128 rows x 64 bf16 of x or h
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kUCol = 384;       // U's first TMEM column
constexpr int kMaxKb = 6;             // d <= 384
constexpr int kMaxSlots = 16;
constexpr int kGatherWarps = 4;
constexpr int kLoaderWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kFirstEpi = 6;
constexpr int kEpiWarps = 8;
constexpr int kFirstDrain = 14;
constexpr int kDrainWarps = 4;
constexpr int kThreads = 32 * (kFirstDrain + kDrainWarps);  // 576
constexpr uint32_t kStaging = kDrainWarps * 32u * 128u;  // per TMEM lane quarter 4 KB: two 32 x 16 fp32 tiles
constexpr uint32_t kBarBytes = 512;
constexpr uint32_t kMaxSmem = 232448;
constexpr int kPairRows = 256;        // rows of a pair tile
constexpr int kStageHalves = 2;       // half-slabs per ring stage (one barrier pair)

struct Params {
  const int32_t* fill;     // [G] rows per expert group (final once the router completed)
  int G, region, per_pair; // G = K + 1 groups of `region` rows; tile run capacity
  const int32_t* row_tok;  // [G][region] pass-relative token of each row
  const float* row_w;      // [G][region] the row's pathway weight
  const uint64_t* shr;     // [T] shared block set of each token of the pass
  int d, H, M, B;
  int n_chunks, num_kb, n_pieces, slots;
  const __nv_bfloat16* x;  // [T][d] the pass's tokens
  float* y32;              // [T][d] fp32 output accumulator of the pass
  float* y32_next;         // the other accumulator, zeroed here for the next pass
  long long next_f4;       // its float4 count
  int* status;
  long long wait_limit;
};

// Bytes of dynamic shared memory for num_kb reduction blocks of x and
// `slots` weight half-slabs (plus the tile table of G groups and per_pair
// pair tiles).
__host__ __device__ constexpr uint32_t smem_bytes(int num_kb, int slots, int G, int per_pair) {
  return 1024u + (uint32_t)num_kb * kXBlock + 2u * kXBlock + (uint32_t)slots * kHalf + kStaging +
         kBarBytes + (uint32_t)((2 * G + 1 + 3 * per_pair) * 4 + 15) / 16u * 16u;
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
// lets the copies and MMAs it started land before the pair releases TMEM.
__device__ __forceinline__ void wait_settle(uint32_t bar, uint32_t parity, long long limit) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > limit) return;
}

// The tiles of TR rows of the groups whose sizes are fill[0..G) (each
// clamped to the region): first_s[g] = first tile of group g (first_s[G] =
// all tiles), cnt_s[g] = its size. Run by one warp.
template <int TR>
__device__ __forceinline__ void pair_tile_table(const int32_t* fill, int G, int region, int lane,
                                                int32_t* first_s, int32_t* cnt_s) {
  int carry = 0;
  for (int g0 = 0; g0 < G; g0 += 32) {
    const int g = g0 + lane;
    const int c = g < G ? min(__ldcg(fill + g), region) : 0;
    const int nt = (c + TR - 1) / TR;
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

// DD = d (128, 256 or 384): the x tile's 64-column blocks and the down
// projection's stages and pieces are compile-time counts, so that the MMA
// warp's per-stage control is a few instructions (it shares its scheduler
// with epilogue warps running GeLU, and a runtime division per stage
// measurably delayed every stage)
template <int DD>
__global__ void __launch_bounds__(kThreads, 1)
ffn_fused_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                 Params p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived from smem_raw by an offset so that the
  // compiler keeps every access through it in the shared state space (the
  // same offsets in both CTAs of the pair: the pair MMAs address the peer's
  // operands at this CTA's addresses)
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  constexpr int num_kb = DD / kBK, npc = DD / kPiece;
  static_assert(num_kb % kStageHalves == 0 && (2 * npc) % kStageHalves == 0,
                "stages never straddle an up or a down projection");
  // The down projection of a chunk: D[:, 256 P .. 256 P + 255] for each
  // 256-column piece P as N = 256 MMAs, each reading h once for 256 output
  // columns (three N = 128 pieces read h three times per chunk, and shared
  // memory bandwidth is what the chunk loop runs against), then the
  // 128-column remainder (d = 128, 384) as N = 128 MMAs. Stages in MMA
  // order: piece P for h half 0, the remainder (both halves), piece P for
  // h half 1, so that h half 0 is released after the second stage as
  // before. Each stage is kStageHalves half-slabs of this CTA.
  constexpr int n256 = DD / 256, kRem = DD % 256 ? 1 : 0;
  constexpr int kDownStages = 2 * n256 + kRem;
  static_assert(kDownStages * kStageHalves == 2 * npc, "the down stages hold the chunk's slabs");
  // true: 256-column piece P of h half hh; false: the remainder piece
  auto down_stage = [](int st, int& hh, int& P) {
    if (st < n256) { hh = 0; P = st; return true; }
    if (kRem && st == n256) { hh = 0; P = 0; return false; }
    hh = 1; P = st - n256 - kRem;
    return true;
  };
  // the last down stage that reads h half 0
  constexpr int kH0Last = kRem ? n256 : n256 - 1;
  const int nch = p.n_chunks;
  const uint32_t sX = smem_u32(smem);
  const uint32_t sH = sX + (uint32_t)num_kb * kXBlock;
  const uint32_t sW = sH + 2u * kXBlock;
  uint8_t* stg_base = smem + (size_t)(num_kb + 2) * kXBlock + (size_t)p.slots * kHalf;
  uint64_t* bars = reinterpret_cast<uint64_t*>(stg_base + kStaging);
  const uint32_t bar0 = smem_u32(bars);
  auto xfull = [&](int kb) { return bar0 + 8u * kb; };
  const uint32_t xempty = bar0 + 8u * 6;
  auto wfull = [&](int s) { return bar0 + 8u * (7 + s); };
  auto wempty = [&](int s) { return bar0 + 8u * (23 + s); };
  const uint32_t ufull = bar0 + 8u * 39, uempty = bar0 + 8u * 40;
  auto hsfull = [&](int h) { return bar0 + 8u * (41 + h); };
  auto hsempty = [&](int h) { return bar0 + 8u * (43 + h); };
  const uint32_t dfull = bar0 + 8u * 45, dempty = bar0 + 8u * 46;
  const uint32_t mma_done = bar0 + 8u * 47;
  const uint32_t fin = bar0 + 8u * 48;  // the peer CTA has finished with the pair's TMEM
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 49);
  static_assert(8 * 49 + 8 <= kBarBytes, "barrier region");
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // tile table: first pair tile and size of every group, then (group,
  // first row, real rows) of each pair tile of this pair's run
  int32_t* first_s = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(bars) + kBarBytes);
  int32_t* gcnt_s = first_s + p.G + 1;
  int32_t* run_s = gcnt_s + p.G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();  // 0: the CTA that issues the MMAs
  const bool leader = rank == 0;
  // the leader's copy of a barrier, as a cluster address (arrivals of both
  // CTAs go there)
  auto at_leader = [&](uint32_t bar) { return mapa_shared(bar, 0); };
  auto arrive_leader = [&](uint32_t bar) {
    if (leader) mbar_arrive(bar);
    else mbar_arrive_cluster(at_leader(bar));
  };

  if (threadIdx.x == 0) {
    // counts: the leader's barriers take the arrivals of both CTAs
    for (int kb = 0; kb < kMaxKb; ++kb) mbar_init(xfull(kb), 2 * kGatherWarps);
    mbar_init(xempty, 1);
    for (int s = 0; s < kMaxSlots; ++s) {
      mbar_init(wfull(s), 1);  // the leader's loader arrives; both halves' bytes land on it
      mbar_init(wempty(s), 1);
    }
    mbar_init(ufull, 1);
    mbar_init(uempty, 2 * kEpiWarps);
    for (int h = 0; h < 2; ++h) {
      mbar_init(hsfull(h), kEpiWarps);  // four warps of each CTA per half
      mbar_init(hsempty(h), 1);
    }
    mbar_init(dfull, 1);
    mbar_init(dempty, 2 * (kDrainWarps + kGatherWarps));
    mbar_init(mma_done, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {  // both CTAs of the pair allocate together
    tmem_alloc_pair(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish_pair();
  }
  const int pair = (int)(blockIdx.x >> 1), n_pairs = (int)(gridDim.x >> 1);
  if (warp == kLoaderWarp) {
    // the group sizes are final once the router completed
    grid_dep_wait();
    pair_tile_table<kPairRows>(p.fill, p.G, p.region, lane, first_s, gcnt_s);
    __syncwarp();
    const int nt = first_s[p.G];
    const int tb = (int)(((long long)pair * nt) / n_pairs);
    const int te = (int)(((long long)(pair + 1) * nt) / n_pairs);
    for (int k = tb + lane; k < te; k += 32) {
      int lo = 0, hi = p.G - 1;  // the last group whose first tile is <= k
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (first_s[mid] <= k) lo = mid; else hi = mid - 1;
      }
      const int i = k - first_s[lo];
      run_s[k - tb] = lo;
      run_s[p.per_pair + k - tb] = lo * p.region + kPairRows * i;
      run_s[2 * p.per_pair + k - tb] = min(kPairRows, gcnt_s[lo] - kPairRows * i);
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  // both CTAs' barriers are initialised before either CTA signals the other
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();
  grid_dep_launch();
  const int nt = first_s[p.G];
  const int t_begin = (int)(((long long)pair * nt) / n_pairs);
  const int n_run = (int)(((long long)(pair + 1) * nt) / n_pairs) - t_begin;
  const uint64_t full = p.B >= 64 ? ~0ull : ((1ull << p.B) - 1ull);
  // Each pair walks the chunks of a tile from its own starting chunk, so
  // that the pairs working on one expert at the same time read different
  // weight slabs; D's sum over the chunks is the same in any order up to
  // the order of the fp32 additions.
  const int rot = pair % nch;
  auto chunk_of = [&](int c) { return c + rot < nch ? c + rot : c + rot - nch; };
  // this CTA's rows of pair tile i: [r0 + 128 rank, + rows_mine)
  auto my_rows = [&](int i, int& r0, int& rows) {
    r0 = run_s[p.per_pair + i] + kBM * (int)rank;
    rows = min(kBM, max(0, run_s[2 * p.per_pair + i] - kBM * (int)rank));
  };
  // y[tok] += w D over columns [c_begin, c_end) of tile i's D, for the 32
  // rows of TMEM lane quarter warp % 4 (thread = row). 16 columns per
  // pass: the thread stages its row's 64 scaled bytes in the warp's 2 KB
  // tile (16-byte chunk c at c ^ ((r >> 1) & 3)), then 4 lanes per row add
  // 8 rows x 64 contiguous bytes per instruction. Returns false if a wait
  // gave up. The D reads end with the arrival on dempty.
  auto drain = [&](int i, int c_begin, int c_end, float* stf) {
    const int q = warp & 3;
    const int r = 32 * q + lane;
    int r0, rows;
    my_rows(i, r0, rows);
    const int tok = r < rows ? p.row_tok[r0 + r] : -1;
    const float w = r < rows ? p.row_w[r0 + r] : 0.f;
    if (!wait_warp(dfull, (uint32_t)i & 1u, abort_flag, p.status, p.wait_limit)) return false;
    tc_fence_after();
    const uint32_t t_row = tmem_base + ((uint32_t)(32 * q) << 16);
    const int r_sub = lane >> 2, c4 = lane & 3;
    const uint32_t sw = (uint32_t)(lane >> 1) & 3u;
#pragma unroll 1
    for (int c = c_begin; c < c_end; c += 16) {
      float v[16];
      tmem_ld16(t_row + (uint32_t)c, v);
#pragma unroll
      for (int jj = 0; jj < 4; ++jj)
        *reinterpret_cast<float4*>(stf + lane * 16 + ((jj ^ sw) << 2)) =
            make_float4(w * v[4 * jj], w * v[4 * jj + 1], w * v[4 * jj + 2], w * v[4 * jj + 3]);
      __syncwarp();
#pragma unroll
      for (int ii = 0; ii < 4; ++ii) {
        const int rr = 8 * ii + r_sub;
        const int tr = __shfl_sync(0xffffffffu, tok, rr);
        const float4 val = *reinterpret_cast<const float4*>(
            stf + rr * 16 + ((c4 ^ ((rr >> 1) & 3)) << 2));
        if (tr >= 0)
          atomicAdd(reinterpret_cast<float4*>(p.y32 + (size_t)tr * DD + c + c4 * 4), val);
      }
      __syncwarp();
    }
    // D has been read: the next tile's down MMAs may overwrite it
    tc_fence_before();
    __syncwarp();
    if (lane == 0) arrive_leader(dempty);
    return true;
  };

  if (warp < kGatherWarps) {
    // ---------------- this CTA's x rows of the tile -------------------------
    // warp w gathers rows 32 w .. 32 w + 31: lane (rsub, j) copies 16-byte
    // chunk j of rows 4 i + rsub into the 128-byte swizzled layout, one
    // commit group per 64-column block, so the first up MMAs can start on
    // the first block while the rest arrive
    const int j8 = lane & 7, rsub = lane >> 3;
    float* stg_gather = reinterpret_cast<float*>(stg_base + (size_t)warp * 4096 + 2048);
    bool ok = true;
    for (int i = 0; i < n_run && ok; ++i) {
      int r0, rows;
      my_rows(i, r0, rows);
      const int r = 32 * warp + lane;
      // padding rows gather the pair tile's first token (their h is masked)
      const int tok = p.row_tok[r < rows ? r0 + r : run_s[p.per_pair + i]];
      ok = wait_warp(xempty, ((uint32_t)i & 1u) ^ 1u, abort_flag, p.status, p.wait_limit);
      if (!ok) break;
      for (int kb = 0; kb < num_kb; ++kb) {
        const uint32_t dst = sX + (uint32_t)kb * kXBlock;
#pragma unroll
        for (int ii = 0; ii < 8; ++ii) {
          const int rr = 4 * ii + rsub;
          const int t = __shfl_sync(0xffffffffu, tok, rr);
          const int row = 32 * warp + rr;
          cp_async16(dst + (uint32_t)row * 128u + ((uint32_t)(j8 ^ (row & 7)) << 4),
                     p.x + (size_t)t * DD + kb * kBK + j8 * 8);
        }
        cp_async_commit();
      }
#pragma unroll
      for (int kb = 0; kb < num_kb; ++kb) {
        cp_async_wait_n(num_kb - 1 - kb);
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) arrive_leader(xfull(kb));
      }
      // idle until the next tile's rows are wanted: drain the second half
      // of the previous tile's D columns beside the drain warps
      if (i > 0) ok = drain(i - 1, DD / 2, DD, stg_gather);
    }
    if (ok && n_run > 0) drain(n_run - 1, DD / 2, DD, stg_gather);
  } else if (warp == kLoaderWarp) {
    // ---------------- this CTA's weight half-slabs, in MMA order ------------
    // Half `rank` of slab u = rows 128 u + 64 rank .. + 63 of the repacked
    // weights. The ring holds stages of kStageHalves consecutive half-slabs
    // (an up or a down projection's k-blocks never straddle a stage) under
    // one barrier pair: per stage one wait, one expect_tx and one commit
    // (each mbarrier round trip costs a thread several hundred cycles), and
    // the stage's loads go out from kStageHalves lanes at once. Both
    // halves of a slab complete on the leader's wfull, which the leader's
    // loader arms with the stage's bytes.
    const int n_stages = p.slots / kStageHalves;
    int s = 0;
    uint32_t ph = 0;
    long long issued = 0;
    bool ok = true;
    // lane j < kStageHalves loads the 64 repacked rows starting at row_j
    // into half-slab slot j of the stage
    auto stage = [&](const CUtensorMap* m, long long row0, long long row1) {
      if (!ok) return;
      // the whole warp waits (lanes parked at a shuffle while one lane
      // waits cost the warp hundreds of cycles to reconverge)
      if (!wait_warp(wempty(s), ph ^ 1u, abort_flag, p.status, p.wait_limit)) {
        ok = false;
        return;
      }
      if (lane == 0 && leader) mbar_expect_tx(wfull(s), 2u * kHalf * kStageHalves);
      __syncwarp();
      if (lane < kStageHalves)
        tma_load_2d_pair(sW + (uint32_t)(s * kStageHalves + lane) * kHalf, m, at_leader(wfull(s)),
                         0, (int)(lane == 0 ? row0 : row1));
      ++issued;
      if (++s == n_stages) { s = 0; ph ^= 1u; }
    };
    // Down stages of chunk c in MMA order (down_stage): a 256-column piece
    // P for h half hh holds this CTA's 128 of its rows, i.e. all of slab
    // (hh, np = 2 P + rank); the 128-column remainder piece holds this
    // CTA's 64-row halves of slabs (0, npc - 1) and (1, npc - 1).
    auto load_down = [&](int e, int c) {
      const long long v0 = (long long)(e * nch + chunk_of(c)) * 2 * npc;
#pragma unroll
      for (int st = 0; st < kDownStages; ++st) {
        int hh, P;
        if (down_stage(st, hh, P)) {
          const long long row = (v0 + hh * npc + 2 * P + rank) * 128;
          stage(&tmV, row, row + 64);
        } else {
          const long long row = (v0 + npc - 1) * 128 + 64 * (long long)rank;
          stage(&tmV, row, row + (long long)npc * 128);
        }
      }
    };
    for (int i = 0; i < n_run && ok; ++i) {
      const int e = run_s[i];
      for (int c = 0; c < nch; ++c) {
        const long long u0 = (long long)(e * nch + chunk_of(c)) * num_kb;
        for (int kb = 0; kb < num_kb; kb += kStageHalves)
          stage(&tmK, (u0 + kb) * 128 + 64 * (long long)rank,
                (u0 + kb + 1) * 128 + 64 * (long long)rank);
        if (c > 0) load_down(e, c - 1);
      }
      load_down(e, nch - 1);
    }
    // the loads still in flight land before the pair exits (their bytes
    // complete on the leader's barriers)
    if (leader && lane == 0)
      for (long long j = issued > n_stages ? issued - n_stages : 0; j < issued; ++j)
        wait_settle(wfull((int)(j % n_stages)), (uint32_t)((j / n_stages) & 1), p.wait_limit);
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issue (the leader CTA) ----------------------------
    if (leader) {
      const uint32_t idesc = idesc_bf16(2 * kBM, kChunk);  // M = 256 over the pair, N = 128
      const uint32_t idesc256 = idesc_bf16(2 * kBM, 256);   // the down projection's wide pieces
      const uint16_t both = 3;
      const uint32_t tU = tmem_base + kUCol;
      const int n_stages = p.slots / kStageHalves;
      int s = 0;
      uint32_t ph = 0, uc = 0, dc = 0;
      bool ok = true, any = false;
      auto next = [&]() {
        if (++s == n_stages) { s = 0; ph ^= 1u; }
      };
      auto up = [&](int i, int c) {
        if (!wait_warp_cluster(uempty, (uc & 1u) ^ 1u, abort_flag, p.status, p.wait_limit))
          return false;
        tc_fence_after();
#pragma unroll
        for (int kb0 = 0; kb0 < num_kb; kb0 += kStageHalves) {
          if (c == 0)
            for (int kb = kb0; kb < kb0 + kStageHalves; ++kb)
              if (!wait_warp_cluster(xfull(kb), (uint32_t)i & 1u, abort_flag, p.status,
                                     p.wait_limit))
                return false;
          if (!wait_warp_cluster(wfull(s), ph, abort_flag, p.status, p.wait_limit)) return false;
          tc_fence_after();
          if (elect_one()) {
#pragma unroll
            for (int j = 0; j < kStageHalves; ++j) {
              const int kb = kb0 + j;
              const uint64_t a = sw128_desc(sX + (uint32_t)kb * kXBlock);
              const uint64_t b = sw128_desc(sW + (uint32_t)(s * kStageHalves + j) * kHalf);
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                umma_bf16_pair(tU, a + 2 * k, b + 2 * k, idesc, (kb | k) != 0 ? 1u : 0u);
            }
            umma_commit_pair(wempty(s), both);
            if (c == nch - 1 && kb0 + kStageHalves == num_kb) umma_commit_pair(xempty, both);
          }
          __syncwarp();
          any = true;
          next();
        }
        if (elect_one()) umma_commit_pair(ufull, both);
        __syncwarp();
        ++uc;
        return true;
      };
      // down stages in the order of down_stage (the loader's order)
      auto down = [&](int i, int c) {
        if (c == 0) {
          if (!wait_warp_cluster(dempty, ((uint32_t)i & 1u) ^ 1u, abort_flag, p.status,
                                 p.wait_limit))
            return false;
          tc_fence_after();
        }
#pragma unroll
        for (int st = 0; st < kDownStages; ++st) {
          int hh, P;
          const bool wide = down_stage(st, hh, P);
          if (st == 0 &&
              !wait_warp_cluster(hsfull(0), dc & 1u, abort_flag, p.status, p.wait_limit))
            return false;
          if (st == n256 &&
              !wait_warp_cluster(hsfull(1), dc & 1u, abort_flag, p.status, p.wait_limit))
            return false;
          if (!wait_warp_cluster(wfull(s), ph, abort_flag, p.status, p.wait_limit)) return false;
          tc_fence_after();
          if (elect_one()) {
            const uint32_t w0 = sW + (uint32_t)(s * kStageHalves) * kHalf;
            if (wide) {
              // N = 256: this CTA's 128 rows of the piece span the stage's
              // two half-slab slots (contiguous, 8-row groups 1 KB apart)
              const uint64_t a = sw128_desc(sH + (uint32_t)hh * kXBlock);
              const uint64_t b = sw128_desc(w0);
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                umma_bf16_pair(tmem_base + (uint32_t)(P * 256), a + 2 * k, b + 2 * k, idesc256,
                               (c | hh | k) != 0 ? 1u : 0u);
            } else {
#pragma unroll
              for (int jj = 0; jj < kStageHalves; ++jj) {
                const uint64_t a = sw128_desc(sH + (uint32_t)jj * kXBlock);
                const uint64_t b = sw128_desc(w0 + (uint32_t)jj * kHalf);
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k)
                  umma_bf16_pair(tmem_base + (uint32_t)(n256 * 256), a + 2 * k, b + 2 * k, idesc,
                                 (c | jj | k) != 0 ? 1u : 0u);
              }
            }
            if (st == kH0Last) umma_commit_pair(hsempty(0), both);
            if (st == kDownStages - 1) umma_commit_pair(hsempty(1), both);
            umma_commit_pair(wempty(s), both);
          }
          __syncwarp();
          next();
        }
        ++dc;
        if (c == nch - 1) {
          if (elect_one()) umma_commit_pair(dfull, both);
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
      // every MMA issued has completed before the pair releases TMEM
      if (any) {
        if (elect_one()) umma_commit_pair(mma_done, 1);
        __syncwarp();
        wait_settle(mma_done, 0u, p.wait_limit);
      }
    } else {
      // The peer's MMA warp has no MMAs to issue: it zeroes its pair's share
      // of the other accumulator, which the next pass adds into (the
      // combine only reads this pass's). It waits for nothing, so a pass
      // whose other roles gave up still leaves the next one clean.
      float4* z = reinterpret_cast<float4*>(p.y32_next);
      const long long per = (p.next_f4 + n_pairs - 1) / n_pairs;
      const long long z0 = (long long)pair * per;
      const long long z1 = min(p.next_f4, z0 + per);
      for (long long k = z0 + lane; k < z1; k += 32) z[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    __syncwarp();
  } else if (warp < kFirstDrain) {
    // ---------------- chunk epilogue: U -> masked bf16 h ---------------------
    // Thread = row 32 q + lane of this CTA's rows, 64 columns (one half of
    // the chunk, one 64-column block of h in the down MMA's A operand).
    const int q = warp & 3, hh = (warp - kFirstEpi) >> 2;
    const int r = 32 * q + lane;
    const uint32_t t_row = tmem_base + ((uint32_t)(32 * q) << 16) + kUCol + (uint32_t)(hh * kBK);
    uint8_t* hrow = smem + (size_t)(num_kb + hh) * kXBlock + (size_t)r * 128;
    uint32_t n = 0;  // chunks done by this CTA
    bool ok = true;
    for (int i = 0; i < n_run && ok; ++i) {
      const int e = run_s[i];
      int r0, rows;
      my_rows(i, r0, rows);
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
        if (lane == 0) arrive_leader(uempty);
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
        if (lane == 0) arrive_leader(hsfull(hh));
      }
    }
  } else {
    // ---------------- drain: y[tok] += w D, the first half of the columns ---
    // (the gather warps, idle between their tiles' gathers, take the second)
    float* stf = reinterpret_cast<float*>(stg_base + (size_t)(warp & 3) * 4096);
    for (int i = 0; i < n_run; ++i)
      if (!drain(i, 0, DD / 2, stf)) break;
  }
  // every warp converged before the CTA barrier; then each CTA tells its
  // peer that it is done with the pair's TMEM (the leader after its MMAs
  // completed), and the TMEM owner warp waits for the peer's word before
  // the pair releases it. (A barrier.cluster arrive at this point stalled
  // ~40 us on GB300, measured, whatever the relaxed or release form.)
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) mbar_arrive_cluster(mapa_shared(fin, rank ^ 1u));
  if (warp == kMmaWarp) {
    wait_settle(fin, 0u, p.wait_limit);
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

// Load-time repacking into operand slabs: 16 KB each, [128 rows][64 bf16]
// row-major (the TMA loads apply the 128-byte swizzle); half r of a slab is
// its rows 64 r .. 64 r + 63, 8 KB contiguous. Up slab (e, c, kb): rows =
// channels 128 c + i of K_e, columns = features 64 kb + j. Down slab (e, c,
// hh, np): rows = output features 128 np + i of V_e, columns = channels
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
    *reinterpret_cast<uint4*>(out + slab * kSlab + i * 128 + q * 16) = v;
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
    *reinterpret_cast<uint4*>(out + slab * kSlab + i * 128 + q * 16) = v;
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

typedef void (*FfnKernel)(CUtensorMap, CUtensorMap, tc::fused::Params);
static FfnKernel ffn_kernel_for(int d) {
  using namespace tc::fused;
  return d == 128 ? ffn_fused_kernel<128> : (d == 256 ? ffn_fused_kernel<256> : ffn_fused_kernel<384>);
}

int gemm_fused_setup(unif_moe_layer* L) {
  using namespace tc::fused;
  const FfnKernel kernel = ffn_kernel_for(L->d);
  const int G = L->K + 1;
  // pair tiles of a pass: at most ceil(rows_e / 256) per expert
  const int64_t max_tiles = (int64_t)G * ((L->region_rows + kPairRows - 1) / kPairRows);
  const int num_kb = L->d / tc::kBK;
  // the weight slabs as [rows][64] bf16 maps, boxes of one half-slab
  const uint64_t slab_rows = (uint64_t)G * (L->H / kChunk) * num_kb * 128;
  const uint64_t vslab_rows = (uint64_t)G * (L->H / kChunk) * 2 * (L->d / kPiece) * 128;
  if (!encode_bf16_map(&L->tm_fk, L->ws.wk_slabs, tc::kBK, slab_rows, tc::kBK, 64, 128) ||
      !encode_bf16_map(&L->tm_fv, L->ws.wv_slabs, tc::kBK, vslab_rows, tc::kBK, 64, 128)) {
    set_error("cuTensorMapEncodeTiled failed for the expert-tile weight slabs");
    return UNIF_MOE_ERR_CUDA;
  }
  // one pair per two SMs, as many pairs as fit at once
  int per_pair_guess = (int)((max_tiles + L->n_sm / 2 - 1) / (L->n_sm / 2));
  uint32_t fixed = smem_bytes(num_kb, 0, G, per_pair_guess);
  int slots = fixed < kMaxSmem ? (int)((kMaxSmem - fixed) / kHalf) : 0;
  if (slots > kMaxSlots) slots = kMaxSlots;
  slots -= slots % kStageHalves;
  if (slots < 2 * kStageHalves) {
    set_error("expert-tile FFN: %d weight slots fit in shared memory (d=%d)", slots, L->d);
    return UNIF_MOE_ERR_SHAPE;
  }
  L->ffn_slots = slots;
  L->ffn_smem = smem_bytes(num_kb, slots, G, per_pair_guess);
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)L->ffn_smem) != cudaSuccess ||
      cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 0) !=
          cudaSuccess) {
    set_error("cudaFuncSetAttribute failed for the expert-tile FFN kernel");
    return UNIF_MOE_ERR_CUDA;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(L->n_sm);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = L->ffn_smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, kernel, &cfg) != cudaSuccess ||
      clusters < 1) {
    set_error("expert-tile FFN: no CTA pair fits on this device");
    return UNIF_MOE_ERR_SHAPE;
  }
  if (clusters > L->n_sm / 2) clusters = L->n_sm / 2;
  L->ffn_pairs = clusters;
  L->ffn_per_cta = (int)((max_tiles + clusters - 1) / clusters);  // pair tiles per pair
  if (L->ffn_per_cta > per_pair_guess) {  // fewer pairs than SMs / 2: a longer run table
    L->ffn_smem = smem_bytes(num_kb, slots, G, L->ffn_per_cta);
    while (L->ffn_smem > kMaxSmem && slots > 2 * kStageHalves) {
      slots -= kStageHalves;
      L->ffn_slots = slots;
      L->ffn_smem = smem_bytes(num_kb, slots, G, L->ffn_per_cta);
    }
    if (L->ffn_smem > kMaxSmem) {
      set_error("expert-tile FFN: a run of %d pair tiles per pair does not fit in shared memory",
                L->ffn_per_cta);
      return UNIF_MOE_ERR_SHAPE;
    }
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)L->ffn_smem) != cudaSuccess) {
      set_error("cudaFuncSetAttribute failed for the expert-tile FFN kernel");
      return UNIF_MOE_ERR_CUDA;
    }
  }
  return UNIF_MOE_OK;
}

cudaError_t launch_ffn_fused(unif_moe_layer* L, const void* x, cudaStream_t s) {
  tc::fused::Params p;
  p.fill = L->ws.grp_fill;
  p.G = L->K + 1;
  p.region = L->region_rows;
  p.per_pair = L->ffn_per_cta;
  p.row_tok = L->ws.row_tok;
  p.row_w = L->ws.row_w;
  p.shr = L->ws.shr_mask + L->rec0;
  p.d = L->d; p.H = L->H; p.M = L->M; p.B = L->B;
  p.n_chunks = L->H / tc::fused::kChunk;
  p.num_kb = L->d / tc::kBK;
  p.n_pieces = L->d / tc::fused::kPiece;
  p.slots = L->ffn_slots;
  p.x = static_cast<const __nv_bfloat16*>(x);
  p.y32 = acc_cur(L);
  p.y32_next = L->acc_sel ? L->ws.y32 : L->ws.y32_b;
  p.next_f4 = (long long)L->pass_tokens * L->d / 4;
  p.status = L->ws.status;
  p.wait_limit = gemm_wait_limit();
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * L->ffn_pairs);
  cfg.blockDim = dim3(tc::fused::kThreads);
  cfg.dynamicSmemBytes = L->ffn_smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, ffn_kernel_for(L->d), L->tm_fk, L->tm_fv, p);
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
