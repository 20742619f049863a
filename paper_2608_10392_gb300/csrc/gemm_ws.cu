// Weight-stationary grouped expert GEMMs (tcgen05 + TMEM) for bf16 layers
// whose per-group weight slice fits in shared memory.
//
// Tiles are numbered group by group, g = (expert e, block b) (from the
// router's group sizes, or the grouping kernels' tile list), so consecutive
// tiles mostly share one weight slice: K_e[:, H_b] (M x d) for the up
// projection, V_e[H_b, :] (d x M) for the down projection (Eqs. 16, 28-29).
// Each CTA takes an equal contiguous run of tiles and keeps the current
// group's slice resident in shared memory, reloading it only when the group
// changes, slab by slab as the last MMAs of the previous group release each
// slab. Only the token rows stream: x rows (gathered) for the up projection,
// h tiles for the down projection, whose A tile then feeds both halves of the
// d output columns.
//
// Roles (one CTA per SM, 15 warps):
//   warps 0-3   up: owners of a 4-deep ring of gathered x stages (16-byte
//               cp.async of 128 token rows per stage); down: warp 0 brings h
//               tiles (3-deep ring, TMA)
//   warp 4      weight loader: TMA of the group's slabs, once per group run
//   warps 5-6   MMA issuers (warp 5 also owns the TMEM allocation)
//   warps 7-14  epilogue: up, GeLU -> bf16 h staged and stored by TMA; down,
//               weight scale -> fp32 atomic add into y. Warp w reads TMEM lane
//               quarter w % 4 and one half of the accumulator's columns.
// Every wait is bounded; a wait that runs out records kStatusTimeout in the
// status word and the CTA unwinds.
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "decide.cuh"
#include "internal.cuh"
#include "tc_common.cuh"

namespace unif {
namespace tc {
namespace ws {

constexpr int kEpiWarps = 8;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccStride = 256;
constexpr int kMaxSlabs = 16;
constexpr uint32_t kBarBytes = 384;
constexpr uint32_t kMaxSmem = 232448;  // 227 KB opt-in per CTA

// Per-projection layout: warps 0-3 bring A (up: the owners of a 4-deep ring
// of gathered x stages; down: warp 0 alone, 3-deep ring of h tiles by TMA),
// warp 4 loads the weight slabs, warps 5-6 issue the MMAs, warps 7-14 run
// the epilogue. Each epilogue warp owns a 32-row x 32-column staging tile:
// bf16 (64-byte rows, 64-byte swizzle) that a TMA store writes to h, or fp32
// (128-byte rows, 128-byte swizzle) that the warp adds into y.
template <int MODE>
struct Cfg {
  static constexpr int kStagesA = MODE == 0 ? 4 : 3;
  static constexpr int kProducerWarps = MODE == 0 ? 4 : 1;
  static constexpr int kLoaderWarp = 4;
  static constexpr int kMmaWarp = 5;        // warps 5 and 6 issue MMAs
  static constexpr int kMmaWarps = 2;
  static constexpr int kFirstEpiWarp = 7;
  static constexpr int kThreads = 32 * (kFirstEpiWarp + kEpiWarps);
  static constexpr uint32_t kStageRowBytes = MODE == 0 ? 64u : 128u;
  static constexpr uint32_t kStaging = kEpiWarps * 32u * kStageRowBytes;
  static constexpr uint32_t kFixed = 1024 + kStagesA * kStageA + kStaging + kBarBytes;
  static_assert(MODE != 0 || kProducerWarps == kStagesA, "one owner warp per up stage");
  static_assert(kEpiWarps == 8, "two warps per TMEM lane quarter");
};

struct Params {
  // Tiles: numbered here from the group sizes (fill != nullptr: per-group
  // regions of `region` rows, the router's grouping), or the tile list of
  // the grouping kernels.
  const int32_t* fill;
  int G, region;
  int per_cta;  // room for this many tiles of a CTA's run in the shared tile table
  // Down projection with n_slices > 1: the work items are (column slice s,
  // tile), slice-major, each with one sub-tile (n_sub = 1) of bn columns at
  // s bn; only one slice's weight slabs are resident at a time.
  int n_slices;
  const int32_t* n_tiles;
  const int32_t* tile_group;
  const int32_t* tile_row0;  // first row of each tile in row_tok / row_w
  const int32_t* tile_rows;  // rows of each tile that are not padding
  const int32_t* row_tok;
  const float* row_w;
  int n_sub, bn, num_kb;
  int B, M, H, d;
  const __nv_bfloat16* x;
  __nv_bfloat16* h;
  float* y32;
  int* status;
  long long wait_limit;
};

template <int MODE>
__global__ void __launch_bounds__(Cfg<MODE>::kThreads, 1)
ws_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               Params p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived from smem_raw by an offset so that the
  // compiler keeps every access through it in the shared state space
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  constexpr int kStagesA = Cfg<MODE>::kStagesA;
  constexpr int kProducerWarps = Cfg<MODE>::kProducerWarps;
  constexpr int kLoaderWarp = Cfg<MODE>::kLoaderWarp;
  constexpr int kMmaWarp = Cfg<MODE>::kMmaWarp;
  constexpr int kFirstEpiWarp = Cfg<MODE>::kFirstEpiWarp;
  const int n_slabs = p.n_sub * p.num_kb;
  const uint32_t slab_bytes = (uint32_t)p.bn * kBK * 2;
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + kStagesA * kStageA;
  uint8_t* tail = smem + kStagesA * kStageA + (size_t)n_slabs * slab_bytes;
  uint8_t* staging = tail;
  uint64_t* bars = reinterpret_cast<uint64_t*>(tail + Cfg<MODE>::kStaging);
  const uint32_t bar0 = smem_u32(bars);
  auto fullA = [&](int s) { return bar0 + 8u * s; };
  auto emptyA = [&](int s) { return bar0 + 8u * (5 + s); };
  auto wfull = [&](int s) { return bar0 + 8u * (10 + s); };
  auto wempty = [&](int s) { return bar0 + 8u * (10 + kMaxSlabs + s); };
  auto accf = [&](int a) { return bar0 + 8u * (10 + 2 * kMaxSlabs + a); };
  auto acce = [&](int a) { return bar0 + 8u * (12 + 2 * kMaxSlabs + a); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 14 + 2 * kMaxSlabs);
  static_assert(8 * (14 + 2 * kMaxSlabs) + 8 <= kBarBytes, "barrier region");
  // tile table (fill != nullptr): first tile and size of every group, then
  // the group, first row and real rows of each tile of this CTA's run
  int32_t* first_s = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(bars) + kBarBytes);
  int32_t* gcnt_s = first_s + p.G + 1;
  int32_t* run_s = gcnt_s + p.G;  // [3][per_cta]
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesA; ++s) {
      mbar_init(fullA(s), 1);
      mbar_init(emptyA(s), Cfg<MODE>::kMmaWarps);
    }
    // With the down projection's two sub-tiles split between the issuers,
    // each accumulator and each weight slab has a single issuer; otherwise
    // both issuers release every one of them.
    const int owners = (MODE == 1 && p.n_sub == 2) ? 1 : Cfg<MODE>::kMmaWarps;
    for (int s = 0; s < n_slabs; ++s) {
      mbar_init(wfull(s), 1);
      mbar_init(wempty(s), owners);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(accf(a), owners);
      mbar_init(acce(a), kEpiWarps);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  if (p.fill && warp == Cfg<MODE>::kThreads / 32 - 1) {
    // the group sizes are final once the router completed: the up
    // projection waits for it here (the down projection starts after it)
    if (MODE == 0) grid_dep_wait();
    tile_table(p.fill, p.G, p.region, lane, first_s, gcnt_s);
    __syncwarp();
    const int nt = p.n_slices == 1 ? first_s[p.G] : 0;  // (slices: cursors, below)
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
  // every warp converged before the CTA barrier (lane 0 of warp 0 ran the
  // barrier setup, the table warp's lanes ran different trip counts)
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // The up projection reads the router's tile list and rows: it waits for
  // the router here. The down projection needs only the up projection's h
  // (its tile list and rows come from the router, which completed before
  // the up projection started), so only its h loader waits, below, and the
  // weight slabs of its first run load meanwhile.
  if (MODE == 0) grid_dep_wait();
  grid_dep_launch();

  // This CTA's contiguous run of tiles (sizes differ by at most one).
  const int n_tiles = p.fill ? first_s[p.G] : p.n_tiles[0];
  // work items: tiles, or (slice, tile) pairs slice-major; "tile" below
  // names an item index
  const int n_items = n_tiles * p.n_slices;
  const int t_begin = (int)(((long long)blockIdx.x * n_items) / gridDim.x);
  const int t_end = (int)(((long long)(blockIdx.x + 1) * n_items) / gridDim.x);
  // For item v (t_begin <= v < t_end): the weight-slab key (slice * G +
  // group), the tile's first row and real rows. With slices, each thread's
  // lookups move forward through the items, so a cursor over the group table
  // finds the group in amortised constant time.
  int cur_g = 0;
  auto tile_of = [&](int v, int& key, int& r0, int& rows) {
    const int slice = v / n_tiles, k = v - slice * n_tiles;
    int g;
    if (p.fill && p.n_slices == 1) {
      const int j = v - t_begin;
      g = run_s[j];
      r0 = run_s[p.per_cta + j];
      rows = run_s[2 * p.per_cta + j];
    } else if (p.fill) {
      if (k < first_s[cur_g]) cur_g = 0;
      while (first_s[cur_g + 1] <= k) ++cur_g;  // first_s[G] = n_tiles > k
      g = cur_g;
      const int i = k - first_s[g];
      r0 = g * p.region + 128 * i;
      rows = min(128, gcnt_s[g] - 128 * i);
    } else {
      g = p.tile_group[k];
      r0 = p.tile_row0[k];
      rows = p.tile_rows[k];
    }
    key = slice * p.G + g;
  };
  // items of the down projection read h tile (v mod n_tiles); their output
  // columns start at slice * n_sub * bn
  auto item_tile = [&](int v) { return v % n_tiles; };
  auto item_col0 = [&](int v) { return (v / n_tiles) * p.n_sub * p.bn; };

  if (MODE == 0 && warp < kProducerWarps) {
    // ---------------- up: A stage owners (x rows gathered) -----------------
    // Stage sequence number sq = (tile - t_begin) * num_kb + kb; warp w owns
    // the stages with sq = w (mod 5). Lane (rsub, j) copies 16-byte chunk j
    // of rows 4 i + rsub, i = 0..31; the tile's 128 row tokens sit in
    // registers (lane l holds rows l, l + 32, l + 64, l + 96) and reach the
    // copying lane by shuffle.
    const int j = lane & 7, rsub = lane >> 3;
    bool ok = true;
    int seq = 0;
    // the next tile's row tokens, loaded one tile ahead (and its first row
    // index two tiles ahead)
    // (padding rows gather token 0; their h rows are never used)
    int tk_nxt[4];
    int gq, r0_nxt = 0, n_nxt = 0;
    if (t_begin + 1 < t_end) tile_of(t_begin + 1, gq, r0_nxt, n_nxt);
    {
      int r0 = 0, n = 0;
      if (t_begin < t_end) tile_of(t_begin, gq, r0, n);
#pragma unroll
      for (int i = 0; i < 4; ++i) tk_nxt[i] = 32 * i + lane < n ? p.row_tok[r0 + 32 * i + lane] : 0;
    }
    for (int tile = t_begin; tile < t_end && ok; ++tile, seq += p.num_kb) {
      int tk[4];
      const int r0n = r0_nxt, nn = n_nxt;
      if (tile + 2 < t_end) tile_of(tile + 2, gq, r0_nxt, n_nxt);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        tk[i] = tk_nxt[i] < 0 ? 0 : tk_nxt[i];
        if (tile + 1 < t_end) tk_nxt[i] = 32 * i + lane < nn ? p.row_tok[r0n + 32 * i + lane] : 0;
      }
      const int first = (warp - seq % kProducerWarps + kProducerWarps) % kProducerWarps;
      if (first >= p.num_kb) continue;
      const __nv_bfloat16* xj = p.x + j * 8;
      for (int kb = first; kb < p.num_kb; kb += kProducerWarps) {
        const int sq = seq + kb;
        const int stage = sq % kStagesA;
        const uint32_t phase = (uint32_t)(sq / kStagesA) & 1u;
        ok = wait_warp(emptyA(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit);
        if (!ok) break;
        const uint32_t a_dst = sA + stage * kStageA;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int r = 4 * i + rsub;
          const int t = __shfl_sync(0xffffffffu, tk[i >> 3], r & 31);
          cp_async16(a_dst + r * 128u + ((j ^ (r & 7)) << 4), xj + (size_t)t * p.d + kb * kBK);
        }
        cp_async_commit();
        cp_async_wait<0>();
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(fullA(stage));
      }
    }
  } else if (MODE == 1 && warp == 0) {
    // ---------------- down: h tiles by TMA ---------------------------------
    grid_dep_wait();
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = t_begin; tile < t_end && ok; ++tile) {
        for (int kb = 0; kb < p.num_kb; ++kb) {
          if (!wait_bounded(emptyA(stage), phase ^ 1u, abort_flag, p.status, p.wait_limit)) {
            ok = false;
            break;
          }
          mbar_expect_tx(fullA(stage), kStageA);
          tma_load_2d(sA + stage * kStageA, &tmA, fullA(stage), kb * kBK, item_tile(tile) * kBM);
          if (++stage == kStagesA) { stage = 0; phase ^= 1u; }
        }
      }
    }
    __syncwarp();
  } else if (warp == kLoaderWarp) {
    // ---------------- weight slabs, once per group run ---------------------
    // Slab s = ns * num_kb + kb holds bn rows x 64 reduction elements. Run r
    // (r >= 1) reuses a slab after the MMAs of run r - 1 released it.
    if (lane == 0) {
      int run = 0, g_prev = -1;
      bool ok = true;
      for (int tile = t_begin; tile < t_end && ok; ++tile) {
        int g, r0_unused, rows_unused;
        tile_of(tile, g, r0_unused, rows_unused);
        if (g == g_prev) continue;
        g_prev = g;
        // key = slice * G + group; group = e * B + blk
        const int slice = g / p.G, grp = g - slice * p.G;
        const int e = grp / p.B, blk = grp % p.B;
        const int col0 = slice * p.n_sub * p.bn;  // the slice's first output column
        for (int s = 0; s < n_slabs; ++s) {
          const int ns = s / p.num_kb, kb = s % p.num_kb;
          if (run > 0 &&
              !wait_bounded(wempty(s), (uint32_t)(run - 1) & 1u, abort_flag, p.status, p.wait_limit)) {
            ok = false;
            break;
          }
          mbar_expect_tx(wfull(s), slab_bytes);
          if (MODE == 0)  // w_up viewed [(K+1) H][d]
            tma_load_2d(sB + s * slab_bytes, &tmB, wfull(s), kb * kBK, e * p.H + blk * p.M + ns * p.bn);
          else            // w_down viewed [(K+1) d][H]
            tma_load_2d(sB + s * slab_bytes, &tmB, wfull(s), blk * p.M + kb * kBK,
                        e * p.d + col0 + ns * p.bn);
        }
        ++run;
      }
    }
    __syncwarp();
  } else if (warp >= kMmaWarp && warp < kMmaWarp + Cfg<MODE>::kMmaWarps) {
    // ---------------- MMA issuers -------------------------------------------
    // Two warps issue MMAs side by side: an MMA issue returns only once the
    // tensor pipe takes it, so one issuer's bookkeeping between MMA groups
    // would leave the pipe idle; the other issuer's MMAs fill those gaps.
    // Up (and a single-sub-tile down): warp m computes columns
    // [m bn/2, (m+1) bn/2) of every accumulator, and every stage, slab and
    // accumulator barrier counts both warps' releases. Down with two
    // sub-tiles: warp m computes sub-tile m; the A stages count both warps,
    // each sub-tile's slabs and accumulator only their own issuer.
    // Within a warp the whole warp runs the loop (warp-uniform values) and an
    // elected lane issues; the next stage's barrier is tested before the
    // current stage's MMAs go out and read back after.
    const int m = warp - kMmaWarp;
    const bool split_n = !(MODE == 1 && p.n_sub == 2);
    // A stages read by one sub-tile only are freed after their MMAs (the up
    // projection, and sliced down projections); otherwise after the tile's
    // last sub-tile
    const bool a_once = MODE == 0 || p.n_sub == 1;
    const int n_mma = split_n ? p.bn / 2 : p.bn;
    const uint32_t idesc = idesc_bf16(kBM, n_mma);
    // B rows and accumulator columns this warp covers (split_n), in 16-byte
    // descriptor units and TMEM columns
    const uint64_t b_off = split_n ? (uint64_t)(m * n_mma * 128 / 16) : 0ull;
    const uint32_t d_off = split_n ? (uint32_t)(m * n_mma) : 0u;
    const uint64_t a_desc0 = sw128_desc(sA), b_desc0 = sw128_desc(sB) + b_off;
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    int run = -1, g_prev = -1;
    bool ok = true;
    bool ready = false;  // fullA(stage) known complete
    // groups of this tile and the next, loaded ahead of use
    int g_cur = -1, g_nxt = -1, r0_unused, rows_unused;
    if (t_begin < t_end) tile_of(t_begin, g_cur, r0_unused, rows_unused);
    if (t_begin + 1 < t_end) tile_of(t_begin + 1, g_nxt, r0_unused, rows_unused);
    for (int tile = t_begin; tile < t_end && ok; ++tile) {
      const int g = g_cur, gn = g_nxt;
      g_cur = g_nxt;
      if (tile + 2 < t_end) tile_of(tile + 2, g_nxt, r0_unused, rows_unused);
      const bool first_of_run = g != g_prev;
      if (first_of_run) { ++run; g_prev = g; }
      // release the slabs after this tile if the next tile of the run
      // belongs to another group
      const bool release = tile + 1 < t_end && gn != g;
      const int st0 = stage;
      const uint32_t ph0 = phase;
      for (int ns = 0; ns < p.n_sub && ok; ++ns) {
        const bool mine = split_n || ns == m;
        if (mine) {
          if (!wait_warp(acce(acc), acc_phase ^ 1u, abort_flag, p.status, p.wait_limit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + (uint32_t)acc * kAccStride + d_off;
          int st = st0;
          uint32_t ph = ph0;
          // stages are waited for in the first sub-tile this warp computes
          const bool first_pass = split_n ? ns == 0 : true;
          for (int kb = 0; kb < p.num_kb; ++kb) {
            const int s = ns * p.num_kb + kb;
            const int st_n = st + 1 == kStagesA ? 0 : st + 1;
            const uint32_t ph_n = st + 1 == kStagesA ? ph ^ 1u : ph;
            if (first_pass && !ready &&
                !wait_warp(fullA(st), ph, abort_flag, p.status, p.wait_limit)) {
              ok = false;
              break;
            }
            if (first_of_run &&
                !wait_warp(wfull(s), (uint32_t)run & 1u, abort_flag, p.status, p.wait_limit)) {
              ok = false;
              break;
            }
            // the stage after this one, in ring order (the next tile's first
            // stage after the last k-block); read back after the MMAs
            const uint32_t next_done =
                first_pass && (a_once || kb + 1 < p.num_kb) ? mbar_test(fullA(st_n), ph_n) : 0u;
            tc_fence_after();
            // descriptor start addresses advance in 16-byte units: +2 per 32 bytes
            const uint64_t a_desc = a_desc0 + (uint64_t)(st * (kStageA >> 4));
            const uint64_t b_desc = b_desc0 + (uint64_t)(s * (slab_bytes >> 4));
            if (elect_one()) {
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                umma_bf16(d_tmem, a_desc + 2 * k, b_desc + 2 * k, idesc, (kb | k) != 0 ? 1u : 0u);
              if (release) umma_commit(wempty(s));
              if (a_once) umma_commit(emptyA(st));  // one pass over A: free it now
            }
            ready = __all_sync(0xffffffffu, next_done != 0u);
            st = st_n;
            ph = ph_n;
          }
          if (!ok) break;
          if (elect_one()) umma_commit(accf(acc));
          __syncwarp();
        }
        // (the other warp's sub-tile: its accumulator and slabs have that
        // warp as their only issuer; an arrival from this warp could run a
        // whole tile or group ahead of the MMAs it stands for)
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      }
      if (!ok) break;
      // advance the A ring past this tile; a down projection with several
      // sub-tiles frees its stages only after all of them read them
      for (int kb = 0; kb < p.num_kb; ++kb) {
        if (!a_once) {
          if (elect_one()) umma_commit(emptyA(stage));
          __syncwarp();
        }
        if (++stage == kStagesA) { stage = 0; phase ^= 1u; }
      }
      if (!a_once) ready = false;
    }
  } else if (warp >= kFirstEpiWarp) {
    // ---------------- epilogue ----------------------------------------------
    const int q = warp & 3;
    const int half = (warp - kFirstEpiWarp) >> 2;
    const int cols = p.bn / 2;
    const int c_begin = half * cols;
    int acc = 0;
    uint32_t acc_phase = 0;
    // down: this thread's row token (-1 for a padding row) and weight, one
    // tile ahead
    int t_nxt = -1;
    float w_nxt = 0.f;
    int gq, r0_nxt = 0, n_nxt = 0;
    if (MODE == 1 && t_begin + 1 < t_end) tile_of(t_begin + 1, gq, r0_nxt, n_nxt);
    if (MODE == 1 && t_begin < t_end) {
      int r0, n;
      tile_of(t_begin, gq, r0, n);
      if (q * 32 + lane < n) {
        t_nxt = p.row_tok[r0 + q * 32 + lane];
        w_nxt = p.row_w[r0 + q * 32 + lane];
      }
    }
    uint8_t* stg = staging + (size_t)(warp - kFirstEpiWarp) * 32 * Cfg<MODE>::kStageRowBytes;
    const uint32_t stg_s = smem_u32(stg);
    bool ok = true;
    for (int tile = t_begin; tile < t_end && ok; ++tile) {
      const int row0 = tile * kBM;
      const int t_cur = t_nxt;
      const float w_cur = w_nxt;
      if (MODE == 1 && tile + 1 < t_end) {
        const int r = r0_nxt + q * 32 + lane;
        t_nxt = q * 32 + lane < n_nxt ? p.row_tok[r] : -1;
        w_nxt = q * 32 + lane < n_nxt ? p.row_w[r] : 0.f;
        if (tile + 2 < t_end) tile_of(tile + 2, gq, r0_nxt, n_nxt);
      }
      for (int ns = 0; ns < p.n_sub; ++ns) {
        if (!wait_warp(accf(acc), acc_phase, abort_flag, p.status, p.wait_limit)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)acc * kAccStride;
        if (MODE == 0) {
          // h = bf16(GeLU(acc)), 32 columns per pass: each thread writes its
          // row's 64 bytes into the warp's staging tile (16-byte chunk c of
          // row r at c ^ ((r >> 1) & 3), the 64-byte swizzle), and lane 0
          // stores the 32 x 32 tile to h with TMA. The tile is rewritten only
          // after the previous store has read it.
          const uint32_t sw = (uint32_t)(lane >> 1) & 3u;
          for (int c = 0; c < cols; c += 32) {
            uint32_t o[16];
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              float v[16];
              tmem_ld16(t_row + c_begin + c + 16 * hh, v);
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) o[8 * hh + jj] = gelu2_bf16x2(v[2 * jj], v[2 * jj + 1]);
            }
            if (lane == 0) bulk_wait_read();
            __syncwarp();
#pragma unroll
            for (int jj = 0; jj < 4; ++jj)
              *reinterpret_cast<uint4*>(stg + lane * 64 + ((jj ^ sw) << 4)) =
                  make_uint4(o[4 * jj], o[4 * jj + 1], o[4 * jj + 2], o[4 * jj + 3]);
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tmA, stg_s, ns * p.bn + c_begin + c, row0 + q * 32);
              bulk_commit();
            }
          }
        } else {
          // y[tok] += w * acc, 32 columns per pass: thread = row stages its
          // 128 scaled bytes (chunk c at c ^ (r & 7)); then 8 lanes per row
          // add 4 rows x 128 contiguous bytes per instruction.
          float* stf = reinterpret_cast<float*>(stg);
          const int r_sub = lane >> 3, c8 = lane & 7;
          float* ybase = p.y32 + item_col0(tile) + ns * p.bn + c_begin;
          for (int c = 0; c < cols; c += 32) {
            float v[32];
            tmem_ld32(t_row + c_begin + c, v);
#pragma unroll
            for (int jj = 0; jj < 8; ++jj)
              *reinterpret_cast<float4*>(stf + lane * 32 + ((jj ^ (lane & 7)) << 2)) =
                  make_float4(w_cur * v[4 * jj], w_cur * v[4 * jj + 1], w_cur * v[4 * jj + 2],
                              w_cur * v[4 * jj + 3]);
            __syncwarp();
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int r = 4 * i + r_sub;
              const int tr = __shfl_sync(0xffffffffu, t_cur, r);
              const float4 val = *reinterpret_cast<const float4*>(stf + r * 32 + ((c8 ^ (r & 7)) << 2));
              if (tr >= 0)
                atomicAdd(reinterpret_cast<float4*>(ybase + (size_t)tr * p.d + c + c8 * 4), val);
            }
            __syncwarp();
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acce(acc));
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      }
    }
    if (MODE == 0 && lane == 0) bulk_wait_all();  // h complete before the CTA retires
  }
  // every warp converged before the CTA barrier (an epilogue warp's lane 0
  // may still wait for its h stores)
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

}  // namespace ws
}  // namespace tc

// Chooses the weight-stationary kernels where their shapes and shared memory
// allow: the up projection needs the whole block width in one accumulator
// (M <= 256); the down projection reuses each h tile across all output
// column sub-tiles, so the tile's M / 64 reduction stages must fit its A ring.
// A handle created with UNIF_MOE_GEMM_STREAMING keeps the streaming kernels.
int gemm_ws_setup(unif_moe_layer* L) {
  using namespace tc::ws;
  L->up_ws = L->down_ws = false;
  if (L->gemm_streaming) return UNIF_MOE_OK;
  // the tile table (first tile and size of every group, the tiles of one
  // CTA's run) follows the barriers
  const uint64_t per_cta = (uint64_t)((L->max_tiles + L->n_sm - 1) / L->n_sm);
  const uint64_t table =
      L->fused_group ? ((uint64_t)(2 * L->G + 1 + 3 * per_cta) * 4 + 15) / 16 * 16 : 0;
  const uint64_t up_slabs = (uint64_t)L->up_nsub * (L->d / tc::kBK);
  const uint64_t up_smem =
      Cfg<0>::kFixed + up_slabs * (uint64_t)L->up_bn * tc::kBK * 2 + table;
  if (L->up_nsub == 1 && up_slabs <= (uint64_t)kMaxSlabs && up_smem <= kMaxSmem) {
    if (cudaFuncSetAttribute(ws_gemm_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)up_smem) != cudaSuccess) {
      set_error("cudaFuncSetAttribute failed for the weight-stationary up kernel");
      return UNIF_MOE_ERR_CUDA;
    }
    if (!encode_bf16_map(&L->tm_h_st, L->ws.hbuf, L->M, (uint64_t)L->max_rows, 32, 32, 64)) {
      set_error("cuTensorMapEncodeTiled failed for the h store map");
      return UNIF_MOE_ERR_CUDA;
    }
    L->up_ws = true;
    L->up_ws_smem = (uint32_t)up_smem;
  }
  // Down: every sub-tile's slabs resident (the h tile feeds all of them),
  // where they fit; else one column slice of the output at a time (items =
  // (slice, tile)), with the widest slice whose slabs fit. Slices re-read
  // each h tile once per slice: they pay off only where the h tile fits the
  // A ring (measured on GB300: ViT-B 440 -> 378 us; BERT-base, whose h tile
  // needs 6 stages, and the stress layer, whose 1.2 GB h is read from HBM,
  // ran slower than the streaming kernel).
  const int down_kb = L->M / tc::kBK;
  const uint64_t down_slabs = (uint64_t)L->down_nsub * down_kb;
  const uint64_t down_smem =
      Cfg<1>::kFixed + down_slabs * (uint64_t)L->down_bn * tc::kBK * 2 + table;
  int bn = 0, nsub = 0, slices = 0;
  uint64_t smem = 0;
  if (down_kb <= Cfg<1>::kStagesA && down_slabs <= (uint64_t)kMaxSlabs && down_smem <= kMaxSmem) {
    bn = L->down_bn; nsub = L->down_nsub; slices = 1; smem = down_smem;
  } else if (down_kb <= Cfg<1>::kStagesA) {
    const uint64_t small_table =
        L->fused_group ? ((uint64_t)(2 * L->G + 1) * 4 + 15) / 16 * 16 : 0;
    for (int b = 256; b >= 64; b -= 64) {
      if (L->d % b != 0) continue;
      const uint64_t sm = Cfg<1>::kFixed + (uint64_t)down_kb * b * tc::kBK * 2 + small_table;
      if (sm <= kMaxSmem) {
        bn = b; nsub = 1; slices = L->d / b; smem = sm;
        break;
      }
    }
  }
  if (bn > 0) {
    if (cudaFuncSetAttribute(ws_gemm_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess) {
      set_error("cudaFuncSetAttribute failed for the weight-stationary down kernel");
      return UNIF_MOE_ERR_CUDA;
    }
    if (!encode_bf16_map(&L->tm_wdown_ws, L->w_down, L->H, ((uint64_t)L->K + 1) * L->d, tc::kBK,
                         bn, 128)) {
      set_error("cuTensorMapEncodeTiled failed for the down weight slabs");
      return UNIF_MOE_ERR_CUDA;
    }
    L->down_ws = true;
    L->down_ws_smem = (uint32_t)smem;
    L->ws_down_bn = bn;
    L->ws_down_nsub = nsub;
    L->down_slices = slices;
  }
  return UNIF_MOE_OK;
}

static tc::ws::Params ws_params(unif_moe_layer* L, const void* x) {
  tc::ws::Params p;
  p.fill = L->fused_group ? L->ws.grp_fill : nullptr;
  p.G = L->G;
  p.region = L->region_rows;
  p.per_cta = (int)((L->max_tiles + L->n_sm - 1) / L->n_sm);
  p.n_slices = 1;
  p.n_tiles = L->ws.n_tiles; p.tile_group = L->ws.tile_group; p.tile_row0 = L->ws.tile_row0;
  p.tile_rows = L->ws.tile_rows; p.row_tok = L->ws.row_tok; p.row_w = L->ws.row_w;
  p.B = L->B; p.M = L->M; p.H = L->H; p.d = L->d;
  p.x = static_cast<const __nv_bfloat16*>(x);
  p.h = static_cast<__nv_bfloat16*>(L->ws.hbuf);
  p.y32 = L->ws.y32;
  p.status = L->ws.status;
  p.wait_limit = gemm_wait_limit();
  return p;
}

cudaError_t launch_up_ws(unif_moe_layer* L, const void* x, cudaStream_t s) {
  tc::ws::Params p = ws_params(L, x);
  p.n_sub = L->up_nsub; p.bn = L->up_bn; p.num_kb = L->d / tc::kBK;
  return launch_dependent(tc::ws::ws_gemm_kernel<0>, dim3(L->n_sm), dim3(tc::ws::Cfg<0>::kThreads),
                          L->up_ws_smem, s, L->tm_h_st, L->tm_wup, p);
}

cudaError_t launch_down_ws(unif_moe_layer* L, cudaStream_t s) {
  tc::ws::Params p = ws_params(L, nullptr);
  p.n_sub = L->ws_down_nsub; p.bn = L->ws_down_bn; p.num_kb = L->M / tc::kBK;
  p.n_slices = L->down_slices;
  return launch_dependent(tc::ws::ws_gemm_kernel<1>, dim3(L->n_sm), dim3(tc::ws::Cfg<1>::kThreads),
                          L->down_ws_smem, s, L->tm_h, L->tm_wdown_ws, p);
}

}  // namespace unif
