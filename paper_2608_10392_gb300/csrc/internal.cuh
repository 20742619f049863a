// Internal declarations shared by the translation units of the UniF-MoE
// library: the handle layout and the kernel launchers. Not part of the ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/unif_moe.h"

namespace unif {

// Rows per tile of the grouped GEMMs (the tcgen05 MMA M).
constexpr int kTileRows = 128;
// Tokens per block in the router and in the permute kernels.
constexpr int kRouterTokens = 64;
constexpr int kChunkTokens = 256;
// Status-word bits written by kernels.
constexpr int kStatusTimeout = 1;
constexpr int kStatusBadIndex = 2;

// Programmatic dependent launch. The kernels of a forward after the router
// are launched with launch_dependent: each may start (prologue: barriers,
// tensor memory, loads that need no result of the kernel before it) while
// the kernel before it still runs, and waits in grid_dep_wait, which
// returns once that kernel has completed and its writes are visible. A
// kernel lets its dependent start with grid_dep_launch. In a kernel launched
// without the attribute grid_dep_wait returns at once.
__device__ __forceinline__ void grid_dep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void grid_dep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

struct Workspace {
  // Routing records of the last forward (one entry per token slot).
  float* alpha = nullptr;        // [T]
  int32_t* b = nullptr;          // [T]
  int32_t* k = nullptr;          // [T]
  uint64_t* shr_mask = nullptr;  // [T]
  uint64_t* exp_mask = nullptr;  // [T] selected residual experts
  float* s = nullptr;            // [T][K] affinities by expert index (Eq. 24)
  // Group table.
  int32_t* chunk_cnt = nullptr;  // [G][T/32]: counts, then exclusive offsets
  int32_t* grp_cnt = nullptr;    // [G]
  int32_t* grp_off = nullptr;    // [G+1] padded offsets
  int32_t* n_tiles = nullptr;    // [1]
  int32_t* tile_group = nullptr; // [max_tiles]
  int32_t* tile_row0 = nullptr;  // [max_tiles]
  int32_t* tile_rows = nullptr;  // [max_tiles] rows of the tile that are not padding
  int32_t* row_tok = nullptr;    // [max_rows], or [G][region] when the router groups (-1 = padding)
  float* row_w = nullptr;        // same layout
  // Fill counters of the grouping inside the router (bf16 layers).
  int32_t* grp_fill = nullptr;   // [G] rows reserved per group (the group sizes once the router completed)
  // Intermediate activations h = GeLU(x K_e[:, H_b]) per row, and the fp32
  // output accumulator.
  void* hbuf = nullptr;          // [max_rows][M] (layer dtype)
  float* y32 = nullptr;          // [max_tokens][d]
  // The expert-tile FFN's second accumulator: a pass adds into one of the
  // two and zeroes the other for the next pass, so that the combine only
  // reads (acc_sel names the one the next pass adds into).
  float* y32_b = nullptr;        // [pass_tokens][d]
  // Expert weights repacked into the expert-tile FFN's 16 KB operand slabs.
  void* wk_slabs = nullptr;      // K_e: [K+1][H/128][d/64] slabs
  void* wv_slabs = nullptr;      // V_e: [K+1][H/128][2][d/128] slabs
  // Host-buffer forward staging.
  void* xn = nullptr;             // [max_tokens][d] LN(x) of a norm-first sublayer
  // Staging buffers of the host-buffer forwards, two slots (the pipelined
  // forward alternates between them; the synchronous one uses slot 0).
  void* x_stage[2] = {nullptr, nullptr};
  void* out_stage[2] = {nullptr, nullptr};
  uint8_t* mask_stage[2] = {nullptr, nullptr};
  int32_t* b_stage[2] = {nullptr, nullptr};
  int32_t* k_stage[2] = {nullptr, nullptr};
  int* status = nullptr;         // device status word
  // Backward pass (UNIF_MOE_FEATURE_BACKWARD).
  void* w_upT = nullptr;         // [K+1][d][H] keys transposed (layer dtype)
  void* w_downT = nullptr;       // [K+1][H][d] values transposed
  void* da = nullptr;            // [max_rows][M] dL/da per group row (rows as h)
  void* hw = nullptr;            // [max_rows][M] w GeLU(a) per group row
  float* dwt = nullptr;          // [max_tokens][K+1] dL/dalpha, dL/ds_j per token
  float* dz = nullptr;           // [max_tokens][K+1] dL/dz (router logits)
  float* wrT = nullptr;          // [K+1][d] the router's W* transposed (fp32)
  float* gram = nullptr;         // [K+1][K+1] W*^T W* - I
  // Diagnostics of Sec. II-B (UNIF_MOE_FEATURE_DIAGNOSTICS).
  uint32_t* diag_sets = nullptr; // [K][K][ceil(H/32)] aligned channel sets S_ij
  int* diag_counts = nullptr;    // [K][K] |S_ij|
  int32_t* diag_pair = nullptr;  // [max_tokens][2] top-2 pair
  float* diag_wts = nullptr;     // [max_tokens][2] its normalised weights
  int32_t* diag_q = nullptr;     // [max_tokens][K] residual order
  float* diag_E = nullptr;       // [max_tokens][K][d] E_e(x)
  float* diag_ES = nullptr;      // [max_tokens][K][d] E_e^{S_ij}(x)
};

}  // namespace unif

struct unif_moe_layer {
  int d = 0, H = 0, K = 0, B = 0, M = 0, G = 0;
  int dtype = 0;
  int max_tokens = 0;
  unif_moe_thresholds th{};
  float tau = 0.f;
  int cb_max = 0;
  int64_t max_rows = 0;
  int64_t max_tiles = 0;
  int max_chunks = 0;
  int router_cols = 0;      // 1 + K + B
  int router_cols_pad = 0;  // padded to a multiple of 32
  int n_sm = 0;
  // bf16 layers: the tensor-core router also lays out the rows of each group
  // in its own region of region_rows rows (no separate grouping kernels).
  bool fused_group = false;
  int region_rows = 0;
  bool tile_list = false;  // a streaming GEMM reads the tile list: build it after the router
  // A forward of more than pass_tokens tokens runs in passes of pass_tokens
  // (bf16 layers): the fp32 accumulator rows of one pass stay in L2. rec0 is
  // the first token of the pass being launched; the routing records of token
  // t of the pass are at rec0 + t.
  int pass_tokens = 0;
  int rec0 = 0;
  unsigned features = 0;        // UNIF_MOE_FEATURE_* workspaces allocated at create time
  bool gemm_streaming = false;  // UNIF_MOE_GEMM_STREAMING: never the weight-stationary kernels
  int device = 0;
  bool loaded = false;
  bool y_dirty = false;  // accumulator / grouping counters may hold state of a forward cut short
  int last_T = -1;
  int last_pass_T = 0;  // tokens of the last forward's last pass
  // Weights (device, owned).
  float* wr = nullptr;      // [d][router_cols_pad]: W_shr, W_g, mu_1..mu_B (fp32)
  __nv_bfloat16* wr_bf = nullptr;  // [router_cols_pad][d] the same matrix in bf16 (bf16 layers)
  float* bias = nullptr;    // [K+1]
  void* w_up = nullptr;     // [K+1][H][d]
  void* w_down = nullptr;   // [K+1][d][H]
  unif::Workspace ws;
  // tcgen05 path: tensor maps of the weights and of h (encoded once).
  CUtensorMap tm_wup;
  CUtensorMap tm_wdown;
  CUtensorMap tm_h;
  CUtensorMap tm_h_st;  // h as 32 x 32 store boxes (64-byte swizzle), up-projection epilogue
  CUtensorMap tm_wr;
  int up_bn = 0, up_nsub = 0, down_bn = 0, down_nsub = 0;
  // Weight-stationary kernels (when the group's weight slice fits in shared
  // memory) and their dynamic shared-memory sizes.
  bool up_ws = false, down_ws = false;
  uint32_t up_ws_smem = 0, down_ws_smem = 0;
  // weight-stationary down projection: sub-tile width and count, and the
  // number of output column slices run as separate work items
  int ws_down_bn = 0, ws_down_nsub = 0, down_slices = 1;
  CUtensorMap tm_wdown_ws;  // w_down slabs of ws_down_bn rows
  // Expert-tile FFN (both projections in one kernel, rows grouped by
  // expert): its weight maps (128 x 64 slabs), shared memory and ring depth.
  bool ffn_fused = false;
  int acc_sel = 0;  // expert-tile FFN: the accumulator the next pass adds into (0: y32, 1: y32_b)
  CUtensorMap tm_fk, tm_fv;  // the repacked K_e / V_e slabs, boxes of one half-slab
  int ffn_pairs = 0;         // CTA pairs launched (clusters of two)
  int ffn_per_cta = 0, ffn_slots = 0;  // pair tiles per pair (run table), ring half-slabs
  uint32_t ffn_smem = 0;
  // backward: transposed weights and the per-row gradient buffers
  CUtensorMap tm_wdownT;    // w_downT [(K+1) H][d], boxes of 64 x up_bn
  CUtensorMap tm_wupT;      // w_upT [(K+1) d][H], boxes of 64 x down_bn
  CUtensorMap tm_da;        // da [max_rows][M], boxes of 64 x 128 (dx GEMM A operand)
  CUtensorMap tm_da_q;      // da, boxes of 64 x 32 (weight-gradient operand)
  CUtensorMap tm_hw_q;      // hw, boxes of 64 x 32
  uint32_t bwd_hidden_smem = 0, bwd_wgrad_smem = 0;
  // Pipelined host-buffer forwards (UNIF_MOE_FEATURE_HOST_IO): the handle's
  // copy streams, and per staging slot the events that order its reuse
  // (input landed, kernels done, output copied out).
  cudaStream_t copy_in = nullptr, copy_out = nullptr;
  cudaEvent_t ev_in[2] = {nullptr, nullptr};
  cudaEvent_t ev_comp[2] = {nullptr, nullptr};
  cudaEvent_t ev_out[2] = {nullptr, nullptr};
  int host_slot = 0;  // slot of the next pipelined forward
  // Optional caller-owned timing events recorded at the stage boundaries.
  cudaEvent_t stage_ev[6] = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
};

namespace unif {

void set_error(const char* fmt, ...);

// Load time.
cudaError_t launch_prototypes(unif_moe_layer* L, const void* w_router, const float* bias,
                              cudaStream_t s);
// Forward steps.
cudaError_t launch_router(unif_moe_layer* L, const void* x, const uint8_t* mask, int T,
                          int32_t* b_out, int32_t* k_out, cudaStream_t s);
cudaError_t launch_permute(unif_moe_layer* L, int T, cudaStream_t s);
cudaError_t launch_combine(unif_moe_layer* L, void* out, int T, cudaStream_t s);
// The fp32 accumulator the pass being launched adds into.
inline float* acc_cur(const unif_moe_layer* L);
cudaError_t launch_layernorm(unif_moe_layer* L, const void* x, void* out, const uint8_t* mask,
                             const void* gamma, const void* beta, float eps, int T,
                             cudaStream_t s);
cudaError_t launch_combine_residual(unif_moe_layer* L, const void* x, void* out,
                                    const uint8_t* mask, const void* gamma, const void* beta,
                                    float eps, bool norm, int T, cudaStream_t s);
// Tile list from the router's group sizes, for streaming grouped GEMMs.
cudaError_t launch_tile_list(unif_moe_layer* L, cudaStream_t s);
// The same from group sizes at `sizes` (the forward's, for the backward).
cudaError_t launch_tile_list_from(unif_moe_layer* L, const int32_t* sizes, cudaStream_t s);
cudaError_t launch_sort_affinities(unif_moe_layer* L, int T, int32_t* q, float* p,
                                   cudaStream_t s);
int forward_chunks(int T);
cudaError_t launch_gemms_simt(unif_moe_layer* L, const void* x, int T, cudaEvent_t mid,
                              cudaStream_t s);
cudaError_t router_setup(unif_moe_layer* L);
// tcgen05 path.
int gemm_tc_setup(unif_moe_layer* L);  // tensor maps of weights and h; returns UNIF_MOE_* code
cudaError_t launch_gemms_tc(unif_moe_layer* L, const void* x, int T, cudaEvent_t mid,
                            cudaStream_t s);
cudaError_t launch_timeout_probe(unif_moe_layer* L, int timeout_us, cudaStream_t s);
int gemm_ws_setup(unif_moe_layer* L);  // picks the weight-stationary kernels where they fit
cudaError_t launch_up_ws(unif_moe_layer* L, const void* x, cudaStream_t s);
cudaError_t launch_down_ws(unif_moe_layer* L, cudaStream_t s);
bool ffn_fused_fits(int d, int H, int M);
int gemm_fused_setup(unif_moe_layer* L);  // the expert-tile FFN's maps and shared memory
cudaError_t launch_ffn_fused(unif_moe_layer* L, const void* x, cudaStream_t s);
cudaError_t launch_repack_slabs(unif_moe_layer* L, cudaStream_t s);  // after the weights load
long long gemm_wait_limit();
bool encode_bf16_map(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows,
                     uint32_t box_cols, uint32_t box_rows, int swizzle_bytes);  // clock cycles before a bounded wait gives up
int router_tc_setup(unif_moe_layer* L);
// Whether the tensor-core router's shared memory holds the grouping's
// counters (and at least one tile of staged rows) for these sizes.
bool router_can_group(int Cp, int K, int G);
cudaError_t launch_router_tc(unif_moe_layer* L, const void* x, const uint8_t* mask, int T,
                             int32_t* b_out, int32_t* k_out, cudaStream_t s);
cudaError_t launch_down_streaming(unif_moe_layer* L, const CUtensorMap& tmA,
                                  const CUtensorMap& tmB, const float* row_w, float* out,
                                  cudaStream_t s);
// Backward pass (backward.cu).
int backward_setup(unif_moe_layer* L);  // workspace maps and kernel attributes
cudaError_t launch_transpose_weights(unif_moe_layer* L, cudaStream_t s);
int backward_run(unif_moe_layer* L, const void* x, const void* dy, int T, const uint8_t* mask,
                 float* dx, float* dw_up, float* dw_down, float* dw_router, float* dbias,
                 float lambda_div, float* l_div, cudaStream_t s);
// Diagnostics (diagnostics.cu); 0 or -1 (CUDA failure).
int diag_alignment(unif_moe_layer* L, float delta, float* rho, cudaStream_t s);
int diag_demand(unif_moe_layer* L, const void* x, int T, const void* w_res, float delta,
                float eps, int32_t* k_eps, float* err, int32_t* pair_out, cudaStream_t s);

inline float* acc_cur(const unif_moe_layer* L) {
  return L->ffn_fused && L->acc_sel ? L->ws.y32_b : L->ws.y32;
}

}  // namespace unif
