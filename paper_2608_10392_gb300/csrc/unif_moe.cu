// Host side of the UniF-MoE C ABI declared in include/unif_moe.h: argument
// checks, workspace allocation at create time, and the launch sequence of a
// forward pass
//   router (Eqs. 17-27; bf16 layers also group the rows, Eqs. 28-29) ->
//   [fp32 layers: permute] -> expert-tile FFN (bf16, d <= 384) or grouped
//   up/down GEMMs (Eq. 16) -> combine (Eq. 30).
#include <algorithm>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>
#include <vector>

#include <new>

#include "internal.cuh"

namespace unif {

static thread_local char g_err[512] = "";

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}

}  // namespace unif

using unif::set_error;

namespace {

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
    else prev = -1;
  }
  ~DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

#define CK(call)                                                              \
  do {                                                                        \
    cudaError_t e_ = (call);                                                  \
    if (e_ != cudaSuccess) {                                                  \
      set_error("%s failed: %s", #call, cudaGetErrorString(e_));              \
      return UNIF_MOE_ERR_CUDA;                                               \
    }                                                                         \
  } while (0)

template <typename T>
int dalloc(T** p, size_t count) {
  *p = nullptr;
  if (count == 0) count = 1;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), sizeof(T) * count);
  if (e != cudaSuccess) {
    set_error("cudaMalloc of %zu bytes failed: %s", sizeof(T) * count, cudaGetErrorString(e));
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

void free_all(unif_moe_layer* L) {
  void* ptrs[] = {L->wr, L->wr_bf, L->bias, L->w_up, L->w_down, L->ws.alpha, L->ws.b, L->ws.k,
                  L->ws.shr_mask, L->ws.exp_mask, L->ws.s, L->ws.chunk_cnt,
                  L->ws.grp_cnt, L->ws.grp_off, L->ws.n_tiles, L->ws.tile_group,
                  L->ws.tile_row0, L->ws.row_tok, L->ws.row_w, L->ws.hbuf, L->ws.y32,
                  L->ws.xn, L->ws.x_stage[0], L->ws.out_stage[0], L->ws.mask_stage[0],
                  L->ws.b_stage[0], L->ws.k_stage[0], L->ws.x_stage[1], L->ws.out_stage[1],
                  L->ws.mask_stage[1], L->ws.b_stage[1], L->ws.k_stage[1], L->ws.status,
                  L->ws.grp_fill,
                  L->ws.tile_rows, L->ws.w_upT, L->ws.w_downT, L->ws.da, L->ws.hw,
                  L->ws.dwt, L->ws.dz, L->ws.wrT, L->ws.gram, L->ws.diag_sets,
                  L->ws.diag_counts, L->ws.diag_pair, L->ws.diag_wts, L->ws.diag_q,
                  L->ws.diag_E, L->ws.diag_ES, L->ws.wk_slabs, L->ws.wv_slabs, L->ws.y32_b};
  for (void* q : ptrs)
    if (q) cudaFree(q);
  for (int i = 0; i < 2; ++i) {
    if (L->ev_in[i]) cudaEventDestroy(L->ev_in[i]);
    if (L->ev_comp[i]) cudaEventDestroy(L->ev_comp[i]);
    if (L->ev_out[i]) cudaEventDestroy(L->ev_out[i]);
  }
  if (L->copy_in) cudaStreamDestroy(L->copy_in);
  if (L->copy_out) cudaStreamDestroy(L->copy_out);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t elt_size(const unif_moe_layer* L) { return L->dtype == UNIF_MOE_BF16 ? 2 : 4; }

}  // namespace

extern "C" {

void unif_moe_default_thresholds(unif_moe_thresholds* th) {
  if (!th) return;
  th->tau = NAN;
  th->alpha_fixed = NAN;
  th->beta_fixed = NAN;
  th->topk_fixed = 0;
  th->prefix_blocks = 0;
}

const char* unif_moe_last_error(void) { return unif::g_err; }

void unif_moe_default_options(unif_moe_options* opts) {
  if (!opts) return;
  opts->features = UNIF_MOE_FEATURES_DEFAULT;
  opts->gemm_kernels = UNIF_MOE_GEMM_AUTO;
}

int unif_moe_create(unif_moe_t* out, int d_model, int d_ff, int n_experts, int n_blocks,
                    const unif_moe_thresholds* th, unif_moe_dtype dtype, int max_tokens) {
  return unif_moe_create_ex(out, d_model, d_ff, n_experts, n_blocks, th, dtype, max_tokens,
                            nullptr);
}

int unif_moe_create_ex(unif_moe_t* out, int d_model, int d_ff, int n_experts, int n_blocks,
                       const unif_moe_thresholds* th, unif_moe_dtype dtype, int max_tokens,
                       const unif_moe_options* opts) {
  unif::g_err[0] = 0;
  if (!out) { set_error("out is NULL"); return UNIF_MOE_ERR_ARG; }
  *out = nullptr;
  unif_moe_options o;
  unif_moe_default_options(&o);
  if (opts) o = *opts;
  if ((o.features & ~(unsigned)UNIF_MOE_FEATURES_ALL) != 0u ||
      (o.gemm_kernels != UNIF_MOE_GEMM_AUTO && o.gemm_kernels != UNIF_MOE_GEMM_STREAMING &&
       o.gemm_kernels != UNIF_MOE_GEMM_GROUPED && o.gemm_kernels != UNIF_MOE_GEMM_EXPERT_TILE)) {
    set_error("bad options: features 0x%x, gemm_kernels %d", o.features, o.gemm_kernels);
    return UNIF_MOE_ERR_ARG;
  }
  if (dtype != UNIF_MOE_F32 && dtype != UNIF_MOE_BF16) { set_error("bad dtype"); return UNIF_MOE_ERR_ARG; }
  if (d_model <= 0 || d_ff <= 0 || n_experts < 1 || n_experts > 64 || n_blocks < 2 ||
      n_blocks > 64 || max_tokens < 1) {
    set_error("bad sizes: d=%d H=%d K=%d B=%d max_tokens=%d (need K in [1,64], B in [2,64])",
              d_model, d_ff, n_experts, n_blocks, max_tokens);
    return UNIF_MOE_ERR_ARG;
  }
  if (d_ff % n_blocks != 0 || d_model % 8 != 0) {
    set_error("need d_ff %% n_blocks == 0 and d_model %% 8 == 0");
    return UNIF_MOE_ERR_SHAPE;
  }
  const int M = d_ff / n_blocks;
  if (dtype == UNIF_MOE_BF16 && (d_model % 64 != 0 || M % 64 != 0)) {
    set_error("bf16 layers need d_model %% 64 == 0 and block width %% 64 == 0 (d=%d, M=%d)",
              d_model, M);
    return UNIF_MOE_ERR_SHAPE;
  }
  unif_moe_thresholds t;
  unif_moe_default_thresholds(&t);
  if (th) t = *th;
  if (t.topk_fixed < 0 || t.topk_fixed > n_experts) {
    set_error("topk_fixed=%d outside [0, K]", t.topk_fixed);
    return UNIF_MOE_ERR_ARG;
  }
  if (!isnan(t.alpha_fixed) && !(t.alpha_fixed >= 0.f && t.alpha_fixed <= 1.f)) {
    set_error("alpha_fixed outside [0, 1]");
    return UNIF_MOE_ERR_ARG;
  }
  if (!isnan(t.tau) && !(t.tau >= 0.f && t.tau <= 0.5f)) {
    set_error("tau outside [0, 1/2]");
    return UNIF_MOE_ERR_ARG;
  }

  unif_moe_layer* L = new (std::nothrow) unif_moe_layer();
  if (!L) { set_error("out of host memory"); return UNIF_MOE_ERR_ARG; }
  L->d = d_model; L->H = d_ff; L->K = n_experts; L->B = n_blocks; L->M = M;
  L->G = (n_experts + 1) * n_blocks;
  L->dtype = dtype; L->max_tokens = max_tokens; L->th = t;
  L->features = o.features;
  L->gemm_streaming = o.gemm_kernels == UNIF_MOE_GEMM_STREAMING;
  L->tau = isnan(t.tau) ? (float)((double)(n_blocks - 1) / ((double)n_blocks * n_blocks)) : t.tau;
  const int kmax = t.topk_fixed > 0 ? t.topk_fixed : n_experts;
  L->cb_max = kmax * n_blocks;  // C_B = b + k (B - b) <= k B for every b >= 0 (Eq. 35)
  // bf16 layers: a forward runs in passes whose fp32 accumulator rows fit in
  // 128 MiB, so that the down projection's reductions stay in the 129 MB L2
  // (measured on GB300 for d = 1024: 62.5 us per 1,000 tokens at 65,536
  // tokens in one pass, 54.7 at 32,768). The GEMM workspace is sized for one
  // pass, the routing records for max_tokens.
  L->pass_tokens = max_tokens;
  if (dtype == UNIF_MOE_BF16) {
    const long long fit = (128ll << 20) / (4ll * d_model) / unif::kTileRows * unif::kTileRows;
    if (fit >= unif::kTileRows && fit < max_tokens) L->pass_tokens = (int)fit;
  }
  const int64_t rows =
      (int64_t)L->pass_tokens * L->cb_max + (int64_t)L->G * (unif::kTileRows - 1);
  L->max_rows = (rows + unif::kTileRows - 1) / unif::kTileRows * unif::kTileRows;
  if (L->max_rows >= (int64_t)1 << 31) {
    set_error("max_tokens=%d needs %lld group rows per pass, above the int32 row index",
              max_tokens, (long long)L->max_rows);
    delete L;
    return UNIF_MOE_ERR_CAPACITY;
  }
  L->max_tiles = L->max_rows / unif::kTileRows;
  L->max_chunks = unif::forward_chunks(max_tokens);
  L->router_cols = 1 + n_experts + n_blocks;
  L->router_cols_pad = (L->router_cols + 31) / 32 * 32;
  if (cudaGetDevice(&L->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&L->n_sm, cudaDevAttrMultiProcessorCount, L->device) != cudaSuccess) {
    set_error("no CUDA device");
    delete L;
    return UNIF_MOE_ERR_CUDA;
  }
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, L->device);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, L->device);
  if (major != 10 || minor != 3) {
    set_error("this library is built for sm_103a (GB300); device is sm_%d%d", major, minor);
    delete L;
    return UNIF_MOE_ERR_CUDA;
  }
  const size_t es = elt_size(L);
  const size_t T = (size_t)max_tokens, K = (size_t)n_experts, E = K + 1;
  unif::Workspace& w = L->ws;
  int rc = UNIF_MOE_OK;
#define ALLOC(ptr, n)                          \
  if (rc == UNIF_MOE_OK) rc = dalloc(&(ptr), (n));
  ALLOC(L->wr, (size_t)L->router_cols_pad * d_model);
  if (dtype == UNIF_MOE_BF16) ALLOC(L->wr_bf, (size_t)L->router_cols_pad * d_model);
  ALLOC(L->bias, E);
  void* wup = nullptr;
  void* wdn = nullptr;
  if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&wup), es * E * d_ff * d_model);
  if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&wdn), es * E * d_ff * d_model);
  L->w_up = wup; L->w_down = wdn;
  ALLOC(w.alpha, T); ALLOC(w.b, T); ALLOC(w.k, T); ALLOC(w.shr_mask, T); ALLOC(w.exp_mask, T);
  ALLOC(w.s, T * K);
  ALLOC(w.chunk_cnt, (size_t)L->G * L->max_chunks);
  ALLOC(w.grp_cnt, (size_t)L->G); ALLOC(w.grp_off, (size_t)L->G + 1); ALLOC(w.n_tiles, 1);
  ALLOC(w.tile_group, (size_t)L->max_tiles); ALLOC(w.tile_row0, (size_t)L->max_tiles);
  ALLOC(w.tile_rows, (size_t)L->max_tiles);
  // bf16 layers group inside the router: each group owns a region of
  // max_tokens rows (rounded up to whole tiles) in the row arrays
  L->fused_group = dtype == UNIF_MOE_BF16 && L->router_cols_pad <= 160 &&
                   unif::router_can_group(L->router_cols_pad, L->K, L->G);
  L->region_rows = (L->pass_tokens + 127) / 128 * 128;
  // rows grouped by expert for the expert-tile FFN (where it applies; the
  // backward pass reads the (expert, block) groups and h of a forward)
  L->ffn_fused = L->fused_group &&
                 (o.gemm_kernels == UNIF_MOE_GEMM_EXPERT_TILE ||
                  o.gemm_kernels == UNIF_MOE_GEMM_AUTO) &&
                 !(o.features & UNIF_MOE_FEATURE_BACKWARD) && unif::ffn_fused_fits(d_model, d_ff, M);
  const size_t row_cap = L->fused_group ? (size_t)L->G * L->region_rows : (size_t)L->max_rows;
  ALLOC(w.row_tok, row_cap); ALLOC(w.row_w, row_cap);
  if (L->fused_group) ALLOC(w.grp_fill, (size_t)L->G);
  void* hb = nullptr;
  if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&hb), es * (size_t)L->max_rows * M);
  w.hbuf = hb;
  ALLOC(w.y32, (size_t)L->pass_tokens * d_model);
  if (L->ffn_fused) ALLOC(w.y32_b, (size_t)L->pass_tokens * d_model);
  if (L->ffn_fused) {  // the expert weights as the expert-tile FFN's operand slabs
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.wk_slabs), es * E * d_ff * d_model);
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.wv_slabs), es * E * d_ff * d_model);
  }
  ALLOC(w.status, 1);
  // optional features: every buffer a later call needs, so that no later
  // call allocates
  if (o.features & UNIF_MOE_FEATURE_NORM_FIRST) {
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.xn), es * T * d_model);
  }
  if (o.features & UNIF_MOE_FEATURE_HOST_IO) {
    for (int i = 0; i < 2; ++i) {
      if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.x_stage[i]), es * T * d_model);
      if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.out_stage[i]), es * T * d_model);
      ALLOC(w.mask_stage[i], T); ALLOC(w.b_stage[i], T); ALLOC(w.k_stage[i], T);
    }
    // the pipelined forward's copy streams and slot events
    bool ok = rc == UNIF_MOE_OK &&
              cudaStreamCreateWithFlags(&L->copy_in, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&L->copy_out, cudaStreamNonBlocking) == cudaSuccess;
    for (int i = 0; i < 2 && ok; ++i)
      ok = cudaEventCreateWithFlags(&L->ev_in[i], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&L->ev_comp[i], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&L->ev_out[i], cudaEventDisableTiming) == cudaSuccess;
    if (rc == UNIF_MOE_OK && !ok) {
      set_error("creating the host-buffer copy streams or events failed");
      rc = UNIF_MOE_ERR_CUDA;
    }
  }
  if (o.features & UNIF_MOE_FEATURE_BACKWARD) {
    if (rc == UNIF_MOE_OK && (dtype != UNIF_MOE_BF16 || !L->fused_group || d_model % 128 != 0)) {
      set_error("the backward pass needs a bf16 layer with d %% 128 == 0 (d=%d)", d_model);
      rc = UNIF_MOE_ERR_SHAPE;
    }
    const size_t wbytes = es * E * d_ff * d_model;
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.w_upT), wbytes);
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.w_downT), wbytes);
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.da), es * (size_t)L->max_rows * M);
    if (rc == UNIF_MOE_OK) rc = dalloc(reinterpret_cast<char**>(&w.hw), es * (size_t)L->max_rows * M);
    ALLOC(w.dwt, T * E); ALLOC(w.dz, T * E);
    ALLOC(w.wrT, E * d_model); ALLOC(w.gram, E * E);
  }
  if (o.features & UNIF_MOE_FEATURE_DIAGNOSTICS) {
    const size_t H32 = ((size_t)d_ff + 31) / 32;
    ALLOC(w.diag_sets, K * K * H32); ALLOC(w.diag_counts, K * K);
    ALLOC(w.diag_pair, 2 * T); ALLOC(w.diag_wts, 2 * T); ALLOC(w.diag_q, T * K);
    ALLOC(w.diag_E, T * K * d_model); ALLOC(w.diag_ES, T * K * d_model);
  }
#undef ALLOC
  if (rc == UNIF_MOE_OK && (cudaMemset(w.status, 0, sizeof(int)) != cudaSuccess ||
                            cudaMemset(w.y32, 0, sizeof(float) * L->pass_tokens * d_model) !=
                                cudaSuccess ||
                            (w.y32_b && cudaMemset(w.y32_b, 0, sizeof(float) * L->pass_tokens *
                                                                   d_model) != cudaSuccess) ||
                            (L->fused_group &&
                             (cudaMemset(w.grp_fill, 0, sizeof(int32_t) * L->G) != cudaSuccess ||
                              // rows hold token indices from the start, also any row a
                              // forward that gave up a wait left unwritten
                              cudaMemset(w.row_tok, 0, sizeof(int32_t) * row_cap) != cudaSuccess)))) {
    set_error("cudaMemset failed");
    rc = UNIF_MOE_ERR_CUDA;
  }
  if (rc == UNIF_MOE_OK && unif::router_setup(L) != cudaSuccess) {
    set_error("router kernel attribute setup failed");
    rc = UNIF_MOE_ERR_CUDA;
  }
  if (rc == UNIF_MOE_OK && dtype == UNIF_MOE_BF16) rc = unif::gemm_tc_setup(L);
  if (rc == UNIF_MOE_OK && L->ffn_fused) {
    rc = unif::gemm_fused_setup(L);
    // AUTO falls back to the grouped kernels (their workspace is allocated
    // either way) when the expert-tile kernel cannot be set up here; an
    // explicit EXPERT_TILE request fails instead
    if (rc != UNIF_MOE_OK && o.gemm_kernels == UNIF_MOE_GEMM_AUTO) {
      L->ffn_fused = false;
      L->tile_list = L->fused_group && !(L->up_ws && L->down_ws);
      cudaGetLastError();  // a failed attribute call must not surface at a later launch
      rc = UNIF_MOE_OK;
    }
  }
  if (rc == UNIF_MOE_OK && dtype == UNIF_MOE_BF16) rc = unif::router_tc_setup(L);
  if (rc == UNIF_MOE_OK && (o.features & UNIF_MOE_FEATURE_BACKWARD)) rc = unif::backward_setup(L);
  if (rc != UNIF_MOE_OK) {
    free_all(L);
    delete L;
    return rc;
  }
  *out = L;
  return UNIF_MOE_OK;
}

int unif_moe_load_weights(unif_moe_t L, const void* w_router, const void* w_up,
                          const void* w_down, const float* router_bias, void* stream) {
  unif::g_err[0] = 0;
  if (!L || !w_router || !w_up || !w_down) { set_error("NULL handle or weight"); return UNIF_MOE_ERR_ARG; }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t bytes = elt_size(L) * (size_t)(L->K + 1) * L->H * L->d;
  CK(cudaMemcpyAsync(L->w_up, w_up, bytes, cudaMemcpyDeviceToDevice, s));
  CK(cudaMemcpyAsync(L->w_down, w_down, bytes, cudaMemcpyDeviceToDevice, s));
  CK(unif::launch_prototypes(L, w_router, router_bias, s));
  if (L->features & UNIF_MOE_FEATURE_BACKWARD) CK(unif::launch_transpose_weights(L, s));
  if (L->ffn_fused) CK(unif::launch_repack_slabs(L, s));
  L->loaded = true;
  return UNIF_MOE_OK;
}

// The residual epilogue of a Transformer sublayer: out = res + y, then LN
// when `norm` (the layer's combine otherwise).
struct SublayerEpilogue {
  const void* res;
  const void* gamma;
  const void* beta;
  float eps;
  bool norm;
};

static int forward_checks(unif_moe_t L, const void* x, void* out, int T,
                          int32_t* shared_counts, int32_t* residual_counts) {
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (T < 0) { set_error("T < 0"); return UNIF_MOE_ERR_ARG; }
  if (T > L->max_tokens) {
    set_error("T=%d exceeds max_tokens=%d", T, L->max_tokens);
    return UNIF_MOE_ERR_CAPACITY;
  }
  if (!L->loaded) { set_error("forward before load_weights"); return UNIF_MOE_ERR_STATE; }
  if (T == 0) return UNIF_MOE_OK;
  if (!x || !out) { set_error("x or out is NULL"); return UNIF_MOE_ERR_ARG; }
  if (!aligned16(x) || !aligned16(out)) {
    set_error("x and out must be 16-byte aligned");
    return UNIF_MOE_ERR_ARG;
  }
  if ((shared_counts && !aligned16(shared_counts)) || (residual_counts && !aligned16(residual_counts))) {
    set_error("count buffers must be 16-byte aligned");
    return UNIF_MOE_ERR_ARG;
  }
  return UNIF_MOE_OK;
}

// One pass of the forward over tokens [t0, t0 + T) of the caller's arrays
// (x, out, mask, counts and, for a sublayer, the residual input already
// offset to t0); `sub` replaces the combine with a sublayer's residual
// epilogue. `timed`: record the stage events around this pass.
static int forward_pass(unif_moe_t L, const void* x, void* out, int T, int t0,
                        const uint8_t* token_mask, int32_t* shared_counts,
                        int32_t* residual_counts, cudaStream_t s, const SublayerEpilogue* sub,
                        bool timed) {
  cudaEvent_t* ev = L->stage_ev;
  cudaEvent_t none[6] = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
  if (!timed) ev = none;
  // The output accumulator and the grouping counters are all zero between
  // passes (each combine zeroes them). A pass that returned before
  // launching its combine leaves them dirty: clear them first.
  if (L->y_dirty) {
    CK(cudaMemsetAsync(L->ws.y32, 0, sizeof(float) * (size_t)L->pass_tokens * L->d, s));
    if (L->ws.y32_b)
      CK(cudaMemsetAsync(L->ws.y32_b, 0, sizeof(float) * (size_t)L->pass_tokens * L->d, s));
    if (L->fused_group) CK(cudaMemsetAsync(L->ws.grp_fill, 0, sizeof(int32_t) * L->G, s));
  }
  L->y_dirty = true;
  L->rec0 = t0;
  if (ev[0]) CK(cudaEventRecord(ev[0], s));
  if (L->dtype == UNIF_MOE_BF16) {
    CK(unif::launch_router_tc(L, x, token_mask, T, shared_counts, residual_counts, s));
  } else {
    CK(unif::launch_router(L, x, token_mask, T, shared_counts, residual_counts, s));
  }
  if (ev[1]) CK(cudaEventRecord(ev[1], s));
  if (!L->fused_group) CK(unif::launch_permute(L, T, s));
  else if (L->tile_list) CK(unif::launch_tile_list(L, s));
  if (ev[2]) CK(cudaEventRecord(ev[2], s));
  if (L->dtype == UNIF_MOE_BF16) {
    CK(unif::launch_gemms_tc(L, x, T, ev[3], s));
  } else {
    CK(unif::launch_gemms_simt(L, x, T, ev[3], s));
  }
  if (ev[4]) CK(cudaEventRecord(ev[4], s));
  if (sub)
    CK(unif::launch_combine_residual(L, sub->res, out, token_mask, sub->gamma, sub->beta,
                                     sub->eps, sub->norm, T, s));
  else
    CK(unif::launch_combine(L, out, T, s));
  L->y_dirty = false;
  // the expert-tile FFN zeroed the other accumulator for the next pass
  if (L->ffn_fused) L->acc_sel ^= 1;
  if (ev[5]) CK(cudaEventRecord(ev[5], s));
  return UNIF_MOE_OK;
}

// The forward after the argument checks (T > 0), in passes of at most
// pass_tokens tokens; the stage events time the last pass.
static int forward_core(unif_moe_t L, const void* x, void* out, int T, const uint8_t* token_mask,
                        int32_t* shared_counts, int32_t* residual_counts, cudaStream_t s,
                        const SublayerEpilogue* sub) {
  const size_t row = elt_size(L) * (size_t)L->d;  // bytes per token row of x and out
  const int P = L->pass_tokens;
  for (int t0 = 0; t0 < T; t0 += P) {
    const int n = T - t0 < P ? T - t0 : P;
    const size_t off = (size_t)t0 * row;
    SublayerEpilogue sp;
    if (sub) {
      sp = *sub;
      sp.res = static_cast<const char*>(sub->res) + off;
    }
    const int rc = forward_pass(
        L, static_cast<const char*>(x) + off, static_cast<char*>(out) + off, n, t0,
        token_mask ? token_mask + t0 : nullptr, shared_counts ? shared_counts + t0 : nullptr,
        residual_counts ? residual_counts + t0 : nullptr, s, sub ? &sp : nullptr, t0 + n >= T);
    L->rec0 = 0;
    if (rc != UNIF_MOE_OK) return rc;
  }
  L->last_T = T;
  L->last_pass_T = T - (T - 1) / P * P;
  return UNIF_MOE_OK;
}

int unif_moe_load_upcycled(unif_moe_t L, const void* w_router, const void* w_up_dense,
                           const void* w_down_dense, const float* router_bias, void* stream) {
  unif::g_err[0] = 0;
  if (!L || !w_router || !w_up_dense || !w_down_dense) {
    set_error("NULL handle or weight");
    return UNIF_MOE_ERR_ARG;
  }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // every expert, the shared one and the K residual ones, starts as the
  // dense FFN: K + 1 copies of each projection
  const size_t bytes = elt_size(L) * (size_t)L->H * L->d;
  for (int e = 0; e <= L->K; ++e) {
    CK(cudaMemcpyAsync(static_cast<char*>(L->w_up) + e * bytes, w_up_dense, bytes,
                       cudaMemcpyDeviceToDevice, s));
    CK(cudaMemcpyAsync(static_cast<char*>(L->w_down) + e * bytes, w_down_dense, bytes,
                       cudaMemcpyDeviceToDevice, s));
  }
  CK(unif::launch_prototypes(L, w_router, router_bias, s));
  if (L->features & UNIF_MOE_FEATURE_BACKWARD) CK(unif::launch_transpose_weights(L, s));
  if (L->ffn_fused) CK(unif::launch_repack_slabs(L, s));
  L->loaded = true;
  return UNIF_MOE_OK;
}

int unif_moe_backward(unif_moe_t L, const void* x, const void* dy, int T, const uint8_t* mask,
                      float* dx, float* dw_up, float* dw_down, float* dw_router, float* dbias,
                      float lambda_div, float* l_div, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (!(L->features & UNIF_MOE_FEATURE_BACKWARD)) {
    set_error("backward on a handle created without UNIF_MOE_FEATURE_BACKWARD");
    return UNIF_MOE_ERR_STATE;
  }
  if (L->last_T < 0 || T != L->last_T) {
    set_error("backward needs the forward of the same T before it (T=%d, last forward %d)", T,
              L->last_T);
    return UNIF_MOE_ERR_STATE;
  }
  if (T > L->pass_tokens) {
    set_error("backward of %d tokens: the forward ran in passes of %d", T, L->pass_tokens);
    return UNIF_MOE_ERR_CAPACITY;
  }
  if (!x || !dy || !dx || !dw_up || !dw_down || !dw_router) {
    set_error("NULL input or output");
    return UNIF_MOE_ERR_ARG;
  }
  if (!aligned16(x) || !aligned16(dy) || !aligned16(dx) || !aligned16(dw_up) ||
      !aligned16(dw_down) || !aligned16(dw_router)) {
    set_error("backward buffers must be 16-byte aligned");
    return UNIF_MOE_ERR_ARG;
  }
  if (T == 0) return UNIF_MOE_OK;
  DeviceGuard dg(L->device);
  return unif::backward_run(L, x, dy, T, mask, dx, dw_up, dw_down, dw_router, dbias, lambda_div,
                            l_div, static_cast<cudaStream_t>(stream));
}

int unif_moe_value_alignment(unif_moe_t L, float delta, float* rho, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (!(L->features & UNIF_MOE_FEATURE_DIAGNOSTICS)) {
    set_error("diagnostics on a handle created without UNIF_MOE_FEATURE_DIAGNOSTICS");
    return UNIF_MOE_ERR_STATE;
  }
  if (!L->loaded) { set_error("no weights loaded"); return UNIF_MOE_ERR_STATE; }
  if (!rho || !isfinite(delta)) { set_error("rho is NULL or delta not finite"); return UNIF_MOE_ERR_ARG; }
  DeviceGuard dg(L->device);
  if (unif::diag_alignment(L, delta, rho, static_cast<cudaStream_t>(stream)) != 0) {
    set_error("value alignment launch failed");
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

int unif_moe_functional_demand(unif_moe_t L, const void* x, int T, const void* w_res,
                               float delta, float eps, int32_t* k_eps, float* err,
                               int32_t* pair, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (!(L->features & UNIF_MOE_FEATURE_DIAGNOSTICS)) {
    set_error("diagnostics on a handle created without UNIF_MOE_FEATURE_DIAGNOSTICS");
    return UNIF_MOE_ERR_STATE;
  }
  if (!L->loaded) { set_error("no weights loaded"); return UNIF_MOE_ERR_STATE; }
  if (L->K < 2 || L->K > 32) {
    set_error("functional demand needs 2 <= K <= 32 (K=%d)", L->K);
    return UNIF_MOE_ERR_SHAPE;
  }
  if (T < 0 || T > L->max_tokens) {
    set_error("T=%d outside [0, max_tokens=%d]", T, L->max_tokens);
    return T < 0 ? UNIF_MOE_ERR_ARG : UNIF_MOE_ERR_CAPACITY;
  }
  if (T == 0) return UNIF_MOE_OK;
  if (!x || !w_res || !k_eps || !isfinite(delta) || !isfinite(eps)) {
    set_error("NULL x, w_res or k_eps, or delta / eps not finite");
    return UNIF_MOE_ERR_ARG;
  }
  DeviceGuard dg(L->device);
  if (unif::diag_demand(L, x, T, w_res, delta, eps, k_eps, err, pair,
                        static_cast<cudaStream_t>(stream)) != 0) {
    set_error("functional demand launch failed");
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

int unif_moe_forward(unif_moe_t L, const void* x, void* out, int T, const uint8_t* token_mask,
                     int32_t* shared_counts, int32_t* residual_counts, void* stream) {
  unif::g_err[0] = 0;
  const int rc = forward_checks(L, x, out, T, shared_counts, residual_counts);
  if (rc != UNIF_MOE_OK || T == 0) return rc;
  DeviceGuard dg(L->device);
  return forward_core(L, x, out, T, token_mask, shared_counts, residual_counts,
                      static_cast<cudaStream_t>(stream), nullptr);
}

int unif_moe_sublayer_forward(unif_moe_t L, const void* x, void* out, int T,
                              const uint8_t* token_mask, int32_t* shared_counts,
                              int32_t* residual_counts, const void* ln_gamma,
                              const void* ln_beta, float eps, int norm_first, void* stream) {
  unif::g_err[0] = 0;
  const int rc = forward_checks(L, x, out, T, shared_counts, residual_counts);
  if (rc != UNIF_MOE_OK) return rc;
  if (!ln_gamma || !ln_beta) { set_error("ln_gamma or ln_beta is NULL"); return UNIF_MOE_ERR_ARG; }
  if (!(eps >= 0.f) || !isfinite(eps)) { set_error("eps must be finite and >= 0"); return UNIF_MOE_ERR_ARG; }
  if (!aligned16(ln_gamma) || !aligned16(ln_beta)) {
    set_error("ln_gamma and ln_beta must be 16-byte aligned");
    return UNIF_MOE_ERR_ARG;
  }
  if (L->d > 1024 || L->d % 8 != 0) {
    set_error("the sublayer needs d <= 1024, a multiple of 8 (d=%d)", L->d);
    return UNIF_MOE_ERR_SHAPE;
  }
  if (T == 0) return UNIF_MOE_OK;
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const SublayerEpilogue sub{x, ln_gamma, ln_beta, eps, !norm_first};
  if (!norm_first)  // out = LN(x + F(x))
    return forward_core(L, x, out, T, token_mask, shared_counts, residual_counts, s, &sub);
  // out = x + F(LN(x)); LN(x) in the layer dtype, in the buffer made at create
  if (!L->ws.xn) {
    set_error("norm-first sublayer on a handle created without UNIF_MOE_FEATURE_NORM_FIRST");
    return UNIF_MOE_ERR_STATE;
  }
  CK(unif::launch_layernorm(L, x, L->ws.xn, token_mask, ln_gamma, ln_beta, eps, T, s));
  return forward_core(L, L->ws.xn, out, T, token_mask, shared_counts, residual_counts, s, &sub);
}

// The device address of pinned, mapped host memory (nullptr for any other
// pointer, including NULL): the kernels can store into it directly.
static void* mapped_host(void* p) {
  if (!p) return nullptr;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();  // an unregistered pointer is not an error here
    return nullptr;
  }
  if (at.type != cudaMemoryTypeHost || !at.devicePointer) return nullptr;
  if ((reinterpret_cast<uintptr_t>(at.devicePointer) & 15u) != 0) return nullptr;
  return at.devicePointer;
}

int unif_moe_forward_host(unif_moe_t L, const void* x_host, void* out_host, int T,
                          const uint8_t* mask_host, int32_t* b_host, int32_t* k_host,
                          void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (T < 0 || T > L->max_tokens) {
    set_error("T=%d outside [0, max_tokens=%d]", T, L->max_tokens);
    return T < 0 ? UNIF_MOE_ERR_ARG : UNIF_MOE_ERR_CAPACITY;
  }
  if (!L->loaded) { set_error("forward before load_weights"); return UNIF_MOE_ERR_STATE; }
  if (!(L->features & UNIF_MOE_FEATURE_HOST_IO)) {
    set_error("host-buffer forward on a handle created without UNIF_MOE_FEATURE_HOST_IO");
    return UNIF_MOE_ERR_STATE;
  }
  if (T == 0) return UNIF_MOE_OK;
  if (!x_host || !out_host) { set_error("x or out is NULL"); return UNIF_MOE_ERR_ARG; }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unif::Workspace& w = L->ws;
  const size_t es = elt_size(L);
  const size_t xb = es * (size_t)T * L->d;
  // slot 0 may still be in use by pipelined forwards
  CK(cudaStreamSynchronize(L->copy_in));
  CK(cudaStreamSynchronize(L->copy_out));
  CK(cudaMemcpyAsync(w.x_stage[0], x_host, xb, cudaMemcpyHostToDevice, s));
  if (mask_host) CK(cudaMemcpyAsync(w.mask_stage[0], mask_host, (size_t)T, cudaMemcpyHostToDevice, s));
  // Outputs in pinned host memory that the device can address are written
  // there by the kernels themselves (the combine, the router), without a
  // staging buffer and a copy back.
  void* out_dev = mapped_host(out_host);
  int32_t* b_dev = static_cast<int32_t*>(mapped_host(b_host));
  int32_t* k_dev = static_cast<int32_t*>(mapped_host(k_host));
  int rc = unif_moe_forward(L, w.x_stage[0], out_dev ? out_dev : w.out_stage[0], T,
                            mask_host ? w.mask_stage[0] : nullptr,
                            b_host ? (b_dev ? b_dev : w.b_stage[0]) : nullptr,
                            k_host ? (k_dev ? k_dev : w.k_stage[0]) : nullptr, stream);
  if (rc != UNIF_MOE_OK) return rc;
  if (!out_dev) CK(cudaMemcpyAsync(out_host, w.out_stage[0], xb, cudaMemcpyDeviceToHost, s));
  if (b_host && !b_dev)
    CK(cudaMemcpyAsync(b_host, w.b_stage[0], sizeof(int32_t) * T, cudaMemcpyDeviceToHost, s));
  if (k_host && !k_dev)
    CK(cudaMemcpyAsync(k_host, w.k_stage[0], sizeof(int32_t) * T, cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  return UNIF_MOE_OK;
}

int unif_moe_forward_host_async(unif_moe_t L, const void* x_host, void* out_host, int T,
                                const uint8_t* mask_host, int32_t* b_host, int32_t* k_host,
                                void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (T < 0 || T > L->max_tokens) {
    set_error("T=%d outside [0, max_tokens=%d]", T, L->max_tokens);
    return T < 0 ? UNIF_MOE_ERR_ARG : UNIF_MOE_ERR_CAPACITY;
  }
  if (!L->loaded) { set_error("forward before load_weights"); return UNIF_MOE_ERR_STATE; }
  if (!(L->features & UNIF_MOE_FEATURE_HOST_IO)) {
    set_error("host-buffer forward on a handle created without UNIF_MOE_FEATURE_HOST_IO");
    return UNIF_MOE_ERR_STATE;
  }
  if (T == 0) return UNIF_MOE_OK;
  if (!x_host || !out_host) { set_error("x or out is NULL"); return UNIF_MOE_ERR_ARG; }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unif::Workspace& w = L->ws;
  const int i = L->host_slot;
  const size_t xb = elt_size(L) * (size_t)T * L->d;
  // input, on the copy-in stream: once the kernels that read this slot two
  // calls ago are done, so that it overlaps the previous call's kernels
  CK(cudaStreamWaitEvent(L->copy_in, L->ev_comp[i], 0));
  CK(cudaMemcpyAsync(w.x_stage[i], x_host, xb, cudaMemcpyHostToDevice, L->copy_in));
  if (mask_host)
    CK(cudaMemcpyAsync(w.mask_stage[i], mask_host, (size_t)T, cudaMemcpyHostToDevice, L->copy_in));
  CK(cudaEventRecord(L->ev_in[i], L->copy_in));
  // kernels, on the caller's stream: after this slot's input has landed and
  // its previous output (and counts) have been copied out
  CK(cudaStreamWaitEvent(s, L->ev_in[i], 0));
  CK(cudaStreamWaitEvent(s, L->ev_out[i], 0));
  const int rc = unif_moe_forward(L, w.x_stage[i], w.out_stage[i], T,
                                  mask_host ? w.mask_stage[i] : nullptr,
                                  b_host ? w.b_stage[i] : nullptr, k_host ? w.k_stage[i] : nullptr,
                                  stream);
  if (rc != UNIF_MOE_OK) return rc;
  CK(cudaEventRecord(L->ev_comp[i], s));
  // output, on the copy-out stream, overlapping the next call's kernels
  CK(cudaStreamWaitEvent(L->copy_out, L->ev_comp[i], 0));
  CK(cudaMemcpyAsync(out_host, w.out_stage[i], xb, cudaMemcpyDeviceToHost, L->copy_out));
  if (b_host)
    CK(cudaMemcpyAsync(b_host, w.b_stage[i], sizeof(int32_t) * T, cudaMemcpyDeviceToHost,
                       L->copy_out));
  if (k_host)
    CK(cudaMemcpyAsync(k_host, w.k_stage[i], sizeof(int32_t) * T, cudaMemcpyDeviceToHost,
                       L->copy_out));
  CK(cudaEventRecord(L->ev_out[i], L->copy_out));
  L->host_slot = i ^ 1;
  return UNIF_MOE_OK;
}

int unif_moe_forward_host_wait(unif_moe_t L) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (!(L->features & UNIF_MOE_FEATURE_HOST_IO)) {
    set_error("host-buffer forward on a handle created without UNIF_MOE_FEATURE_HOST_IO");
    return UNIF_MOE_ERR_STATE;
  }
  DeviceGuard dg(L->device);
  CK(cudaStreamSynchronize(L->copy_in));
  CK(cudaStreamSynchronize(L->copy_out));
  return UNIF_MOE_OK;
}

int unif_moe_get_routing(unif_moe_t L, float* alpha, uint64_t* shared_mask, uint64_t* expert_mask,
                         int32_t* q, float* p, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (L->last_T < 0) { set_error("no forward has run"); return UNIF_MOE_ERR_STATE; }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t T = (size_t)L->last_T;
  const cudaMemcpyKind dd = cudaMemcpyDeviceToDevice;
  if (T > 0) {
    if (alpha) CK(cudaMemcpyAsync(alpha, L->ws.alpha, sizeof(float) * T, dd, s));
    if (shared_mask) CK(cudaMemcpyAsync(shared_mask, L->ws.shr_mask, sizeof(uint64_t) * T, dd, s));
    if (expert_mask) CK(cudaMemcpyAsync(expert_mask, L->ws.exp_mask, sizeof(uint64_t) * T, dd, s));
    if (q || p) CK(unif::launch_sort_affinities(L, (int)T, q, p, s));
  }
  CK(cudaStreamSynchronize(s));
  return UNIF_MOE_OK;
}

int unif_moe_get_groups(unif_moe_t L, int32_t* counts, int32_t* offsets, int32_t* row_token,
                        float* row_weight, int64_t* n_rows, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  if (L->last_T < 0) { set_error("no forward has run"); return UNIF_MOE_ERR_STATE; }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const cudaMemcpyKind dh = cudaMemcpyDeviceToHost;
  int32_t total = 0;
  if (L->last_T > 0 && !L->fused_group)
    CK(cudaMemcpyAsync(&total, L->ws.grp_off + L->G, sizeof(int32_t), dh, s));
  CK(cudaStreamSynchronize(s));
  if (L->last_T > 0 && L->ffn_fused) {
    // the device grouped the rows by expert; the (expert, block) table of
    // the forward's last pass follows from its routing records: token t
    // runs blocks shr(t) of the shared expert (weight alpha) and the
    // complementary blocks of each selected residual expert j (weight s_j)
    const int tok_base = L->last_T - L->last_pass_T;
    const size_t n = (size_t)L->last_pass_T, K = (size_t)L->K;
    std::vector<float> al(n), sv(n * K);
    std::vector<uint64_t> sh(n), em(n);
    CK(cudaMemcpyAsync(al.data(), L->ws.alpha + tok_base, sizeof(float) * n, dh, s));
    CK(cudaMemcpyAsync(sh.data(), L->ws.shr_mask + tok_base, sizeof(uint64_t) * n, dh, s));
    CK(cudaMemcpyAsync(em.data(), L->ws.exp_mask + tok_base, sizeof(uint64_t) * n, dh, s));
    CK(cudaMemcpyAsync(sv.data(), L->ws.s + (size_t)tok_base * K, sizeof(float) * n * K, dh, s));
    CK(cudaStreamSynchronize(s));
    const int B = L->B;
    const uint64_t full = B >= 64 ? ~0ull : ((1ull << B) - 1ull);
    std::vector<int32_t> cnt(L->G, 0), off(L->G + 1), pos(L->G);
    for (int pass = 0; pass < 2; ++pass) {
      if (pass == 1) {
        off[0] = 0;
        for (int g = 0; g < L->G; ++g) off[g + 1] = off[g] + (cnt[g] + 127) / 128 * 128;
        for (int g = 0; g < L->G; ++g) pos[g] = off[g];
      }
      for (size_t t = 0; t < n; ++t) {
        for (int e = 0; e <= L->K; ++e) {
          uint64_t bl = e == 0 ? sh[t] : (((em[t] >> (e - 1)) & 1ull) ? (~sh[t] & full) : 0ull);
          const float w = e == 0 ? al[t] : sv[t * K + e - 1];
          for (; bl != 0ull; bl &= bl - 1ull) {
            const int g = e * B + (__builtin_ffsll((long long)bl) - 1);
            if (pass == 0) { ++cnt[g]; continue; }
            if (row_token) row_token[pos[g]] = tok_base + (int32_t)t;
            if (row_weight) row_weight[pos[g]] = w;
            ++pos[g];
          }
        }
      }
    }
    total = off[L->G];
    for (int g = 0; g < L->G; ++g)
      for (int r = pos[g]; r < off[g + 1]; ++r) {
        if (row_token) row_token[r] = -1;
        if (row_weight) row_weight[r] = 0.f;
      }
    if (counts) memcpy(counts, cnt.data(), sizeof(int32_t) * L->G);
    if (offsets) memcpy(offsets, off.data(), sizeof(int32_t) * (L->G + 1));
  } else if (L->last_T > 0 && L->fused_group) {
    // rows live in per-group regions on the device, each group's rows in the
    // order the router CTAs reserved them: gather them group by group into
    // the contiguous padded layout, in token order
    // (the combine copied the group sizes to grp_cnt; offsets pad each group
    // to whole 128-row tiles)
    std::vector<int32_t> cnt(L->G), off(L->G + 1);
    // the table is that of the forward's last pass; its rows hold tokens
    // relative to the pass's first token
    const int tok_base = L->last_T - L->last_pass_T;
    CK(cudaMemcpyAsync(cnt.data(), L->ws.grp_cnt, sizeof(int32_t) * L->G, dh, s));
    CK(cudaStreamSynchronize(s));
    off[0] = 0;
    for (int g = 0; g < L->G; ++g) off[g + 1] = off[g] + (cnt[g] + 127) / 128 * 128;
    total = off[L->G];
    if (counts) memcpy(counts, cnt.data(), sizeof(int32_t) * L->G);
    if (offsets) memcpy(offsets, off.data(), sizeof(int32_t) * (L->G + 1));
    for (int g = 0; g < L->G; ++g) {
      const size_t n = (size_t)cnt[g];
      const size_t src = (size_t)g * L->region_rows;
      // padding rows (the device leaves them untouched): token -1, weight 0
      for (int r = off[g] + cnt[g]; r < off[g + 1]; ++r) {
        if (row_token) row_token[r] = -1;
        if (row_weight) row_weight[r] = 0.f;
      }
      if (n == 0 || (!row_token && !row_weight)) continue;
      std::vector<int32_t> tok(n);
      std::vector<float> wt(n);
      std::vector<size_t> ord(n);
      CK(cudaMemcpyAsync(tok.data(), L->ws.row_tok + src, sizeof(int32_t) * n, dh, s));
      CK(cudaMemcpyAsync(wt.data(), L->ws.row_w + src, sizeof(float) * n, dh, s));
      CK(cudaStreamSynchronize(s));
      for (size_t i = 0; i < n; ++i) ord[i] = i;
      std::sort(ord.begin(), ord.end(), [&](size_t a, size_t b) { return tok[a] < tok[b]; });
      for (size_t i = 0; i < n; ++i) {
        if (row_token) row_token[off[g] + i] = tok_base + tok[ord[i]];
        if (row_weight) row_weight[off[g] + i] = wt[ord[i]];
      }
    }
  } else if (L->last_T > 0) {
    if (counts) CK(cudaMemcpyAsync(counts, L->ws.grp_cnt, sizeof(int32_t) * L->G, dh, s));
    if (offsets) CK(cudaMemcpyAsync(offsets, L->ws.grp_off, sizeof(int32_t) * (L->G + 1), dh, s));
    if (row_token && total > 0) CK(cudaMemcpyAsync(row_token, L->ws.row_tok, sizeof(int32_t) * total, dh, s));
    if (row_weight && total > 0) CK(cudaMemcpyAsync(row_weight, L->ws.row_w, sizeof(float) * total, dh, s));
  } else {
    if (counts) memset(counts, 0, sizeof(int32_t) * L->G);
    if (offsets) memset(offsets, 0, sizeof(int32_t) * (L->G + 1));
  }
  if (n_rows) *n_rows = total;
  CK(cudaStreamSynchronize(s));
  return UNIF_MOE_OK;
}

int64_t unif_moe_max_rows(unif_moe_t L) { return L ? L->max_rows : -1; }

int unif_moe_pass_tokens(unif_moe_t L) { return L ? L->pass_tokens : -1; }

int unif_moe_kernels_per_forward(unif_moe_t L) {
  if (!L) return -1;
  if (L->ffn_fused) return 3;  // router, expert-tile FFN, combine
  return L->fused_group ? (L->tile_list ? 5 : 4) : 6;
}

int unif_moe_set_stage_events(unif_moe_t L, void* const* events) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  for (int i = 0; i < 6; ++i) {
    L->stage_ev[i] = events ? static_cast<cudaEvent_t>(events[i]) : nullptr;
    if (events && !events[i]) { set_error("event %d is NULL", i); return UNIF_MOE_ERR_ARG; }
  }
  return UNIF_MOE_OK;
}

int unif_moe_sync_status(unif_moe_t L, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  DeviceGuard dg(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int st = 0;
  CK(cudaMemcpyAsync(&st, L->ws.status, sizeof(int), cudaMemcpyDeviceToHost, s));
  CK(cudaMemsetAsync(L->ws.status, 0, sizeof(int), s));
  CK(cudaStreamSynchronize(s));
  if (st & unif::kStatusTimeout) {
    set_error("a kernel gave up a bounded wait (status 0x%x)", st);
    return UNIF_MOE_ERR_TIMEOUT;
  }
  if (st) {
    set_error("kernel status 0x%x", st);
    return UNIF_MOE_ERR_CUDA;
  }
  return UNIF_MOE_OK;
}

int unif_moe_selftest_timeout(unif_moe_t L, int timeout_us, void* stream) {
  unif::g_err[0] = 0;
  if (!L) { set_error("NULL handle"); return UNIF_MOE_ERR_ARG; }
  DeviceGuard dg(L->device);
  CK(unif::launch_timeout_probe(L, timeout_us, static_cast<cudaStream_t>(stream)));
  return UNIF_MOE_OK;
}

void unif_moe_destroy(unif_moe_t L) {
  if (!L) return;
  {
    DeviceGuard dg(L->device);
    cudaDeviceSynchronize();
    free_all(L);
  }
  delete L;
}

}  // extern "C"
