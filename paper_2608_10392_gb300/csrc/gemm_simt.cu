// Grouped expert GEMMs on CUDA cores (FP32 FMA), used for fp32 layers: the
// tcgen05 tf32 kind rounds operands to 10 mantissa bits, which an fp32 layer
// cannot afford, so fp32 layers keep full-precision FMA.
//
// Both kernels walk the same tile list as the tensor-core path:
//   up   : h[row] = GeLU(x[tok(row)] K_e[:, H_b])           (Eq. 16, inner part)
//   down : y[tok(row)] += w(row) * h[row] V_e[H_b, :]       (Eqs. 16, 28-30)
// where (e, b) is the tile's group and w(row) is alpha or p_i.
#include "internal.cuh"

namespace unif {
namespace {

constexpr int kBM = 128, kBN = 64, kBK = 16, kThreads = 256;

__device__ __forceinline__ float ld_f32(const float* p) { return *p; }
__device__ __forceinline__ void st_out(float* p, float v) { *p = v; }

__device__ __forceinline__ float gelu_erf(float v) {
  return 0.5f * v * (1.0f + erff(v * 0.70710678118654752f));
}

struct SimtArgs {
  const int32_t* n_tiles;
  const int32_t* tile_group;
  const int32_t* tile_row0;
  const int32_t* row_tok;
  const float* row_w;
  int d, H, B, M;
  float* y32;
};

// MODE 0: up-projection + GeLU into h. MODE 1: down-projection, weighted,
// accumulated into y32 with atomics.
template <int MODE, typename TA, typename TW, typename TH>
__global__ void __launch_bounds__(kThreads)
simt_gemm_kernel(const TA* __restrict__ A, const TW* __restrict__ W, TH* __restrict__ h,
                 SimtArgs a) {
  __shared__ float As[kBK][kBM + 4];
  __shared__ float Ws[kBK][kBN + 4];
  __shared__ int tok_s[kBM];
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int N = (MODE == 0) ? a.M : a.d;     // output columns of the group
  const int Kdim = (MODE == 0) ? a.d : a.M;  // reduction length
  const int n_chunks = (N + kBN - 1) / kBN;
  const int n_items = a.n_tiles[0] * n_chunks;
  for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
    const int tile = item / n_chunks, nc = item % n_chunks;
    const int g = a.tile_group[tile], row0 = a.tile_row0[tile];
    const int e = g / a.B, blk = g % a.B;
    __syncthreads();
    if (tid < kBM) tok_s[tid] = a.row_tok[row0 + tid];
    __syncthreads();
    float acc[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < Kdim; k0 += kBK) {
      // A tile: 128 rows x 16; row r of the tile is x[tok] (up) or h[row0+r] (down).
      for (int idx = tid; idx < kBM * kBK; idx += kThreads) {
        const int r = idx / kBK, kk = idx % kBK;
        float v = 0.f;
        if (k0 + kk < Kdim) {
          if (MODE == 0) {
            const int t = tok_s[r];
            if (t >= 0) v = ld_f32(A + (size_t)t * a.d + k0 + kk);
          } else {
            v = ld_f32(A + (size_t)(row0 + r) * a.M + k0 + kk);
          }
        }
        As[kk][r] = v;
      }
      // W tile: 64 output columns x 16.
      for (int idx = tid; idx < kBN * kBK; idx += kThreads) {
        const int c = idx / kBK, kk = idx % kBK;
        const int n = nc * kBN + c;
        float v = 0.f;
        if (n < N && k0 + kk < Kdim) {
          if (MODE == 0)  // w_up [(K+1)H][d]
            v = ld_f32(W + ((size_t)e * a.H + blk * a.M + n) * a.d + k0 + kk);
          else            // w_down [(K+1)d][H]
            v = ld_f32(W + ((size_t)e * a.d + n) * a.H + blk * a.M + k0 + kk);
        }
        Ws[kk][c] = v;
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < kBK; ++kk) {
        float av[8], wv[4];
#pragma unroll
        for (int i = 0; i < 8; ++i) av[i] = As[kk][ty * 8 + i];
#pragma unroll
        for (int j = 0; j < 4; ++j) wv[j] = Ws[kk][tx * 4 + j];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], wv[j], acc[i][j]);
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = ty * 8 + i;
      const int row = row0 + r;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int n = nc * kBN + tx * 4 + j;
        if (n >= N) continue;
        if (MODE == 0) {
          st_out(h + (size_t)row * a.M + n, gelu_erf(acc[i][j]));
        } else {
          const int t = tok_s[r];
          if (t >= 0) atomicAdd(a.y32 + (size_t)t * a.d + n, a.row_w[row] * acc[i][j]);
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_gemms_simt(unif_moe_layer* L, const void* x, int T, cudaEvent_t mid,
                              cudaStream_t s) {
  (void)T;
  SimtArgs a;
  a.n_tiles = L->ws.n_tiles; a.tile_group = L->ws.tile_group; a.tile_row0 = L->ws.tile_row0;
  a.row_tok = L->ws.row_tok; a.row_w = L->ws.row_w;
  a.d = L->d; a.H = L->H; a.B = L->B; a.M = L->M; a.y32 = L->ws.y32;
  const int grid = L->n_sm * 4;
  float* h = static_cast<float*>(L->ws.hbuf);
  simt_gemm_kernel<0, float, float, float><<<grid, kThreads, 0, s>>>(
      static_cast<const float*>(x), static_cast<const float*>(L->w_up), h, a);
  if (mid) cudaEventRecord(mid, s);
  simt_gemm_kernel<1, float, float, float><<<grid, kThreads, 0, s>>>(
      h, static_cast<const float*>(L->w_down), nullptr, a);  // (output: the accumulator)
  return cudaGetLastError();
}

}  // namespace unif
