// Diagnostics of Sec. II-B on a layer's K residual experts (experts 1..K of
// the loaded weights; router columns 1..K): an analysis tool, not part of
// the forward. CUDA cores, fp32 except the per-token ridge fits (fp64).
//
//   value alignment (Eq. shared-set): c_ijh = V_i[h,:] . V_j[h,:] /
//       (|V_i[h,:]| |V_j[h,:]|), S_ij(delta) = {h : c_ijh >= delta},
//       rho_ij = |S_ij| / H (a value row of zero norm aligns with nothing);
//   functional demand (Eqs. diagnostic-original .. functional-demand): per
//       token, its top-2 pair (i, j) of s = softmax(x W_g) (ties to the lower
//       index), s~ = s / (s_i + s_j), y_orig = sum s~_e E_e, S_bar = sum s~_e
//       E_e^{S_ij}, r = y_orig - S_bar, the residual order q of x W_r, R_m the
//       rows E_{q_1..q_m}^{R_ij}, a* = (R_m R_m^T + gamma_m I)^{-1} R_m r with
//       gamma_m = 1e-6 tr(R_m R_m^T) / m (a = 0 when R_m = 0), e_m =
//       |a*^T R_m - r| / max(|y_orig|, 1e-12), k_eps = min{m : e_m <= eps}
//       or K + 1.
#include <math.h>
#include <stdio.h>

#include "internal.cuh"

namespace unif {
namespace {

template <typename T> __device__ __forceinline__ float ld_f(const T* p);
template <> __device__ __forceinline__ float ld_f<float>(const float* p) { return *p; }
template <> __device__ __forceinline__ float ld_f<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}

// One warp per (pair (a, b), 32 consecutive channels): lane = channel.
template <typename Tw>
__global__ void __launch_bounds__(256)
alignment_kernel(const Tw* __restrict__ w_down, int K, int d, int H, float delta,
                 uint32_t* __restrict__ sets, int* __restrict__ counts) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  const int H32 = (H + 31) / 32;
  if (warp >= K * K * H32) return;
  const int pair = warp / H32, word = warp % H32;
  const int a = pair / K, b = pair % K;
  const int h = word * 32 + lane;
  bool aligned = false;
  if (h < H) {
    const Tw* va = w_down + (size_t)(1 + a) * d * H + h;  // V_{1+a}[h, i] at i * H
    const Tw* vb = w_down + (size_t)(1 + b) * d * H + h;
    float dot = 0.f, na = 0.f, nb = 0.f;
    for (int i = 0; i < d; ++i) {
      const float x = ld_f(va + (size_t)i * H), y = ld_f(vb + (size_t)i * H);
      dot = fmaf(x, y, dot);
      na = fmaf(x, x, na);
      nb = fmaf(y, y, nb);
    }
    const float den = sqrtf(na) * sqrtf(nb);
    aligned = den > 0.f && dot / den >= delta;
  }
  const uint32_t bits = __ballot_sync(0xffffffffu, aligned);
  if (lane == 0) {
    sets[(size_t)pair * H32 + word] = bits;
    if (bits) atomicAdd(counts + pair, __popc(bits));
  }
}

__global__ void alignment_finish_kernel(const int* __restrict__ counts, int KK, int H,
                                        float* __restrict__ rho) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k < KK) rho[k] = (float)counts[k] / (float)H;
}

// One warp per token: the top-2 pair of s = softmax(x W_g + bias) and its
// normalised weights, and the residual order q of x W_r (ranks; ties to the
// lower index). Lane l scores experts l and l + 32.
template <typename Tx>
__global__ void __launch_bounds__(256)
demand_route_kernel(const Tx* __restrict__ x, int T, int d, int K, const float* __restrict__ wr,
                    int Cp, const float* __restrict__ bias, const Tx* __restrict__ w_res,
                    int32_t* __restrict__ pair, float* __restrict__ wts,
                    int32_t* __restrict__ q) {
  const int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (t >= T) return;
  const Tx* xt = x + (size_t)t * d;
  float zg[2] = {-INFINITY, -INFINITY}, zr[2] = {-INFINITY, -INFINITY};
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int j = lane + 32 * u;
    if (j < K) {
      float g = 0.f, r = 0.f;
      for (int i = 0; i < d; ++i) {
        const float xv = ld_f(xt + i);
        g = fmaf(xv, wr[(size_t)i * Cp + 1 + j], g);
        r = fmaf(xv, ld_f(w_res + (size_t)i * K + j), r);
      }
      zg[u] = g + bias[1 + j];
      zr[u] = r;
    }
  }
  // the two largest affinities (softmax is monotone: rank the logits)
  int best = -1, second = -1;
  float bz = -INFINITY, sz = -INFINITY;
  for (int j = 0; j < K; ++j) {
    const float zj = __shfl_sync(0xffffffffu, zg[j >> 5], j & 31);
    if (best < 0 || zj > bz) {
      second = best; sz = bz;
      best = j; bz = zj;
    } else if (second < 0 || zj > sz) {
      second = j; sz = zj;
    }
  }
  // residual order: rank of each expert's score
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int j = lane + 32 * u;
    int rank = 0;
    for (int i = 0; i < K; ++i) {
      const float zi = __shfl_sync(0xffffffffu, zr[i >> 5], i & 31);
      rank += (zi > zr[u]) || (zi == zr[u] && i < j);
    }
    if (j < K) q[(size_t)t * K + rank] = j;
  }
  if (lane == 0) {
    // s_second / s_best = exp(z_second - z_best)
    const float ratio = expf(sz - bz);
    pair[2 * t] = best;
    pair[2 * t + 1] = second;
    wts[2 * t] = 1.0f / (1.0f + ratio);
    wts[2 * t + 1] = ratio / (1.0f + ratio);
  }
}

// One block per (token, expert): G[h] = GeLU(x K_e[:, h]) for every channel,
// then E_e[i] = sum_h G[h] V_e[h, i] and E_e^S[i] over the token's pair set.
template <typename Tw>
__global__ void __launch_bounds__(256)
demand_expert_kernel(const Tw* __restrict__ x, int T, int d, int H, int K,
                     const Tw* __restrict__ w_up, const Tw* __restrict__ w_down,
                     const uint32_t* __restrict__ sets, const int32_t* __restrict__ pair,
                     float* __restrict__ E, float* __restrict__ ES) {
  extern __shared__ float sm[];
  float* xs = sm;       // [d]
  float* G = xs + d;    // [H]
  uint32_t* S = reinterpret_cast<uint32_t*>(G + H);  // [H32]
  const int t = blockIdx.x / K, e = blockIdx.x % K;
  const int H32 = (H + 31) / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int i = threadIdx.x; i < d; i += blockDim.x) xs[i] = ld_f(x + (size_t)t * d + i);
  const uint32_t* st = sets + ((size_t)pair[2 * t] * K + pair[2 * t + 1]) * H32;
  for (int w = threadIdx.x; w < H32; w += blockDim.x) S[w] = st[w];
  __syncthreads();
  const Tw* ku = w_up + (size_t)(1 + e) * H * d;
  for (int h = warp; h < H; h += nw) {
    const Tw* kh = ku + (size_t)h * d;
    float a = 0.f;
    for (int i = lane; i < d; i += 32) a = fmaf(xs[i], ld_f(kh + i), a);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
    if (lane == 0) G[h] = 0.5f * a * (1.0f + erff(a * 0.70710678118654752f));
  }
  __syncthreads();
  const Tw* vd = w_down + (size_t)(1 + e) * d * H;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const Tw* vi = vd + (size_t)i * H;  // V_e[h, i] over h
    float all = 0.f, shr = 0.f;
    for (int h = 0; h < H; ++h) {
      const float p = G[h] * ld_f(vi + h);
      all += p;
      if ((S[h >> 5] >> (h & 31)) & 1u) shr += p;
    }
    E[((size_t)t * K + e) * d + i] = all;
    ES[((size_t)t * K + e) * d + i] = shr;
  }
}

// One warp per token: the ridge fits of Eq. diagnostic-projection for every
// prefix m (fp64 Gram matrix, right-hand side and Cholesky solve), the
// errors of Eq. diagnostic-error and k_eps. Shared memory per warp: the
// Gram matrix [K][K], b [K], a [K] (fp64).
__global__ void __launch_bounds__(32)
demand_fit_kernel(int T, int d, int K, const float* __restrict__ E, const float* __restrict__ ES,
                  const int32_t* __restrict__ pair, const float* __restrict__ wts,
                  const int32_t* __restrict__ q, float eps, int32_t* __restrict__ k_eps,
                  float* __restrict__ err) {
  extern __shared__ double dm[];
  double* Gm = dm;            // [K][K]
  double* bv = Gm + K * K;    // [K]
  double* av = bv + K;        // [K]
  double* Lc = av + K;        // [K][K] Cholesky factor
  const int t = blockIdx.x, lane = threadIdx.x;
  const int pi = pair[2 * t], pj = pair[2 * t + 1];
  const float wi = wts[2 * t], wj = wts[2 * t + 1];
  const float* Et = E + (size_t)t * K * d;
  const float* ESt = ES + (size_t)t * K * d;
  auto rrow = [&](int e, int i) { return (double)Et[e * d + i] - (double)ESt[e * d + i]; };
  auto target = [&](int i) {  // r = y_orig - S_bar
    return (double)wi * rrow(pi, i) + (double)wj * rrow(pj, i);
  };
  auto warp_sum = [&](double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
  };
  double yn = 0.0;
  for (int i = lane; i < d; i += 32) {
    const double y = (double)wi * Et[pi * d + i] + (double)wj * Et[pj * d + i];
    yn += y * y;
  }
  yn = fmax(sqrt(warp_sum(yn)), 1e-12);
  int kfound = K + 1;
  for (int m = 1; m <= K; ++m) {
    const int em = q[(size_t)t * K + m - 1];
    // new row m-1 of the Gram matrix and of b
    for (int k = 0; k < m; ++k) {
      const int ek = q[(size_t)t * K + k];
      double g = 0.0;
      for (int i = lane; i < d; i += 32) g += rrow(em, i) * rrow(ek, i);
      g = warp_sum(g);
      if (lane == 0) { Gm[(m - 1) * K + k] = g; Gm[k * K + m - 1] = g; }
    }
    double b = 0.0;
    for (int i = lane; i < d; i += 32) b += rrow(em, i) * target(i);
    b = warp_sum(b);
    if (lane == 0) bv[m - 1] = b;
    __syncwarp();
    if (lane == 0) {
      double tr = 0.0;
      for (int k = 0; k < m; ++k) tr += Gm[k * K + k];
      if (tr > 0.0) {
        const double gam = 1e-6 * tr / m;
        // Cholesky of G_m + gamma I, then the two triangular solves
        for (int r = 0; r < m; ++r) {
          for (int c = 0; c <= r; ++c) {
            double v = Gm[r * K + c] + (r == c ? gam : 0.0);
            for (int k = 0; k < c; ++k) v -= Lc[r * K + k] * Lc[c * K + k];
            Lc[r * K + c] = r == c ? sqrt(fmax(v, 1e-300)) : v / Lc[c * K + c];
          }
        }
        for (int r = 0; r < m; ++r) {
          double v = bv[r];
          for (int k = 0; k < r; ++k) v -= Lc[r * K + k] * av[k];
          av[r] = v / Lc[r * K + r];
        }
        for (int r = m - 1; r >= 0; --r) {
          double v = av[r];
          for (int k = r + 1; k < m; ++k) v -= Lc[k * K + r] * av[k];
          av[r] = v / Lc[r * K + r];
        }
      } else {
        for (int r = 0; r < m; ++r) av[r] = 0.0;
      }
    }
    __syncwarp();
    // e_m = |a^T R_m - r| / max(|y_orig|, 1e-12)
    double res = 0.0;
    for (int i = lane; i < d; i += 32) {
      double v = -target(i);
      for (int k = 0; k < m; ++k) v += av[k] * rrow(q[(size_t)t * K + k], i);
      res += v * v;
    }
    const double e_m = sqrt(warp_sum(res)) / yn;
    if (lane == 0 && err) err[(size_t)t * K + m - 1] = (float)e_m;
    if (kfound == K + 1 && e_m <= (double)eps) kfound = m;
    __syncwarp();
  }
  if (lane == 0) k_eps[t] = kfound;
}

}  // namespace

int diag_alignment(unif_moe_layer* L, float delta, float* rho, cudaStream_t s) {
  Workspace& w = L->ws;
  const int K = L->K, H32 = (L->H + 31) / 32;
  if (cudaMemsetAsync(w.diag_counts, 0, sizeof(int) * K * K, s) != cudaSuccess) return -1;
  const int warps = K * K * H32;
  if (L->dtype == UNIF_MOE_BF16)
    alignment_kernel<<<(warps * 32 + 255) / 256, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(L->w_down), K, L->d, L->H, delta, w.diag_sets,
        w.diag_counts);
  else
    alignment_kernel<<<(warps * 32 + 255) / 256, 256, 0, s>>>(
        static_cast<const float*>(L->w_down), K, L->d, L->H, delta, w.diag_sets, w.diag_counts);
  if (rho)
    alignment_finish_kernel<<<(K * K + 255) / 256, 256, 0, s>>>(w.diag_counts, K * K, L->H, rho);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

int diag_demand(unif_moe_layer* L, const void* x, int T, const void* w_res, float delta,
                float eps, int32_t* k_eps, float* err, int32_t* pair_out, cudaStream_t s) {
  Workspace& w = L->ws;
  const int K = L->K, d = L->d, H = L->H;
  if (diag_alignment(L, delta, nullptr, s) != 0) return -1;
  const int rt_blocks = (T * 32 + 255) / 256;
  const size_t esm = sizeof(float) * ((size_t)d + H) + sizeof(uint32_t) * ((H + 31) / 32);
  if (L->dtype == UNIF_MOE_BF16) {
    const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
    demand_route_kernel<<<rt_blocks, 256, 0, s>>>(
        xb, T, d, K, L->wr, L->router_cols_pad, L->bias,
        static_cast<const __nv_bfloat16*>(w_res), w.diag_pair, w.diag_wts, w.diag_q);
    demand_expert_kernel<<<T * K, 256, esm, s>>>(
        xb, T, d, H, K, static_cast<const __nv_bfloat16*>(L->w_up),
        static_cast<const __nv_bfloat16*>(L->w_down), w.diag_sets, w.diag_pair, w.diag_E,
        w.diag_ES);
  } else {
    const float* xf = static_cast<const float*>(x);
    demand_route_kernel<<<rt_blocks, 256, 0, s>>>(
        xf, T, d, K, L->wr, L->router_cols_pad, L->bias, static_cast<const float*>(w_res),
        w.diag_pair, w.diag_wts, w.diag_q);
    demand_expert_kernel<<<T * K, 256, esm, s>>>(
        xf, T, d, H, K, static_cast<const float*>(L->w_up), static_cast<const float*>(L->w_down),
        w.diag_sets, w.diag_pair, w.diag_E, w.diag_ES);
  }
  demand_fit_kernel<<<T, 32, sizeof(double) * (2 * (size_t)K * K + 2 * K), s>>>(
      T, d, K, w.diag_E, w.diag_ES, w.diag_pair, w.diag_wts, w.diag_q, eps, k_eps, err);
  if (pair_out &&
      cudaMemcpyAsync(pair_out, w.diag_pair, sizeof(int32_t) * 2 * (size_t)T,
                      cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return -1;
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace unif
