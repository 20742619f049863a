// Measurement probe (not part of the layer's C ABI; built into its own
// library, libunif_probe.so): the L2 throughput of fp32 row reductions in
// the pattern the down projection's epilogue uses, so that a benchmark can
// set the down projection's time against the rate its reductions allow.
//
// n_rows rows of d fp32 values (d a multiple of 32) are added into
// y[tok[r]][0 .. d) for random tokens. Each warp adds 32 rows at a time in
// 32-column passes: a warp instruction covers 4 rows x 128 contiguous bytes
// (lane l: row 4 i + l / 8, bytes 16 (l % 8) .. of the pass), one
// red.global.add.v4.f32 per lane, as the epilogue does from its staging tile.
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr int kWarps = 8;

__global__ void __launch_bounds__(32 * kWarps)
l2_reduction_probe(float* __restrict__ y, const int32_t* __restrict__ tok, int n_rows, int d,
                   int rows_per_cta) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r_sub = lane >> 3, c8 = lane & 7;
  const int r_begin = blockIdx.x * rows_per_cta;
  const int r_end = min(n_rows, r_begin + rows_per_cta);
  for (int r0 = r_begin + 32 * warp; r0 < r_end; r0 += 32 * kWarps) {
    int t[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = r0 + 4 * i + r_sub;
      t[i] = r < r_end ? tok[r] : -1;
    }
    for (int c = 0; c < d; c += 32) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (t[i] < 0) continue;
        float* dst = y + (size_t)t[i] * d + c + 4 * c8;
        asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dst), "f"(1.f),
                     "f"(1.f), "f"(1.f), "f"(1.f)
                     : "memory");
      }
    }
  }
}

}  // namespace

// Launches the probe on `stream`: rows split evenly over n_cta CTAs. y is
// [T][d] fp32 (device), tok [n_rows] int32 (device, every entry < T).
// Returns 0, or -1 for bad arguments, or the CUDA error code of the launch.
extern "C" __attribute__((visibility("default"))) int unif_probe_l2_reductions(
    float* y, const int32_t* tok, int n_rows, int d, int n_cta, void* stream) {
  if (!y || !tok || n_rows <= 0 || d <= 0 || d % 32 != 0 || n_cta <= 0) return -1;
  const int rows_per_cta = (n_rows + n_cta - 1) / n_cta;
  l2_reduction_probe<<<n_cta, 32 * kWarps, 0, static_cast<cudaStream_t>(stream)>>>(
      y, tok, n_rows, d, rows_per_cta);
  return (int)cudaGetLastError();
}
