/*
 * UniF-MoE layer forward pass: plain CPU oracle in fp64.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path may call, link or
 * load this file: only the tests, the smoke check and the benchmark's CPU
 * baseline leg use it. It shares no code, header, table or constant with the
 * CUDA implementation.
 *
 * Every function follows the paper ("Share First, Route What Remains",
 * Sec. III) one equation at a time, in the paper's notation:
 *   x        one token, 1 x d
 *   W*       = [W_shr, W_g], d x (K+1)                        (Eq. 17)
 *   alpha    = tau + (1 - 2 tau) sigmoid(x W_shr), tau=(B-1)/B^2 (Eq. 18)
 *   b        = round(B alpha)                                  (Eq. 19)
 *   mu_b     = (1/M) sum_{h in H_b} K_shr[:, h]                (Eq. 20)
 *   u_b      = x mu_b                                          (Eq. 21)
 *   I_shr    = TopK(u, b), I_res = complement                  (Eqs. 22-23)
 *   s        = softmax(x W_g)                                  (Eq. 24)
 *   q, p     = experts sorted by decreasing s                  (Eq. 25)
 *   beta     = 1 - alpha                                       (Eq. 26)
 *   k        = min{n : sum_{i<=n} p_i >= beta}                 (Eq. 27)
 *   E_j^(b)  = sum_{h in H_b} GeLU(x K_j[:,h]) V_j[h,:]        (Eq. 16)
 *   y        = alpha sum_{b in I_shr} E_shr^(b)
 *              + sum_{i<=k} p_i sum_{b in I_res} E_{q_i}^(b)   (Eqs. 28-30)
 *
 * Weight layouts (torch.nn.Linear convention):
 *   w_router [d][K+1]     column 0 = W_shr, columns 1..K = W_g
 *   w_up     [K+1][H][d]  expert 0 = shared; w_up[e][h][:] = K_e[:, h]
 *   w_down   [K+1][d][H]  w_down[e][:][h] = V_e[h, :]
 *
 * Readings where the paper is silent (each also listed with the design notes):
 *   - round() in Eq. 19 is round-half-to-even (the C default rounding mode).
 *   - TopK in Eq. 22 and the sort in Eq. 25 break ties toward the lower index.
 *   - If rounding leaves every prefix of Eq. 27 below beta, k is clamped to K.
 *   - GeLU is the exact erf form 0.5 v (1 + erf(v / sqrt 2)).
 *   - The prototypes mu_b are formed exactly from the stored shared keys and
 *     rounded once, to nearest-even, to the precision the router weights are
 *     stored in (fp32 or bf16); the same rounded mu is then used in Eq. 21.
 *   - Optional router bias (one value per router column) is added to x W*;
 *     the paper omits biases for clarity, the value 0 reproduces it.
 *   - Ablation switches (Table IV): a fixed alpha, a fixed beta (theta), a
 *     fixed residual count (top-k) and prefix block selection.
 *   - Masked (padding) tokens take no decision and produce y = 0.
 *
 * Near-tie margins (per token, in fp64): (i) |B alpha - (floor(B alpha)+1/2)|/B,
 * (ii) u_(b) - u_(b+1) over sorted priorities, (iii) min(P_k - beta,
 * beta - P_{k-1}), (iv) p_k - p_{k+1}. A switch that is fixed has margin +inf.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_MAX_K 64
#define ORACLE_MAX_B 64

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* Round an fp64 value to the nearest bfloat16 (8 significant bits), ties to
 * even, with one rounding step. */
static double round_to_bf16(double v) {
  if (v == 0.0 || !isfinite(v)) return v;
  if (fabs(v) < 0x1p-126) return nearbyint(v * 0x1p133) * 0x1p-133; /* subnormal */
  int e;
  double m = frexp(v, &e); /* v = m 2^e, 0.5 <= |m| < 1 */
  return ldexp(nearbyint(ldexp(m, 8)), e - 8);
}

static double round_to(double v, int mode) {
  if (mode == 1) return (double)(float)v;
  if (mode == 2) return round_to_bf16(v);
  return v;
}

/* Eq. 20: mu_b = (1/M) sum_{h in H_b} K_shr[:, h], one d-vector per block.
 * w_up0 is the shared expert's up-projection [H][d]. round_mode: 0 keep
 * fp64, 1 round to fp32, 2 round to bf16. mu is [B][d]. */
int oracle_prototypes(const double* w_up0, int d, int H, int B, int round_mode,
                      double* mu) {
  if (!w_up0 || !mu || d <= 0 || H <= 0 || B <= 0 || H % B) return -1;
  const int M = H / B;
  for (int b = 0; b < B; ++b) {
    for (int i = 0; i < d; ++i) {
      double sum = 0.0;
      for (int h = b * M; h < (b + 1) * M; ++h) sum += w_up0[(size_t)h * d + i];
      mu[(size_t)b * d + i] = round_to(sum / (double)M, round_mode);
    }
  }
  return 0;
}

static double sigmoid(double z) { return 1.0 / (1.0 + exp(-z)); }

static double gelu(double v) { return 0.5 * v * (1.0 + erf(v * M_SQRT1_2)); }

/* Order indices 0..n-1 by decreasing value; equal values keep the lower
 * index first. Plain insertion sort. */
static void sort_desc(const double* val, int n, int* order) {
  for (int i = 0; i < n; ++i) order[i] = i;
  for (int i = 1; i < n; ++i) {
    int cur = order[i];
    int j = i - 1;
    while (j >= 0 && (val[order[j]] < val[cur] ||
                      (val[order[j]] == val[cur] && order[j] > cur))) {
      order[j + 1] = order[j];
      --j;
    }
    order[j + 1] = cur;
  }
}

/* Routing decisions for T tokens (Eqs. 17-27).
 *   x [T][d], mask [T] (NULL = all real), w_router [d][K+1],
 *   bias [K+1] or NULL, mu [B][d] (from oracle_prototypes),
 *   th[5] = {tau (NaN = (B-1)/B^2), alpha_fixed (NaN = adaptive),
 *            beta_fixed (NaN = 1 - alpha), topk_fixed (0 = cumulative),
 *            prefix_blocks (0 = prototype TopK)}.
 * Outputs (all [T] or [T][n]):
 *   alpha, beta, b, k, shr_mask (bit blk set = block blk shared),
 *   q [T][K] residual experts 0..K-1 by decreasing affinity, p [T][K] their
 *   affinities, s [T][K] unsorted affinities (Eq. 24), u [T][B] priorities,
 *   margin [T][4] near-tie margins (i)-(iv). */
int oracle_route(int T, int d, int K, int B, const double* x, const uint8_t* mask,
                 const double* w_router, const double* bias, const double* mu,
                 const double* th, double* alpha_out, double* beta_out,
                 int32_t* b_out, int32_t* k_out, uint64_t* shr_mask_out,
                 int32_t* q_out, double* p_out, double* s_out, double* u_out,
                 double* margin_out) {
  if (T < 0 || d <= 0 || K <= 0 || K > ORACLE_MAX_K || B < 1 || B > ORACLE_MAX_B)
    return -1;
  const double tau = isnan(th[0]) ? (double)(B - 1) / ((double)B * B) : th[0];
  const double alpha_fixed = th[1], beta_fixed = th[2];
  const int topk_fixed = (int)th[3], prefix_blocks = (int)th[4];
  if (topk_fixed < 0 || topk_fixed > K) return -1;

#pragma omp parallel for schedule(dynamic, 64)
  for (int t = 0; t < T; ++t) {
    const double* xt = x + (size_t)t * d;
    int32_t* q = q_out + (size_t)t * K;
    double* p = p_out + (size_t)t * K;
    double* s = s_out + (size_t)t * K;
    double* u = u_out + (size_t)t * B;
    double* mg = margin_out + (size_t)t * 4;
    if (mask && !mask[t]) { /* padding: no decision, no work */
      alpha_out[t] = 0.0; beta_out[t] = 0.0; b_out[t] = 0; k_out[t] = 0;
      shr_mask_out[t] = 0;
      for (int j = 0; j < K; ++j) { q[j] = j; p[j] = 0.0; s[j] = 0.0; }
      for (int j = 0; j < B; ++j) u[j] = 0.0;
      for (int j = 0; j < 4; ++j) mg[j] = INFINITY;
      continue;
    }
    /* Eq. 17: router logits x W* (+ optional bias). */
    double z[ORACLE_MAX_K + 1];
    for (int j = 0; j <= K; ++j) {
      double acc = 0.0;
      for (int i = 0; i < d; ++i) acc += xt[i] * w_router[(size_t)i * (K + 1) + j];
      z[j] = acc + (bias ? bias[j] : 0.0);
    }
    /* Eq. 18: shared demand; Eq. 19: shared block count. */
    const double alpha = isnan(alpha_fixed) ? tau + (1.0 - 2.0 * tau) * sigmoid(z[0])
                                            : alpha_fixed;
    int b = (int)nearbyint((double)B * alpha);
    if (b < 0) b = 0;
    if (b > B) b = B;
    /* Eq. 21: block priorities; Eqs. 22-23: shared / residual blocks. */
    for (int blk = 0; blk < B; ++blk) {
      double acc = 0.0;
      for (int i = 0; i < d; ++i) acc += xt[i] * mu[(size_t)blk * d + i];
      u[blk] = acc;
    }
    int uorder[ORACLE_MAX_B];
    sort_desc(u, B, uorder);
    uint64_t shr = 0;
    for (int r = 0; r < b; ++r) shr |= 1ull << (prefix_blocks ? r : uorder[r]);
    /* Eq. 24: affinities over the K residual experts. */
    double zmax = z[1];
    for (int j = 2; j <= K; ++j) zmax = z[j] > zmax ? z[j] : zmax;
    double den = 0.0;
    for (int j = 0; j < K; ++j) { s[j] = exp(z[j + 1] - zmax); den += s[j]; }
    for (int j = 0; j < K; ++j) s[j] /= den;
    /* Eq. 25: sorted affinities. */
    int order[ORACLE_MAX_K];
    sort_desc(s, K, order);
    for (int i = 0; i < K; ++i) { q[i] = order[i]; p[i] = s[order[i]]; }
    /* Eq. 26: residual demand; Eq. 27: smallest sufficient prefix. */
    const double beta = isnan(beta_fixed) ? 1.0 - alpha : beta_fixed;
    int k = K;
    double P = 0.0, P_k = 0.0;
    if (topk_fixed > 0) {
      k = topk_fixed;
    } else {
      for (int n = 1; n <= K; ++n) {
        P += p[n - 1];
        if (P >= beta) { k = n; break; }
      }
    }
    P_k = 0.0;
    for (int i = 0; i < k; ++i) P_k += p[i];
    alpha_out[t] = alpha;
    beta_out[t] = beta;
    b_out[t] = b;
    k_out[t] = k;
    shr_mask_out[t] = shr;
    /* Near-tie margins. */
    if (isnan(alpha_fixed)) {
      const double r = (double)B * alpha;
      mg[0] = fabs(r - (floor(r) + 0.5)) / (double)B;
    } else {
      mg[0] = INFINITY;
    }
    mg[1] = (prefix_blocks || b <= 0 || b >= B) ? INFINITY : u[uorder[b - 1]] - u[uorder[b]];
    if (topk_fixed > 0) {
      mg[2] = INFINITY;
    } else {
      double prev = 0.0;
      for (int i = 0; i < k - 1; ++i) prev += p[i];
      mg[2] = fmin(P_k - beta, beta - prev);
    }
    mg[3] = (k < K) ? p[k - 1] - p[k] : INFINITY;
  }
  return 0;
}

/* Layer output (Eqs. 16, 28-30) for given decisions.
 *   alpha [T], b [T] (informational), shr_mask [T], k [T], q [T][K], p [T][K]
 *   as produced by oracle_route (or any other decisions to evaluate),
 *   mask [T] or NULL, y [T][d] output.
 * E_j^(b)(x) is evaluated channel by channel exactly as Eq. 16 writes it. */
int oracle_forward(int T, int d, int H, int K, int B, const double* x,
                   const uint8_t* mask, const double* w_up, const double* w_down,
                   const double* alpha, const uint64_t* shr_mask, const int32_t* k_in,
                   const int32_t* q_in, const double* p_in, double* y) {
  if (T < 0 || d <= 0 || H <= 0 || K <= 0 || B <= 0 || H % B || B > ORACLE_MAX_B)
    return -1;
  const int M = H / B;
  /* Layout copy only: value rows V_j[h, :] made contiguous. */
  double* V = (double*)malloc(sizeof(double) * (size_t)(K + 1) * H * d);
  if (!V) return -2;
  for (int e = 0; e <= K; ++e)
    for (int i = 0; i < d; ++i)
      for (int h = 0; h < H; ++h)
        V[((size_t)e * H + h) * d + i] = w_down[((size_t)e * d + i) * H + h];

#pragma omp parallel
  {
    double* acc = (double*)malloc(sizeof(double) * (size_t)d);
#pragma omp for schedule(dynamic, 16)
    for (int t = 0; t < T; ++t) {
      const double* xt = x + (size_t)t * d;
      double* yt = y + (size_t)t * d;
      for (int i = 0; i < d; ++i) yt[i] = 0.0;
      if (mask && !mask[t]) continue;
      /* One expert's selected blocks: sum_{blk in set} E_e^(blk)(x). */
#define EXPERT_BLOCKS(e, want_shared)                                              \
  do {                                                                             \
    for (int i = 0; i < d; ++i) acc[i] = 0.0;                                      \
    for (int blk = 0; blk < B; ++blk) {                                            \
      const int in_shr = (int)((shr_mask[t] >> blk) & 1ull);                       \
      if (in_shr != (want_shared)) continue;                                       \
      for (int h = blk * M; h < (blk + 1) * M; ++h) {                              \
        const double* key = w_up + ((size_t)(e) * H + h) * d;                      \
        double a = 0.0;                                                            \
        for (int i = 0; i < d; ++i) a += xt[i] * key[i];                           \
        const double g = gelu(a);                                                  \
        const double* val = V + ((size_t)(e) * H + h) * d;                         \
        for (int i = 0; i < d; ++i) acc[i] += g * val[i];                          \
      }                                                                            \
    }                                                                              \
  } while (0)
      /* Eq. 28 weighted by alpha (Eq. 30, first term). */
      EXPERT_BLOCKS(0, 1);
      for (int i = 0; i < d; ++i) yt[i] += alpha[t] * acc[i];
      /* Eq. 29 for each selected residual expert, weighted by p_i (Eq. 30). */
      for (int r = 0; r < k_in[t]; ++r) {
        const int j = q_in[(size_t)t * K + r];
        EXPERT_BLOCKS(1 + j, 0);
        const double pr = p_in[(size_t)t * K + r];
        for (int i = 0; i < d; ++i) yt[i] += pr * acc[i];
      }
#undef EXPERT_BLOCKS
    }
    free(acc);
  }
  free(V);
  return 0;
}

/* Group table: the (expert, block) pairs of Eqs. 28-29 gathered by pair.
 * Group g = e*B + blk, e = 0 for the shared expert and e = 1+j for residual
 * expert j. For each group, its tokens in increasing token order with the
 * pathway weight (alpha for the shared expert, p_i for residual expert q_i).
 * counts [(K+1)B]; rows_token / rows_weight hold the groups one after
 * another (group 0 first), sum(counts) entries, which is sum_t C_B(t)
 * (Eq. 35). Returns the total number of rows, or -1 if it exceeds cap. */
long long oracle_groups(int T, int K, int B, const uint8_t* mask, const double* alpha,
                        const uint64_t* shr_mask, const int32_t* k_in,
                        const int32_t* q_in, const double* p_in, int32_t* counts,
                        int32_t* rows_token, double* rows_weight, long long cap) {
  const int G = (K + 1) * B;
  long long total = 0;
  for (int g = 0; g < G; ++g) {
    const int e = g / B, blk = g % B;
    int c = 0;
    for (int t = 0; t < T; ++t) {
      if (mask && !mask[t]) continue;
      const int shared_blk = (int)((shr_mask[t] >> blk) & 1ull);
      double w = 0.0;
      int hit = 0;
      if (e == 0) {
        if (shared_blk) { hit = 1; w = alpha[t]; }
      } else if (!shared_blk) {
        for (int r = 0; r < k_in[t]; ++r)
          if (q_in[(size_t)t * K + r] == e - 1) { hit = 1; w = p_in[(size_t)t * K + r]; }
      }
      if (!hit) continue;
      if (total >= cap) return -1;
      rows_token[total] = t;
      rows_weight[total] = w;
      ++total;
      ++c;
    }
    counts[g] = c;
  }
  return total;
}

/* The layer inside a Transformer sublayer (the converted FFN layers of the
 * paper's DeiT-S and BERT backbones, Appendix A, Architecture details):
 * layer normalisation of each token over its d features, in the standard form
 *   LN(v) = gamma * (v - mean(v)) / sqrt(var(v) + eps) + beta,
 * mean and var over the d features, var the biased (1/d) second central
 * moment. Rows whose mask entry is 0 (padding) give 0. The result is
 * rounded per round_mode (the precision the layer's inputs are kept in).
 * v, out [T][d]; gamma, beta [d]; mask [T] or NULL. */
int oracle_layernorm(int T, int d, const double* v, const uint8_t* mask, const double* gamma,
                     const double* beta, double eps, int round_mode, double* out) {
  if (T < 0 || d <= 0 || !v || !gamma || !beta || !out || !(eps >= 0.0)) return -1;
  for (int t = 0; t < T; ++t) {
    const double* row = v + (size_t)t * d;
    double* o = out + (size_t)t * d;
    if (mask && !mask[t]) {
      for (int i = 0; i < d; ++i) o[i] = 0.0;
      continue;
    }
    double mean = 0.0;
    for (int i = 0; i < d; ++i) mean += row[i];
    mean /= (double)d;
    double var = 0.0;
    for (int i = 0; i < d; ++i) var += (row[i] - mean) * (row[i] - mean);
    var /= (double)d;
    const double inv = 1.0 / sqrt(var + eps);
    for (int i = 0; i < d; ++i) o[i] = round_to(gamma[i] * (row[i] - mean) * inv + beta[i], round_mode);
  }
  return 0;
}

/* ------------------------------------------------------------------------
 * Training (Sec. III-E): gradients of a loss through the layer output.
 * ------------------------------------------------------------------------ */

/* d GeLU / dv = Phi(v) + v phi(v), the derivative of the exact erf form. */
static double gelu_grad(double v) {
  return 0.5 * (1.0 + erf(v * M_SQRT1_2)) + v * exp(-0.5 * v * v) / sqrt(2.0 * M_PI);
}

/* Gradient of a scalar loss L given dL/dy (dy [T][d]) through the output of
 * Eq. 30, with the discrete decisions held fixed: the shared block set
 * (shr_mask, Eq. 22) and the set of selected residual experts (expert_mask,
 * bit j = expert j, Eq. 27) are piecewise constant in the parameters (the
 * rounding of Eq. 19, the TopK of Eq. 22 and the smallest prefix of Eq. 27
 * move only at ties), so gradients flow through the pathway weights alpha
 * (Eq. 18) and p_i = s_{q_i} (Eqs. 24-25), which are recomputed here from x
 * and the router, and through the expert weights (Eq. 16). With alpha fixed
 * (th[1] not NaN) it has no gradient; the prototypes mu_b only rank blocks
 * and receive none.
 *   y = alpha sum_{b in I_shr} E_shr^(b) + sum_{j selected} s_j sum_{b not in I_shr} E_j^(b)
 * Per token and block channel h of expert e with weight w (alpha or s_j),
 * a = x K_e[:, h]:
 *   dL/dV_e[h, :] += w GeLU(a) dy,   dL/da = w (dy . V_e[h, :]) GeLU'(a),
 *   dL/dK_e[:, h] += (dL/da) x,      dL/dx += (dL/da) K_e[:, h],
 *   dL/dw += GeLU(a) (dy . V_e[h, :]);
 * then alpha = tau + (1 - 2 tau) sigmoid(z_0) and s = softmax(z_1..z_K),
 * z = x W* + bias, give dL/dz and dL/dW* = x^T dL/dz, dL/dbias = dL/dz,
 * dL/dx += dL/dz W*^T.
 * Outputs (overwritten): dx [T][d], dw_up [K+1][H][d], dw_down [K+1][d][H],
 * dw_router [d][K+1], dbias [K+1] or NULL. Padding tokens (mask 0) add
 * nothing and get dx = 0. */
int oracle_backward(int T, int d, int H, int K, int B, const double* x, const uint8_t* mask,
                    const double* w_router, const double* bias, const double* w_up,
                    const double* w_down, const double* th, const uint64_t* shr_mask,
                    const uint64_t* expert_mask, const double* dy, double* dx,
                    double* dw_up, double* dw_down, double* dw_router, double* dbias) {
  if (T < 0 || d <= 0 || H <= 0 || K <= 0 || K > ORACLE_MAX_K || B <= 0 || H % B ||
      B > ORACLE_MAX_B)
    return -1;
  const int M = H / B;
  const int K1 = K + 1;
  const double tau = isnan(th[0]) ? (double)(B - 1) / ((double)B * B) : th[0];
  const int adaptive = isnan(th[1]);
  double* dz = (double*)calloc((size_t)T * K1, sizeof(double));
  /* alpha and s of every token, kept for the weight gradients of pass 2 */
  double* alpha_all = (double*)calloc((size_t)T, sizeof(double));
  double* s_all = (double*)calloc((size_t)T * K, sizeof(double));
  /* Layout copies only: value rows V_e[h, :] contiguous, and their
   * gradients accumulated in the same layout before the transposition into
   * dw_down. */
  double* V = (double*)malloc(sizeof(double) * (size_t)K1 * H * d);
  double* dV = (double*)malloc(sizeof(double) * (size_t)K1 * H * d);
  if (!dz || !alpha_all || !s_all || !V || !dV) {
    free(dz);
    free(alpha_all);
    free(s_all);
    free(V);
    free(dV);
    return -2;
  }
  for (int e = 0; e < K1; ++e)
    for (int i = 0; i < d; ++i)
      for (int h = 0; h < H; ++h)
        V[((size_t)e * H + h) * d + i] = w_down[((size_t)e * d + i) * H + h];

  /* The pathway weight of expert e for token t (0: not used by t). */
#define PATH_WEIGHT(e, alpha_t, s_t, t)                                                 \
  ((e) == 0 ? (shr_mask[t] != 0 ? (alpha_t) : 0.0)                                     \
            : (((expert_mask[t] >> ((e) - 1)) & 1ull) ? (s_t)[(e) - 1] : 0.0))
  /* Whether expert e runs block blk for token t (Eqs. 28-29). */
#define RUNS_BLOCK(e, blk, t) \
  ((e) == 0 ? (int)((shr_mask[t] >> (blk)) & 1ull) : !(int)((shr_mask[t] >> (blk)) & 1ull))

  /* Router scores of token t: alpha (Eq. 18) and s (Eq. 24) from z = x W* + bias. */
#define ROUTER_SCORES(t, z, alpha_t, s_t)                                               \
  do {                                                                                  \
    const double* xt_ = x + (size_t)(t) * d;                                            \
    for (int c = 0; c < K1; ++c) {                                                      \
      double acc = 0.0;                                                                 \
      for (int i = 0; i < d; ++i) acc += xt_[i] * w_router[(size_t)i * K1 + c];         \
      (z)[c] = acc + (bias ? bias[c] : 0.0);                                            \
    }                                                                                   \
    (alpha_t) = adaptive ? tau + (1.0 - 2.0 * tau) * sigmoid((z)[0]) : th[1];            \
    double zm = (z)[1];                                                                 \
    for (int j = 2; j <= K; ++j) zm = (z)[j] > zm ? (z)[j] : zm;                        \
    double den = 0.0;                                                                   \
    for (int j = 0; j < K; ++j) { (s_t)[j] = exp((z)[j + 1] - zm); den += (s_t)[j]; }  \
    for (int j = 0; j < K; ++j) (s_t)[j] /= den;                                        \
  } while (0)

  /* Pass 1, per token: dL/dx through the experts, dL/dalpha and dL/ds, then
   * dL/dz and its share of dL/dx. */
#pragma omp parallel for schedule(dynamic, 16)
  for (int t = 0; t < T; ++t) {
    double* dxt = dx + (size_t)t * d;
    for (int i = 0; i < d; ++i) dxt[i] = 0.0;
    if (mask && !mask[t]) continue;
    const double* xt = x + (size_t)t * d;
    const double* gt = dy + (size_t)t * d;
    double z[ORACLE_MAX_K + 1], s[ORACLE_MAX_K], dw[ORACLE_MAX_K + 1];
    double alpha;
    ROUTER_SCORES(t, z, alpha, s);
    alpha_all[t] = alpha;
    for (int j = 0; j < K; ++j) s_all[(size_t)t * K + j] = s[j];
    for (int e = 0; e < K1; ++e) {
      dw[e] = 0.0;
      const double w = PATH_WEIGHT(e, alpha, s, t);
      if (e > 0 && !((expert_mask[t] >> (e - 1)) & 1ull)) continue;
      if (e == 0 && shr_mask[t] == 0) continue;
      for (int blk = 0; blk < B; ++blk) {
        if (!RUNS_BLOCK(e, blk, t)) continue;
        for (int h = blk * M; h < (blk + 1) * M; ++h) {
          const double* key = w_up + ((size_t)e * H + h) * d;
          const double* val = V + ((size_t)e * H + h) * d;
          double a = 0.0, gv = 0.0;
          for (int i = 0; i < d; ++i) a += xt[i] * key[i];
          for (int i = 0; i < d; ++i) gv += gt[i] * val[i];
          dw[e] += gelu(a) * gv;
          const double da = w * gv * gelu_grad(a);
          for (int i = 0; i < d; ++i) dxt[i] += da * key[i];
        }
      }
    }
    /* Eq. 18: d alpha / d z_0 = (1 - 2 tau) sigma (1 - sigma). */
    double* dzt = dz + (size_t)t * K1;
    if (adaptive) {
      const double sg = sigmoid(z[0]);
      dzt[0] = dw[0] * (1.0 - 2.0 * tau) * sg * (1.0 - sg);
    }
    /* Eq. 24: softmax Jacobian, ds -> dz_j = s_j (ds_j - sum_l s_l ds_l). */
    double dot = 0.0;
    for (int j = 0; j < K; ++j) dot += s[j] * dw[1 + j];
    for (int j = 0; j < K; ++j) dzt[1 + j] = s[j] * (dw[1 + j] - dot);
    for (int c = 0; c < K1; ++c)
      for (int i = 0; i < d; ++i) dxt[i] += dzt[c] * w_router[(size_t)i * K1 + c];
  }

  /* Pass 2, per expert channel (e, h): the weight gradients, summed over the
   * tokens that run h's block of expert e. */
#pragma omp parallel for schedule(dynamic, 4)
  for (int eh = 0; eh < K1 * H; ++eh) {
    const int e = eh / H, h = eh % H, blk = h / M;
    double* gk = dw_up + ((size_t)e * H + h) * d;
    double* gvr = dV + ((size_t)e * H + h) * d;
    for (int i = 0; i < d; ++i) {
      gk[i] = 0.0;
      gvr[i] = 0.0;
    }
    const double* key = w_up + ((size_t)e * H + h) * d;
    const double* val = V + ((size_t)e * H + h) * d;
    for (int t = 0; t < T; ++t) {
      if (mask && !mask[t]) continue;
      if (!RUNS_BLOCK(e, blk, t)) continue;
      if (e > 0 && !((expert_mask[t] >> (e - 1)) & 1ull)) continue;
      const double* xt = x + (size_t)t * d;
      const double* gt = dy + (size_t)t * d;
      const double* s = s_all + (size_t)t * K;
      const double w = PATH_WEIGHT(e, alpha_all[t], s, t);
      double a = 0.0, gv = 0.0;
      for (int i = 0; i < d; ++i) a += xt[i] * key[i];
      for (int i = 0; i < d; ++i) gv += gt[i] * val[i];
      const double da = w * gv * gelu_grad(a);
      const double wg = w * gelu(a);
      for (int i = 0; i < d; ++i) {
        gk[i] += da * xt[i];
        gvr[i] += wg * gt[i];
      }
    }
  }
  for (int e = 0; e < K1; ++e)
    for (int i = 0; i < d; ++i)
      for (int h = 0; h < H; ++h)
        dw_down[((size_t)e * d + i) * H + h] = dV[((size_t)e * H + h) * d + i];

  /* Pass 3: dL/dW* = x^T dL/dz (Eq. 17), dL/dbias = sum_t dL/dz. */
#pragma omp parallel for schedule(static)
  for (int i = 0; i < d; ++i) {
    for (int c = 0; c < K1; ++c) {
      double acc = 0.0;
      for (int t = 0; t < T; ++t)
        if (!mask || mask[t]) acc += x[(size_t)t * d + i] * dz[(size_t)t * K1 + c];
      dw_router[(size_t)i * K1 + c] = acc;
    }
  }
  if (dbias) {
    for (int c = 0; c < K1; ++c) {
      double acc = 0.0;
      for (int t = 0; t < T; ++t)
        if (!mask || mask[t]) acc += dz[(size_t)t * K1 + c];
      dbias[c] = acc;
    }
  }
#undef PATH_WEIGHT
#undef RUNS_BLOCK
#undef ROUTER_SCORES
  free(dz);
  free(alpha_all);
  free(s_all);
  free(V);
  free(dV);
  return 0;
}

/* Gram regulariser of the router embeddings (Eq. diversity-loss):
 *   L_div = || W*^T W* - I_{K+1} ||_F,  W* = w_router [d][K+1],
 * and, with A = W*^T W* - I (symmetric), its gradient
 *   dL_div / dW* = 2 W* A / L_div   (0 where L_div = 0).
 * grad [d][K+1] may be NULL. Returns L_div. */
double oracle_diversity(int d, int K1, const double* w_router, double* grad) {
  double* A = (double*)malloc(sizeof(double) * (size_t)K1 * K1);
  if (!A) return NAN;
  double ss = 0.0;
  for (int a = 0; a < K1; ++a)
    for (int b = 0; b < K1; ++b) {
      double g = 0.0;
      for (int i = 0; i < d; ++i) g += w_router[(size_t)i * K1 + a] * w_router[(size_t)i * K1 + b];
      A[a * K1 + b] = g - (a == b ? 1.0 : 0.0);
      ss += A[a * K1 + b] * A[a * K1 + b];
    }
  const double L = sqrt(ss);
  if (grad) {
    for (int i = 0; i < d; ++i)
      for (int b = 0; b < K1; ++b) {
        double g = 0.0;
        for (int a = 0; a < K1; ++a) g += w_router[(size_t)i * K1 + a] * A[a * K1 + b];
        grad[(size_t)i * K1 + b] = L > 0.0 ? 2.0 * g / L : 0.0;
      }
  }
  free(A);
  return L;
}
