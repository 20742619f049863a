"""The pins must catch plausible mistakes in the oracle. Each case below
plants one mistake in a copy of the oracle's C source (on the CPU, in a
temporary directory), builds it, and runs the pin suite against it with the
wrapper pointed at the broken library, or plants it in a copy of the Python
wrapper and runs the pins next to it: at least one pin has to fail."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "unif_moe_oracle.c")

MUTANTS = {
    # dropped factor (1 - 2 tau) in Eq. 18
    "alpha_dropped_term": ("tau + (1.0 - 2.0 * tau) * sigmoid(z[0])", "tau + sigmoid(z[0])"),
    # wrong sign inside the logistic function
    "sigmoid_sign": ("return 1.0 / (1.0 + exp(-z));", "return 1.0 / (1.0 + exp(z));"),
    # prototypes from the wrong expert's keys (Eq. 20 uses the shared expert)
    "prototype_off_by_one": ("sum += w_up0[(size_t)h * d + i];",
                             "sum += w_up0[(size_t)((h + 1) % H) * d + i];"),
    # sum instead of mean in Eq. 20 (changes nothing under exact TopK, but the
    # priorities pin sees it)
    "prototype_sum": ("round_to(sum / (double)M, round_mode)", "round_to(sum, round_mode)"),
    # transposed value matrix
    "value_transposed": ("  for (int e = 0; e <= K; ++e)\n    for (int i = 0; i < d; ++i)\n"
                         "      for (int h = 0; h < H; ++h)\n"
                         "        V[((size_t)e * H + h) * d + i] = w_down[((size_t)e * d + i) * H + h];",
                         "  for (int e = 0; e <= K; ++e)\n    for (int i = 0; i < d; ++i)\n"
                         "      for (int h = 0; h < H; ++h)\n"
                         "        V[((size_t)e * H + h) * d + i] = w_down[((size_t)e * H + h) * d + i];"),
    # the backward's value rows read transposed
    "bwd_value_transposed": ("  for (int e = 0; e < K1; ++e)\n    for (int i = 0; i < d; ++i)\n"
                             "      for (int h = 0; h < H; ++h)\n"
                             "        V[((size_t)e * H + h) * d + i] = w_down[((size_t)e * d + i) * H + h];",
                             "  for (int e = 0; e < K1; ++e)\n    for (int i = 0; i < d; ++i)\n"
                             "      for (int h = 0; h < H; ++h)\n"
                             "        V[((size_t)e * H + h) * d + i] = w_down[((size_t)e * H + h) * d + i];"),
    # residual experts run the shared blocks instead of the complement (Eq. 23)
    "residual_blocks": ("EXPERT_BLOCKS(1 + j, 0);", "EXPERT_BLOCKS(1 + j, 1);"),
    # shared pathway weighted by beta instead of alpha (Eq. 30)
    "shared_weight": ("yt[i] += alpha[t] * acc[i];", "yt[i] += (1.0 - alpha[t]) * acc[i];"),
    # TopK of the smallest priorities (Eq. 22)
    "topk_reversed": ("shr |= 1ull << (prefix_blocks ? r : uorder[r]);",
                      "shr |= 1ull << (prefix_blocks ? r : uorder[B - 1 - r]);"),
    # the selected prefix one expert too long (Eq. 27 asks for the smallest)
    "k_plus_one": ("if (P >= beta) { k = n; break; }", "if (P >= beta) { k = n < K ? n + 1 : K; break; }"),
    # affinity of the unsorted expert index used as the weight (Eq. 25)
    "p_unsorted": ("for (int i = 0; i < K; ++i) { q[i] = order[i]; p[i] = s[order[i]]; }",
                   "for (int i = 0; i < K; ++i) { q[i] = order[i]; p[i] = s[i]; }"),
    # round() replaced by truncation (Eq. 19)
    "b_truncated": ("int b = (int)nearbyint((double)B * alpha);", "int b = (int)((double)B * alpha);"),
    # GeLU without the 1/sqrt(2) scaling
    "gelu_scale": ("return 0.5 * v * (1.0 + erf(v * M_SQRT1_2));",
                   "return 0.5 * v * (1.0 + erf(v));"),
    # layer normalisation with the unbiased (1/(d-1)) variance
    "ln_unbiased_variance": ("    var /= (double)d;", "    var /= (double)(d - 1);"),
    # eps added outside the square root
    "ln_eps_outside": ("const double inv = 1.0 / sqrt(var + eps);",
                       "const double inv = 1.0 / (sqrt(var) + eps);"),
    # beta scaled by gamma (the affine step applied before the shift)
    "ln_beta_scaled": ("o[i] = round_to(gamma[i] * (row[i] - mean) * inv + beta[i], round_mode);",
                       "o[i] = round_to(gamma[i] * ((row[i] - mean) * inv + beta[i]), round_mode);"),
    # prefix block selection counted from the last block (Table IV: the first b)
    "prefix_from_end": ("shr |= 1ull << (prefix_blocks ? r : uorder[r]);",
                        "shr |= 1ull << (prefix_blocks ? B - 1 - r : uorder[r]);"),
    # prefix switch ignored (prototype TopK always)
    "prefix_ignored": ("shr |= 1ull << (prefix_blocks ? r : uorder[r]);",
                       "shr |= 1ull << uorder[r];"),
    # router bias left out of the logits
    "bias_dropped": ("z[j] = acc + (bias ? bias[j] : 0.0);", "z[j] = acc;"),
    # router bias added to the neighbouring column
    "bias_wrong_column": ("z[j] = acc + (bias ? bias[j] : 0.0);",
                          "z[j] = acc + (bias ? bias[(j + 1) % (K + 1)] : 0.0);"),
    # margin (ii) measured from the top priority instead of the b-th
    "margin_ii_wrong_rank": ("u[uorder[b - 1]] - u[uorder[b]]", "u[uorder[0]] - u[uorder[b]]"),
    # margin (iii) with P_k in place of P_{k-1} on the lower side
    "margin_iii_prefix": ("for (int i = 0; i < k - 1; ++i) prev += p[i];",
                          "for (int i = 0; i < k; ++i) prev += p[i];"),
    # margin (iii) one-sided (only the distance above beta)
    "margin_iii_one_sided": ("mg[2] = fmin(P_k - beta, beta - prev);", "mg[2] = P_k - beta;"),
    # training: GeLU derivative without the v phi(v) term
    "gelu_grad_phi_only": ("return 0.5 * (1.0 + erf(v * M_SQRT1_2)) + v * exp(-0.5 * v * v) / sqrt(2.0 * M_PI);",
                           "return 0.5 * (1.0 + erf(v * M_SQRT1_2));"),
    # sigmoid derivative without the (1 - sigma) factor
    "dalpha_sigmoid": ("dw[0] * (1.0 - 2.0 * tau) * sg * (1.0 - sg)", "dw[0] * (1.0 - 2.0 * tau) * sg"),
    # the (1 - 2 tau) scale of Eq. 18 left out of the chain rule
    "dalpha_scale": ("dw[0] * (1.0 - 2.0 * tau) * sg * (1.0 - sg)", "dw[0] * sg * (1.0 - sg)"),
    # softmax Jacobian without the mean term
    "softmax_jacobian": ("dzt[1 + j] = s[j] * (dw[1 + j] - dot);", "dzt[1 + j] = s[j] * dw[1 + j];"),
    # value gradient with the pre-activation instead of GeLU of it
    "dv_preactivation": ("const double wg = w * gelu(a);", "const double wg = w * a;"),
    # key gradient without the pathway weight
    "dk_unweighted": ("      const double da = w * gv * gelu_grad(a);\n      const double wg",
                      "      const double da = gv * gelu_grad(a);\n      const double wg"),
    # router gradient to x through the transposed router matrix
    "dx_router_transposed": ("dxt[i] += dzt[c] * w_router[(size_t)i * K1 + c];",
                             "dxt[i] += dzt[c] * w_router[(size_t)c * d + i];"),
    # Gram regulariser gradient without the factor 2
    "gram_grad_half": ("2.0 * g / L : 0.0", "g / L : 0.0"),
    # Gram matrix without the identity subtracted
    "gram_no_identity": ("A[a * K1 + b] = g - (a == b ? 1.0 : 0.0);", "A[a * K1 + b] = g;"),
}

# Mistakes planted in the Python side of the oracle: (file, old, new).
PY_MUTANTS = {
    # given experts listed by increasing affinity
    "with_decisions_ascending": ("__init__.py", "sel.sort(key=lambda j: (-r.s[t, j], j))",
                                 "sel.sort(key=lambda j: (r.s[t, j], j))"),
    # the unselected experts placed first, so the first k are the wrong ones
    "with_decisions_rest_first": ("__init__.py", "order = sel + rest", "order = rest + sel"),
    # affinities left in expert order instead of following q
    "with_decisions_p_unsorted": ("__init__.py", "p[t] = r.s[t, order]", "p[t] = r.s[t]"),
    # the shared set with a strict threshold
    "diag_strict_threshold": ("diagnostics.py", "S[i, j] = c >= delta", "S[i, j] = c > delta"),
    # residual order by increasing score
    "diag_order_ascending": ("diagnostics.py", "np.argsort(-(xa @ _f64(w_res))",
                             "np.argsort((xa @ _f64(w_res))"),
    # residual outputs taken from the shared positions
    "diag_residual_rows": ("diagnostics.py", "ER = E - ES", "ER = ES"),
    # error relative to the residual target instead of the original output
    "diag_error_scale": ("diagnostics.py", "ynorm = max(np.linalg.norm(y[t]), 1e-12)",
                         "ynorm = max(np.linalg.norm(r[t]), 1e-12)"),
    # ridge weight without the 1/m
    "diag_gamma_scale": ("diagnostics.py", "1e-6 * tr / m * np.eye(m)", "1e-6 * tr * np.eye(m)"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, "mutation anchor not found: " + name
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src.replace(old, new))
    lib = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O2", "-ffp-contract=off", "-fopenmp", "-shared", "-fPIC", "-o",
                    str(lib), str(mutated), "-lm"], check=True)
    env = dict(os.environ, UNIF_MOE_ORACLE_LIB=str(lib), OMP_NUM_THREADS="2")
    res = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                          os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                         cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert res.returncode != 0, "no pin caught mutant %s:\n%s" % (name, res.stdout[-2000:])


def run_pins_in_copy(tmp_path, fname, old, new):
    """Runs the pins in a tree of their own holding a copy of the oracle
    package whose Python file `fname` has `old` replaced by `new`."""
    (tmp_path / "oracle").mkdir()
    for f in os.listdir(os.path.join(ROOT, "oracle")):
        if f.endswith((".py", ".c")):
            shutil.copy(os.path.join(ROOT, "oracle", f), tmp_path / "oracle" / f)
    src = open(os.path.join(ROOT, "oracle", fname)).read()
    assert src.count(old) == 1, "mutation anchor not found: " + old
    (tmp_path / "oracle" / fname).write_text(src.replace(old, new))
    (tmp_path / "tests").mkdir()
    for f in ("conftest.py", "test_oracle_pins.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), tmp_path / "tests" / f)
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), tmp_path / "tests" / "golden")
    env = dict(os.environ, OMP_NUM_THREADS="2")
    env.pop("UNIF_MOE_ORACLE_LIB", None)
    return subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                           str(tmp_path / "tests" / "test_oracle_pins.py")],
                          cwd=str(tmp_path), env=env, capture_output=True, text=True, timeout=600)


def test_unmutated_copy_passes(tmp_path):
    """Control for the Python mutants: the copied tree itself passes, so a
    mutant's failure comes from its planted mistake."""
    res = run_pins_in_copy(tmp_path, "__init__.py", "order = sel + rest", "order = sel + rest")
    assert res.returncode == 0, res.stdout[-2000:]


@pytest.mark.parametrize("name", sorted(PY_MUTANTS))
def test_pins_catch_python_mutant(name, tmp_path):
    """The same check for the Python wrapper: a copy of the oracle package
    with one planted mistake, next to copies of the pins."""
    fname, old, new = PY_MUTANTS[name]
    res = run_pins_in_copy(tmp_path, fname, old, new)
    assert res.returncode != 0, "no pin caught mutant %s:\n%s" % (name, res.stdout[-2000:])
