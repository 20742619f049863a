import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build()
    return oracle


def pytest_sessionfinish(session, exitstatus):
    """Renders the parity report (JSON lines appended by the GPU parity
    comparisons when UNIF_MOE_PARITY_REPORT names a file) as a Markdown table
    next to it."""
    path = os.environ.get("UNIF_MOE_PARITY_REPORT")
    if not path or not os.path.exists(path):
        return
    import json
    rows = [json.loads(l) for l in open(path) if l.strip()]

    def hist(h):
        return " ".join("%s:%s" % (k, v) for k, v in sorted(h.items(), key=lambda kv: int(kv[0])))

    out = ["| test | workload | thresholds | tokens (valid) | near-ties <= 1e-3 (i/ii/iii/iv) "
           "| margin <= 1e-5 | decisions differ (near / clear) | max rel err (tol) | mean C_B |",
           "|---|---|---|---|---|---|---|---|---|"]
    for r in rows:
        th = ", ".join("%s=%s" % (k, v) for k, v in r["thresholds"].items() if v)
        test = r["test"].split("::")[-1] + (" [%s]" % r["label"] if r["label"] else "")
        nb = r["near_by_margin"]
        out.append("| %s | %s d=%d H=%d K=%d B=%d %s | %s | %d (%d) | %d (%s) | %d | %d (%d / %d) "
                   "| %.2e (%.0e) | %.2f |"
                   % (test, r["workload"], r["d"], r["H"], r["K"], r["B"], r["dtype"],
                      th or "adaptive", r["n_tokens"], r["n_valid"], r["n_near"],
                      "/".join(str(v) for v in nb), r["n_margin_below_1e5"], r["n_mismatch"],
                      r["n_mismatch"] - r["n_mismatch_clear"], r["n_mismatch_clear"],
                      r["max_rel"], r["tol"], r["mean_cb"]))
    out += ["", "Decision histograms (GPU counts, valid tokens; value:count):", ""]
    for r in rows:
        test = r["test"].split("::")[-1] + (" [%s]" % r["label"] if r["label"] else "")
        out.append("- %s: b {%s}; k {%s}; C_B {%s}" % (test, hist(r["hist_b"]), hist(r["hist_k"]),
                                                       hist(r["hist_cb"])))
    with open(path + ".md", "w") as f:
        f.write("\n".join(out) + "\n")
