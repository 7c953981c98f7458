"""Numbers printed in the paper, checked against the library's parameter layout."""
import json
import os

from paper_2606_27748_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "param_overhead.json")


def frequency_params_per_head(variant: str, M: int, d: int) -> int:
    """Size of the per-head frequency tensors the C ABI takes: W1 [M, d] (+ W2 [M, d])."""
    return (1 if variant == "s" else 2) * M * d


def test_parameter_overhead_matches_paper_table():
    g = json.load(open(GOLDEN))
    n = g["n_frequencies"]
    for name, m in g["models"].items():
        for variant, pct in m["rel_increase_pct"].items():
            extra = m["layers"] * m["heads"] * frequency_params_per_head(variant, n,
                                                                         m["head_size"])
            ours = 100.0 * extra / m["total_params"]
            # the table's totals are rounded to 2-3 significant digits (41M, 247M)
            assert abs(ours - pct) <= 0.03 * pct, (name, variant, ours, pct)


def test_workload_frequency_shapes_follow_layout():
    for w in workloads.ORDERED:
        ins = workloads.make_inputs(w.replace(B=1, H=2, N=3))
        assert ins["W1"].shape == (2, w.M, w.d)
        assert (ins["W2"] is None) == (w.variant == "s")
