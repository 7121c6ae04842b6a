"""The fp64 oracle against values fixed by the paper and by mathematics (CPU)."""
import pytest

import oracle_pins as P
from oracle import meqmuon as O


@pytest.mark.parametrize("check", P.ALL_CHECKS, ids=lambda f: f.__name__)
def test_oracle_pin(check):
    if check is P.check_ns_exact_integer:
        pytest.importorskip("mpmath")
    check(O)


def test_state_memory_table5():
    P.check_state_memory_table()


def test_llama_hidden_sets_match_paper_counts():
    """The llama130m / llama350m workloads are the paper's hidden sets: their
    element counts equal N_h of Llama-130M / Llama-350M (Table 11)."""
    from paper_2609_35701_gb300 import workloads as W
    g = P.golden()["architecture"]
    for wl, arch in (("llama130m", "Llama-130M"), ("llama350m", "Llama-350M")):
        Nh, Rh = P.llama_hidden_counts(g[arch])
        w = W.get_workload(wl)
        assert w.numel == Nh
        assert sum(r for _, r, _ in w.shapes) == Rh
