import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (a GB300) and the built CUDA library")
    config.addinivalue_line("markers", "slow: long-running case")


@pytest.fixture(scope="session")
def ea_lib():
    """The in-tree CUDA library (built here with nvcc if needed); loading needs no GPU."""
    from paper_2205_14473_gb300 import build as B
    import paper_2205_14473_gb300 as ea

    B.build()
    return ea.lib()


def pytest_terminal_summary(terminalreporter):
    """Totals of the GPU-vs-oracle lockstep comparisons of this session (tests/parity.py)."""
    parity = sys.modules.get("parity")
    runs = getattr(parity, "RUNS", None)
    if not runs:
        return
    tr = terminalreporter
    tr.section("parity: GPU vs oracle, every round")
    width = max(len(r["test"].split("::")[-1]) for r in runs)
    for r in runs:
        tr.write_line(f"{r['test'].split('::')[-1]:<{width}}  d={r['d']:>13,} oracle d={r['d_oracle']:>12,} "
                      f"n={r['n']:>2} rounds={r['rounds']:>4} codes={r['code_positions']:>14,} "
                      f"values={r['values']:>15,} mismatches={r['mismatches']} (within 2 ulp: {r['flagged']})")
    tot = {k: sum(r[k] for r in runs) for k in ("rounds", "code_positions", "values", "scales", "mismatches")}
    tr.write_line(f"total: {len(runs)} lockstep runs, {tot['rounds']:,} rounds, {tot['code_positions']:,} code "
                  f"positions, {tot['scales']:,} scales and {tot['values']:,} state values compared; "
                  f"code mismatches: {tot['mismatches']}")
