import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture(scope="session")
def grkv_lib():
    """The CUDA library; GPU tests fail loudly if it cannot be built or loaded."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test run without a CUDA device")
    from paper_2605_31105_gb300 import binding
    return binding.load()


def pytest_terminal_summary(terminalreporter):
    """Retained-set differences seen by the end-to-end GPU checks."""
    mod = sys.modules.get("tests.gpu_cases")
    log = getattr(mod, "SWAP_LOG", None) if mod else None
    if not log:
        return
    tr = terminalreporter
    tr.section("retained-set differences against the oracle (end-to-end units)")
    n_sw = sum(1 for r in log if r["swaps"])
    tr.write_line(f"{len(log)} units compared, {n_sw} with swaps; "
                  f"{sum(1 for r in log if r['max_gap'] > 1e-6)} beyond the 1e-6 tie width")
    for r in log:
        if r["swaps"] or not r["fixed_same"]:
            tr.write_line(f"  {r['workload']} unit {r['unit']}: {r['swaps']} swap(s), largest gap "
                          f"{r['max_gap']:.2e} (bound {r['bound']:.2e}), fixed set "
                          f"{'same' if r['fixed_same'] else 'differs'}, v_out err {r['v_err']:.2e}")
    worst = max(log, key=lambda r: r["v_err"])
    tr.write_line(f"  worst v_out row-relative error {worst['v_err']:.2e} "
                  f"({worst['workload']} unit {worst['unit']})")
