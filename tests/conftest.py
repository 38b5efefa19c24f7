import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_sessionfinish(session, exitstatus):
    mod = sys.modules.get("_oracle_pool")
    if mod is not None:
        mod.shutdown()


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Per configuration: images whose GPU selection was checked against the oracle, how many
    matched the oracle's pick order exactly, and the sub-margin steps (oracle margin <= 1e-4,
    where either near-best token is valid) met on the way."""
    mod = sys.modules.get("_oracle_pool")
    if mod is None or not mod.SELECTION_STATS:
        return
    tr = terminalreporter
    tr.section("selection parity against the oracle")
    tr.write_line(f"{'configuration':58s} {'images':>6s} {'identical':>9s} {'w/ sub-margin':>13s} "
                  f"{'sub-margin steps':>16s} {'max score rel err':>17s}")
    for label, n, ident, with_sub, steps, err in mod.SELECTION_STATS:
        e = "" if err is None else f"{err:.2e}"
        tr.write_line(f"{label:58s} {n:6d} {ident:9d} {with_sub:13d} {steps:16d} {e:>17s}")
