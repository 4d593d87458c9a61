import sys
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parent.parent
if str(ROOT) not in sys.path:
    sys.path.insert(0, str(ROOT))


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built libarckv.so")


@pytest.fixture(scope="session")
def lib():
    """Build (if needed) and load libarckv.so; loading needs no GPU."""
    from paper_2609_36835_gb300 import _build
    _build.build()
    import paper_2609_36835_gb300 as pk
    return pk.load_library()


# Figures the GPU parity tests record for the end-of-run summary: the widest
# anchor tie gap each test accepted, and the end-to-end held-out output error
# of the call a user makes (its own anchors and assignment), with the number of
# keys whose assignment differs from the oracle's (-1: the anchor sets differ).
PARITY_REPORT = []


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    if not PARITY_REPORT:
        return
    terminalreporter.write_sep("-", "parity figures (widest accepted anchor gap relative to the t-th score; "
                                    "end-to-end held-out output error)")
    widest = max(r["gap"] for r in PARITY_REPORT)
    agreed = [r["o_err"] for r in PARITY_REPORT if r["ties"] == 0]
    worst_o = max(agreed) if agreed else float("nan")
    for r in PARITY_REPORT:
        terminalreporter.write_line(
            "%-58s h=%-2d exch=%-3d gap=%.2e o_e2e=%.2e assign_diff=%d unassisted=%s"
            % (r["test"][:58], r["head"], r["exch"], r["gap"], r["o_err"], r["ties"], r["outputs"]))
    terminalreporter.write_line("widest accepted anchor gap %.3e (band 1e-5, widening capped at 2e-5); worst "
                                "end-to-end held-out error where decisions agree %.3e (bound 2e-3); %d of %d "
                                "sampled heads agree on every decision" % (widest, worst_o, len(agreed),
                                                                           len(PARITY_REPORT)))
