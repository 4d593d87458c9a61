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
