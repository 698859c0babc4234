import os
import sys
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]
if str(ROOT) not in sys.path:
    sys.path.insert(0, str(ROOT))


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU; runs the CUDA path through the C ABI")


@pytest.fixture(scope="session")
def kvq_lib():
    """Build (if stale) and load libkvq.so; on a GPU machine a failure is an error."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_16248_gb300 import build, kvq
    build.build()
    kvq.lib()
    return kvq
