import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_terminal_summary(terminalreporter):
    # how many weight elements passed only because the tolerance is taken at the scale of
    # the update's operands rather than of the result alone (tests/parity.py)
    mod = sys.modules.get("parity")
    if mod is None or not mod.WEIGHT_TOTALS["compared"]:
        return
    t = mod.WEIGHT_TOTALS
    terminalreporter.write_line(
        f"parity: {t['compared']} weight elements compared with the oracle, {t['differ']} differ, "
        f"{t['widened_only']} of them within 1 ulp / rel 1e-5 only at the operand scale "
        f"(max(|W_oracle|, |W_before|, |U||C||V|^T)), not at |W_oracle| alone")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def read_golden_rows(name):
    """Rows of a whitespace-separated fixture under tests/golden, comments skipped."""
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            rows.append(line.split())
    return rows


@pytest.fixture(scope="session")
def golden():
    return read_golden_rows


def ensure_library():
    """Build libsubzero_zo.so in-tree if it is missing or stale (nvcc cross-compiles on CPU)."""
    from paper_2608_15665_gb300 import build
    return build.build()


def cuda_available():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


@pytest.fixture(scope="session")
def lib():
    ensure_library()
    from paper_2608_15665_gb300 import binding
    return binding


@pytest.fixture(scope="session")
def gpu(lib):
    if not cuda_available():
        pytest.fail("GPU test selected but no CUDA device is visible")
    import torch
    torch.cuda.init()
    return torch.device("cuda:0")
