import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built library")
    config.addinivalue_line("markers", "slow: long-running CPU test")


@pytest.fixture(scope="session")
def golden_dir():
    return os.path.join(ROOT, "tests", "golden")


def pytest_terminal_summary(terminalreporter):
    """Prints the output errors every GPU parity test recorded (max-norm relative
    error and the elementwise 99.9th percentile, both over max|oracle|), and
    writes them as JSON to $SR_PARITY_REPORT when that is set."""
    from tests._helpers import PARITY_RECORDS
    if not PARITY_RECORDS:
        return
    tr = terminalreporter
    tr.write_sep("-", "output parity against the fp64 oracle")
    tr.write_line(f"{'case':58s} {'max-norm':>10s} {'p99.9':>10s} {'bar':>7s} {'elements':>11s}")
    for case, err, p999, tol, n, note in PARITY_RECORDS:
        tr.write_line(f"{case:58s} {err:10.3e} {p999:10.3e} {tol:7.0e} {n:11d}  {note}")
    path = os.environ.get("SR_PARITY_REPORT")
    if path:
        import json
        with open(path, "w") as f:
            json.dump([{"case": c, "max_norm_rel": e, "p999_rel": p, "bar": t, "elements": n,
                        "note": nt} for c, e, p, t, n, nt in PARITY_RECORDS], f, indent=1)
