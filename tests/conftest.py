import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running oracle or full-size check")


def pytest_terminal_summary(terminalreporter):
    """Print the achieved parity errors of the full-size checks (normwise error against
    its bound, and the elementwise relative error over |ref| >= 1e-2 max|ref|)."""
    try:
        from tests import parity_util
    except Exception:
        return
    if not parity_util.MARGINS:
        return
    tr = terminalreporter
    tr.write_sep("-", "parity margins (normwise err / bound; elementwise rel err, info)")
    by_check = {}
    for (chk, tensor), (err, bound, elem) in sorted(parity_util.MARGINS.items()):
        by_check.setdefault(chk, []).append(f"{tensor} {err:.2e}/{bound:.0e} ({elem:.1e})")
    for chk, parts in by_check.items():
        tr.write_line(f"{chk}: " + ", ".join(parts))
