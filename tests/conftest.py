import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Report the near-tie rows of every GPU/oracle decision comparison."""
    try:
        from tests.helpers import NEAR_TIES
    except ImportError:
        return
    if not NEAR_TIES:
        return
    tr = terminalreporter
    tr.write_sep("-", "near-ties (rows in the accept / resample band; rows excused)")
    tot = [0, 0, 0, 0]
    for what, rows, ta, tres, exc in NEAR_TIES:
        tr.write_line(f"{what or '?'}: {rows} rows, accept band {ta}, resample band {tres}, "
                      f"excused {exc}")
        for i, x in enumerate((rows, ta, tres, exc)):
            tot[i] += x
    tr.write_line(f"total: {tot[0]} rows, accept band {tot[1]}, resample band {tot[2]}, "
                  f"excused {tot[3]}")
