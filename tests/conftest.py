import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_terminal_summary(terminalreporter):
    """The largest O and score errors against the oracle, per parity test."""
    mod = sys.modules.get("parity_utils")
    errors = getattr(mod, "ERRORS", None) if mod else None
    if not errors:
        return
    tr = terminalreporter
    tr.section("parity: largest errors against the fp64 oracle (O bar 2e-2, scores 1e-5)")
    for name in sorted(errors):
        o, s = errors[name]
        tr.write_line(f"{o:10.3e} {s:10.3e}  {name}")
    tr.write_line(f"max over all: O {max(e[0] for e in errors.values()):.3e}, "
                  f"scores {max(e[1] for e in errors.values()):.3e}")
