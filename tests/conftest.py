import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    # the worst output error of every full-size parity step that ran (shown without -s)
    mod = sys.modules.get("tests.parity")
    lines = getattr(mod, "REPORT", None) if mod else None
    if lines:
        terminalreporter.section("full-size parity")
        for line in lines:
            terminalreporter.write_line(line)
