import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
for p in (ROOT, os.path.dirname(os.path.abspath(__file__))):
    if p not in sys.path:
        sys.path.insert(0, p)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the CUDA library's kernels)")


def pytest_sessionstart(session):
    # Build (or refresh) the in-tree CUDA library and the C oracle before
    # collection; both builds are no-ops when up to date.
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "_pe_build", os.path.join(ROOT, "paper_2609_04875_gb300", "build.py"))
    pe_build = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(pe_build)
    pe_build.build()
    import oracle
    oracle.build()


def pytest_sessionfinish(session, exitstatus):
    # PE_PARITY_REPORT=<file>: the errors of every block the GPU parity tests
    # checked (absolute and normalised by the oracle's size), one JSON object.
    path = os.environ.get("PE_PARITY_REPORT")
    if not path:
        return
    try:
        import gpu_common
    except Exception:
        return
    import json
    with open(path, "w") as f:
        json.dump([{"what": w, **e} for w, e in gpu_common.PARITY_LOG], f, indent=0)
