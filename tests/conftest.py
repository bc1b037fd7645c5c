import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the libgleam.so kernels)")
    config.addinivalue_line("markers", "slow: full-size workload, minutes of work")


import pytest  # noqa: E402


@pytest.fixture(params=["one-kernel", "three-kernels", "write-through"])
def call_path(request, monkeypatch):
    """Runs a test three times: as the library runs it (a call of at most 64
    chunks and 256 KiB as one single-block kernel, the write-through of likely
    misses in its automatic mode), with every call on the three-launch path
    (hash kernel, cooperative resolve kernel, pack kernel), and with the
    write-through on for every eligible chunk, so that each path meets every
    parity case.  Outputs must not differ."""
    if request.param != "one-kernel":
        from paper_2607_23115_gb300 import binding as B
        from paper_2607_23115_gb300.cache import Cache

        init = Cache.__init__
        what, value = ((B.GLEAM_DEBUG_SMALL_CALLS, 0) if request.param == "three-kernels"
                       else (B.GLEAM_DEBUG_SPECULATE, 1))

        def init_path(self, *args, **kwargs):
            init(self, *args, **kwargs)
            self.debug_set(what, value)

        monkeypatch.setattr(Cache, "__init__", init_path)
    return request.param
