import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: large generated workloads")


_CACHE = {}


@pytest.fixture(scope="session")
def workload():
    """Session cache of generated layers/stacks keyed by shape (generation takes seconds)."""
    import synth

    def get(shape, **kw):
        key = (shape, tuple(sorted(kw.items())))
        if key not in _CACHE:
            if isinstance(shape, synth.StackShape):
                _CACHE[key] = synth.make_stack(shape, **kw)
            else:
                _CACHE[key] = synth.make_layer(shape)
        return _CACHE[key]

    return get
