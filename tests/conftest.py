import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture
def knobs():
    """Set ISM_* switches for one test.  The library reads them once when it is
    loaded, so each change is followed by ism_debug_reload_env(); the previous
    values are restored (and reloaded) when the test ends."""
    saved = {}

    def reload():
        from paper_2408_00539_gb300 import ism
        ism.load().ism_debug_reload_env()

    def set_knob(name, value):
        if name not in saved:
            saved[name] = os.environ.get(name)
        os.environ[name] = str(value)
        reload()

    yield set_knob
    for name, value in saved.items():
        if value is None:
            os.environ.pop(name, None)
        else:
            os.environ[name] = value
    if saved:
        reload()
