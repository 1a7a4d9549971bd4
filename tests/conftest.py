import functools
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 and the CUDA library")


@functools.lru_cache(maxsize=None)
def cached_blob(model_name: str, seed: int, gamma_range=None):
    from paper_2306_04235_gb300 import synth
    return synth.build_blob(synth.MODELS[model_name], seed, gamma_range=gamma_range)
