"""Shared test fixtures.

Markers: ``gpu`` -- needs a CUDA device and the compiled sm_103a library.
Everything unmarked runs on a CPU-only machine.
"""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU and the compiled sm_103a library")


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.lib()
    return oracle


@pytest.fixture(scope="session")
def sdd():
    """The CUDA path through its C-ABI binding.  On a machine with a GPU a missing
    library is an error, never a skip."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_14787_gb300 as pkg
    pkg.load()          # raises if libsdd.so is missing or fails to load
    return pkg
