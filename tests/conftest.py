import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (sm_103a) and the built library")


def _oracle_from_source(src):
    """A private copy of the oracle package compiled from another oracle.c (the mutation
    test of the oracle's pins plants mistakes in a copy; oracle.h must sit beside it)."""
    import importlib.util

    spec = importlib.util.spec_from_file_location("oracle_variant", os.path.join(ROOT, "oracle", "__init__.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    here = os.path.dirname(os.path.abspath(src))
    mod._HERE, mod._SRC, mod._LIB_PATH = here, os.path.abspath(src), os.path.join(here, "liboracle.so")
    mod.build(force=True)
    return mod


@pytest.fixture(scope="session")
def orc():
    src = os.environ.get("TDA_ORACLE_SOURCE")
    if src:
        return _oracle_from_source(src)
    import oracle

    oracle.build()
    return oracle
