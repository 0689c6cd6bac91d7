import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) GPU and the CUDA library")


def _load_relations(name):
    rel = {}
    with open(os.path.join(ROOT, "tests", "golden", name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            mode, qb, kb, bit = line.split()
            rel[(mode, qb, kb)] = bool(int(bit))
    return rel


@pytest.fixture(scope="session")
def paper_relations():
    """Block visibility restated from Sec. 3.3, Sec. 3.2 and Sec. 4.1 (golden text)."""
    rel = _load_relations("mask_sec3_3.txt")
    rel.update(_load_relations("mask_alt_reading.txt"))
    return rel


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle

    oracle.build()
    return oracle
