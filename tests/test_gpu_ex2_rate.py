"""refcache_ex2_rate: the exponential unit's rate on this GPU, which the bench
reports as the softmax's secondary limit (one ex2 per visible (query, key)
pair of one head).  The probe must report a plausible, repeatable rate: a
whole number of lanes per clock per SM within a factor of two of 32 (the rate
of a sub-partition issuing one warp-wide ex2 every four clocks), and two
calls within 10 % of each other; a NULL output is refused."""
import ctypes

import pytest
import torch

from paper_2608_21229_gb300 import refcache as rcb

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    rcb.load()


def test_ex2_rate_is_plausible_and_repeatable():
    a, b = rcb.ex2_rate(), rcb.ex2_rate()
    assert 16.0 <= a <= 64.0, a
    assert abs(a - b) <= 0.1 * max(a, b), (a, b)
    assert rcb.status() == rcb.OK


def test_ex2_rate_refuses_null_output():
    assert rcb.load().refcache_ex2_rate(None, None) == rcb.ERR_INVALID_ARG
