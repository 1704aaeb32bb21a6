"""Failure detection without a GPU fault: a bounded device-side wait runs
out and is reported through the device error word, the call returns
cleanly, and the device stays usable (the next call matches the oracle)."""
import pytest

from gpu_cases import AttnCase, assert_attention_close, ensure_built
from paper_2512_21857_gb300 import binding as B

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def test_attention_wait_that_runs_out_is_reported_and_the_device_stays_usable():
    # 16 heads x 8 key splits (clusters of 8 CTAs, 2-3 chunks each): with a
    # bound of one poll, waits for loads and products that take microseconds
    # give up.
    case = AttnCase([64], [2400], 16, 16, 128, seed=55)
    ref, _ = case.run_oracle()
    B.adt_get_device_error()
    try:
        B.adt_testing_set_wait_limit(1)
        case.run_gpu()  # the launch itself succeeds; its outputs are unspecified
    finally:
        B.adt_testing_set_wait_limit(0)
    bits = B.adt_get_device_error()
    assert bits & B.DEVERR_TIMEOUT
    assert B.adt_get_device_error() == 0  # read and cleared
    for _ in range(2):
        got, _, _ = case.run_gpu()
        assert B.adt_get_device_error() == 0
        assert_attention_close(got, ref)
