"""CPU pins of the fp64 oracle's decode attention (no GPU needed)."""
import numpy as np
import pytest

import oracle
from _pins import ATTENTION_PINS, _random_batch


@pytest.fixture(scope="module")
def orc():
    return oracle.default()


@pytest.mark.parametrize("pin", ATTENTION_PINS, ids=lambda f: f.__name__)
def test_attention_pin(orc, pin):
    pin(orc)


def test_attention_rejects_bad_page_index(orc):
    q, kp, vp, table, cl, _, _ = _random_batch(30, [20, 5], 2, 1, 64)
    table = table.copy()
    table[1, 0] = kp.shape[0]               # one past the pool
    with pytest.raises(oracle.OracleError, match="block-table"):
        orc.decode_attention(q, kp, vp, table, cl)


def test_attention_rejects_length_beyond_table(orc):
    q, kp, vp, table, cl, _, _ = _random_batch(31, [20, 5], 2, 1, 64)
    cl = cl.copy()
    cl[0] = table.shape[1] * 16 + 1
    with pytest.raises(oracle.OracleError, match="context length"):
        orc.decode_attention(q, kp, vp, table, cl)


def test_attention_thread_count_does_not_change_result(orc):
    q, kp, vp, table, cl, _, _ = _random_batch(32, [300, 17, 64], 8, 2, 64)
    a = orc.decode_attention(q, kp, vp, table, cl, num_threads=1)
    b = orc.decode_attention(q, kp, vp, table, cl, num_threads=4)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])


from _pins import APPEND_PINS  # noqa: E402


@pytest.mark.parametrize("pin", APPEND_PINS, ids=lambda f: f.__name__)
def test_append_pin(orc, pin):
    pin(orc)


from _pins import PREFILL_PINS  # noqa: E402


@pytest.mark.parametrize("pin", PREFILL_PINS, ids=lambda f: f.__name__)
def test_prefill_pin(orc, pin):
    pin(orc)
