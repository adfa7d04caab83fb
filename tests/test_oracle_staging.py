"""CPU pins of the oracle's prefix staging gather and its inverse."""
import numpy as np
import pytest

import oracle
from _pins import STAGE_PINS, _staging_case


@pytest.fixture(scope="module")
def orc():
    return oracle.default()


@pytest.mark.parametrize("pin", STAGE_PINS, ids=lambda f: f.__name__)
def test_stage_pin(orc, pin):
    pin(orc)


def test_stage_rejects_bad_layer_range(orc):
    kpool, vpool, table, cl, _, _ = _staging_case(40, [5], 2, 1, 8)
    with pytest.raises(oracle.OracleError):
        orc.prefix_stage(kpool, vpool, table, cl, 1, 3)


def test_stage_rejects_bad_page_index(orc):
    kpool, vpool, table, cl, _, _ = _staging_case(41, [5, 18], 1, 1, 8)
    table = table.copy()
    table[1, 1] = -1
    with pytest.raises(oracle.OracleError, match="block-table"):
        orc.prefix_stage(kpool, vpool, table, cl, 0, 1)
