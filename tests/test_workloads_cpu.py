"""Host checks of the seeded workload generators (no GPU)."""
import numpy as np
import pytest

from paper_2609_36899_gb300.workloads import (COMPOSITIONS, composition_lengths,
                                              composition_workload)


@pytest.mark.parametrize("comp", COMPOSITIONS)
@pytest.mark.parametrize("b", [1, 8, 32, 128])
def test_composition_total_and_floor(comp, b):
    c = 4096
    lens = composition_lengths(b, c, comp)
    assert lens.shape == (b,) and lens.dtype == np.int32
    assert lens.min() >= 16
    if comp == "uniform":
        assert (lens >= c // 2).all() and (lens <= 3 * c // 2).all()
    else:  # B * C tokens up to rounding
        assert abs(int(lens.sum()) - b * c) <= b


def test_composition_shapes():
    b, c = 32, 4096
    assert (composition_lengths(b, c, "equal") == c).all()
    bim = composition_lengths(b, c, "bimodal")
    assert sorted(set(bim.tolist())) == [c // 2, 9 * c // 2]
    assert (bim == 9 * c // 2).sum() == b // 8
    giant = composition_lengths(b, c, "one_giant")
    assert giant.max() == b * c // 2 and (giant == giant.max()).sum() == 1
    logn = composition_lengths(b, c, "lognormal")
    assert logn.max() > 2 * c  # heavy tail


def test_composition_is_seeded_and_workload_fits():
    a = composition_lengths(128, 4096, "lognormal")
    assert (a == composition_lengths(128, 4096, "lognormal")).all()
    assert not (a == composition_lengths(128, 4096, "lognormal", seed=1)).all()
    w = composition_workload(128, 4096, "one_giant")
    assert w.lengths == "fixed" and len(w.length_args) == 128
    assert w.max_len >= max(w.length_args) and w.max_len % w.page_size == 0
    with pytest.raises(ValueError):
        composition_lengths(8, 4096, "nonsense")
