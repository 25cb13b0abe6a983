"""The native bit-width allocator (jab_allocate_bits, host code in libjab.so) against the oracle's
allocate_bits (Eq. 7, App. B "Allocators"): identical widths on random score tables, including tied
scores, for both walks; and its argument checks. No GPU is needed."""
import numpy as np
import pytest

from oracle import jab_oracle as O


@pytest.fixture(scope="module")
def J():
    from paper_2609_34866_gb300 import binding, build
    build.build()
    binding._LIB = None
    return binding


@pytest.mark.parametrize("method", ["greedy", "pareto"])
def test_native_allocator_matches_the_oracle(J, method):
    rng = np.random.default_rng(30)
    widths = [2, 3, 4, 8, 16]
    for trial in range(300):
        L = int(rng.integers(1, 13))
        if trial % 3 == 0:   # small integer scores: ties between layers and dominated widths
            om = rng.integers(0, 4, size=(L, len(widths))).astype(np.float64)
        else:
            om = rng.random((L, len(widths))) ** 3
        n = rng.integers(1, 10_000, size=L)
        avg = float(rng.uniform(2.0, 16.5))
        assert J.jab_allocate_bits(om, widths, n, avg, method) == O.allocate_bits(om, widths, n, avg,
                                                                                   method), trial


def test_native_allocator_rejects_bad_arguments(J):
    om = np.ones((2, 3))
    with pytest.raises(J.JabError):
        J.jab_allocate_bits(om, [2, 4, 8], [10, 10], 1.5)            # below the cheapest allocation
    with pytest.raises(J.JabError):
        J.jab_allocate_bits(om, [2, 8, 4], [10, 10], 4.0)            # widths not increasing
    with pytest.raises(J.JabError):
        J.jab_allocate_bits(np.array([[1.0, np.nan, 0.0]] * 2), [2, 4, 8], [10, 10], 4.0)
    with pytest.raises(J.JabError):
        J.jab_allocate_bits(om, [2, 4, 8], [10, 0], 4.0)             # empty layer
