"""The library's host-side greedy replication against the oracle (no GPU needed)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import build as BUILD
from tests.test_offline_pins import _random_replication_case


@pytest.fixture(scope="module", autouse=True)
def lib():
    BUILD.build()
    B.lib()


@pytest.mark.parametrize("seed", range(8))
def test_library_replication_equals_oracle(seed):
    cfg, om, tables, lam, rho, size, cap, place = _random_replication_case(seed, N=4, E=6, M=5)
    want, n_want = O.replicate(om, lam, rho, size, cap, place)
    got, n_got = B.trimmoe_replicate(lam, rho, tables["trans"], size, cap, place)
    assert np.array_equal(got, want) and n_got == n_want


def test_library_replication_rejects_uncovered_expert():
    cfg, om, tables, lam, rho, size, cap, place = _random_replication_case(0)
    place = place.copy()
    place[1, 2] = 0
    with pytest.raises(B.TrimmoeError) as ei:
        B.trimmoe_replicate(lam, rho, tables["trans"], size, cap, place)
    assert ei.value.status == -5
