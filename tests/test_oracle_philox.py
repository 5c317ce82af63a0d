"""Pins the oracle's Philox4x32-10 to the published known-answer vectors."""
import os

import numpy as np

from conftest import GOLDEN


def _kat():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                w = [int(x, 16) for x in line.split()]
                rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_known_answer_vectors(orc):
    rows = _kat()
    assert len(rows) == 3
    for ctr, key, expect in rows:
        got = orc.philox4x32_10(ctr, key)
        assert [int(x) for x in got] == expect


def test_counter_words_all_matter(orc):
    base = orc.philox4x32_10([1, 2, 3, 4], [5, 6])
    for i in range(4):
        c = [1, 2, 3, 4]
        c[i] ^= 1
        assert not np.array_equal(orc.philox4x32_10(c, [5, 6]), base)
    assert not np.array_equal(orc.philox4x32_10([1, 2, 3, 4], [5, 7]), base)
