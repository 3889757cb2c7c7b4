"""Pins of the oracle's Philox4x32-10 and of the draws made from it."""
import numpy as np
import pytest

from oracle import philox


# Known-answer vectors published with the Random123 library for philox4x32_10
# (Salmon et al., SC'11): (counter, key) -> output.
KAT = [
    ((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
    ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
    ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
     (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1)),
]


@pytest.mark.parametrize("ctr,key,expect", KAT)
def test_philox_known_answers(ctr, key, expect):
    out = philox.philox4x32_10(np.array(ctr, np.uint32), np.array(key, np.uint32))
    assert tuple(int(x) for x in out) == expect


def test_uniform_ranges():
    w = np.array([0, 0xFF, 0x100, 0xFFFFFFFF], np.uint32)
    u = philox.word_to_uniform(w)
    assert u[0] == 0.0 and u[1] == 0.0 and u[2] == np.float32(2 ** -24)
    assert u[3] == np.float32(1 - 2 ** -24) and u[3] < 1.0
    uo = philox.word_to_open_uniform(w)
    assert (uo > 0).all() and (uo < 1).all()
    assert uo[3] == np.float32(1 - 2 ** -24) and uo[0] == np.float32(2 ** -24)


def test_gumbel_max_samples_softmax():
    # Gumbel-max: argmax(x + G) is distributed as softmax(x).  Chi-square over 16 ids.
    from scipy.stats import chisquare
    x = np.linspace(-2.0, 1.0, 16).astype(np.float32)
    p = np.exp(x.astype(np.float64) - x.max()); p /= p.sum()
    n = 6000
    counts = np.zeros(16)
    for s in range(n):
        g = philox.gumbel_noise(seed=11, seq=3, step=s, row=1, tag=philox.TAG_DRAFT, vocab=16)
        counts[int(np.argmax(x + g))] += 1
    stat = chisquare(counts, p * n)
    assert stat.pvalue > 1e-3


def test_streams_are_distinct():
    a = philox.gumbel_noise(1, 0, 5, 1, philox.TAG_DRAFT, 64)
    b = philox.gumbel_noise(1, 0, 5, 2, philox.TAG_DRAFT, 64)
    c = philox.gumbel_noise(1, 0, 5, 1, philox.TAG_RESIDUAL, 64)
    d = philox.gumbel_noise(1, 1, 5, 1, philox.TAG_DRAFT, 64)
    assert not np.array_equal(a, b) and not np.array_equal(a, c) and not np.array_equal(a, d)
    np.testing.assert_array_equal(a, philox.gumbel_noise(1, 0, 5, 1, philox.TAG_DRAFT, 64))
