"""Pins for the oracle's R1 (logsumexp and sampled-token log-probability, Eq. 1 factors).

Each case is fixed by mathematics, not by the oracle itself: closed forms,
shift invariance, and an independent brute-force evaluation with math.fsum.
"""

import math

import numpy as np
import pytest

from oracle import token_logprob


@pytest.mark.parametrize("V", [1, 2, 7, 4096, 151936])
def test_uniform_logits_closed_form(V):
    # z = c everywhere: lse = c + log V and every token has log-probability -log V.
    c = 3.25
    z = np.full((2, V), c)
    ids = np.array([0, V - 1])
    logp, lse = token_logprob(z, ids)
    np.testing.assert_allclose(lse, c + math.log(V), rtol=0, atol=1e-12)
    np.testing.assert_allclose(logp, -math.log(V), rtol=0, atol=1e-12)


def test_two_way_closed_form():
    # V = 2: log pi(y) = -log(1 + exp(z_other - z_y)).
    rng = np.random.default_rng(1)
    z = rng.normal(0, 4, size=(50, 2))
    ids = rng.integers(0, 2, size=50)
    logp, _ = token_logprob(z, ids)
    other = z[np.arange(50), 1 - ids]
    mine = z[np.arange(50), ids]
    expect = -np.log1p(np.exp(other - mine))
    np.testing.assert_allclose(logp, expect, rtol=0, atol=1e-13)


def test_one_hot_peak_closed_form():
    # z = K at y, 0 elsewhere: log pi(y) = -log(1 + (V-1) e^{-K}), which tends to 0.
    V = 1000
    for K in (5.0, 20.0, 60.0):
        z = np.zeros((1, V))
        z[0, 17] = K
        logp, _ = token_logprob(z, np.array([17]))
        expect = -math.log1p((V - 1) * math.exp(-K))
        assert abs(logp[0] - expect) < 1e-13
    assert abs(logp[0]) < 1e-20


def test_brute_force_fsum_tiny():
    rng = np.random.default_rng(2)
    for V in (1, 3, 8, 9, 16):
        z = rng.normal(0, 3, size=(4, V))
        ids = rng.integers(0, V, size=4)
        logp, lse = token_logprob(z, ids)
        for t in range(4):
            ref = math.log(math.fsum(math.exp(v) for v in z[t]))
            assert abs(lse[t] - ref) < 1e-13
            assert abs(logp[t] - (z[t, ids[t]] - ref)) < 1e-13


def test_shift_invariance_and_normalisation():
    # log-probabilities are invariant to adding a constant per row, and
    # exp(logp) over all ids of a row sums to one.
    rng = np.random.default_rng(3)
    V = 257
    z = rng.normal(0, 2, size=(3, V))
    all_ids = np.arange(V)
    for t in range(3):
        lp, _ = token_logprob(np.repeat(z[t:t + 1], V, axis=0), all_ids)
        lp2, _ = token_logprob(np.repeat(z[t:t + 1] + 41.5, V, axis=0), all_ids)
        np.testing.assert_allclose(lp, lp2, rtol=0, atol=1e-12)
        assert abs(math.fsum(np.exp(lp)) - 1.0) < 1e-13


def test_large_logits_do_not_overflow():
    z = np.array([[1000.0, 999.0, -1000.0]])
    logp, lse = token_logprob(z, np.array([0]))
    assert abs(lse[0] - (1000.0 + math.log1p(math.exp(-1.0)))) < 1e-12
    assert abs(logp[0] + math.log1p(math.exp(-1.0))) < 1e-13


def test_bad_id_is_nan_and_empty_batch():
    logp, _ = token_logprob(np.zeros((2, 4)), np.array([4, -1]))
    assert np.isnan(logp).all()
    logp, lse = token_logprob(np.zeros((0, 4)), np.zeros(0, dtype=np.int64))
    assert logp.shape == (0,) and lse.shape == (0,)
