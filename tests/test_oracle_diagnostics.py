"""Pins for the oracle's R11 (entropy and KL diagnostics of the reference lag).

Closed forms (uniform rows, two-way rows), Gibbs' inequality, KL(p||p) = 0,
shift invariance and brute force with math.fsum.
"""

import math

import numpy as np

from oracle import token_entropy, token_kl


def test_uniform_and_two_way_closed_forms():
    for V in (1, 2, 5, 4096):
        assert np.allclose(token_entropy(np.full((2, V), 1.7)), math.log(V), atol=1e-12)
    rng = np.random.default_rng(0)
    z = rng.normal(0, 3, size=(40, 2))
    p = 1.0 / (1.0 + np.exp(z[:, 1] - z[:, 0]))
    H = -(p * np.log(p) + (1 - p) * np.log1p(-p))
    np.testing.assert_allclose(token_entropy(z), H, rtol=0, atol=1e-12)
    zo = rng.normal(0, 3, size=(40, 2))
    q = 1.0 / (1.0 + np.exp(zo[:, 1] - zo[:, 0]))
    KL = q * np.log(q / p) + (1 - q) * np.log((1 - q) / (1 - p))
    np.testing.assert_allclose(token_kl(zo, z), KL, rtol=1e-10, atol=1e-13)


def test_gibbs_identity_and_shift_invariance():
    rng = np.random.default_rng(1)
    z = rng.normal(0, 2, size=(30, 17))
    zo = z + rng.normal(0, 0.5, size=z.shape)
    kl = token_kl(zo, z)
    assert np.all(kl > 0)
    np.testing.assert_allclose(token_kl(z, z), 0.0, atol=1e-14)
    np.testing.assert_allclose(token_kl(zo + 3.0, z - 7.0), kl, atol=1e-12)
    np.testing.assert_allclose(token_entropy(z + 11.0), token_entropy(z), atol=1e-12)
    assert np.all(token_entropy(z) <= math.log(17) + 1e-12)


def test_brute_force_fsum():
    rng = np.random.default_rng(2)
    z = rng.normal(0, 2, size=(3, 9))
    zo = rng.normal(0, 2, size=(3, 9))
    H = token_entropy(z)
    K = token_kl(zo, z)
    for t in range(3):
        den = math.fsum(math.exp(v) for v in z[t])
        p = [math.exp(v) / den for v in z[t]]
        deno = math.fsum(math.exp(v) for v in zo[t])
        q = [math.exp(v) / deno for v in zo[t]]
        assert abs(H[t] + math.fsum(pi * math.log(pi) for pi in p)) < 1e-13
        assert abs(K[t] - math.fsum(qi * math.log(qi / pi) for qi, pi in zip(q, p))) < 1e-13
