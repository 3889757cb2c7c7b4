"""Pins of the speculative rejection-sampling rule (Sec. 3.1, App. A.4).

The rule must leave the target's distribution unchanged in exact arithmetic.
A 16-token toy vocabulary with prefix-dependent target conditionals and
position-wise independent draft distributions lets every outcome be
enumerated."""
import itertools

import numpy as np
import pytest

from oracle import acceptance, philox

V = 16


def _table(seed, n_rows):
    rng = np.random.default_rng(seed)
    z = rng.normal(0.0, 1.5, size=(n_rows, V))
    z[:, 3] -= 30.0          # one token the target almost never produces
    p = np.exp(z - z.max(1, keepdims=True))
    return p / p.sum(1, keepdims=True)


def _target_conditional_factory(seed):
    table = _table(seed, 4096)

    def cond(prefix):
        h = 0
        for t in prefix:
            h = (h * 31 + t + 1) % 4096
        return table[h]
    return cond


def _target_joint(cond, n):
    out = {}
    for seq in itertools.product(range(V), repeat=n):
        pr = 1.0
        for i in range(n):
            pr *= cond(seq[:i])[seq[i]]
        out[seq] = pr
    return out


def _complete(outcomes, cond, n):
    """Extend each emitted prefix to n tokens with exact target conditionals."""
    joint = {}

    def rec(prefix, w):
        if len(prefix) == n:
            joint[prefix] = joint.get(prefix, 0.0) + w
            return
        p = cond(prefix)
        for t in range(V):
            if p[t] > 0:
                rec(prefix + (t,), w * p[t])
    for em, w in outcomes.items():
        if len(em) >= n:
            joint[em[:n]] = joint.get(em[:n], 0.0) + w
        else:
            rec(em, w)
    return joint


@pytest.mark.parametrize("k,seed", [(1, 0), (2, 1), (3, 2)])
def test_rejection_rule_preserves_target_distribution_exactly(k, seed):
    cond = _target_conditional_factory(seed)
    q_rows = _table(seed + 100, k)
    q_rows[0, 3] = 0.2                     # drafts the near-impossible token often
    q_rows[0] /= q_rows[0].sum()
    outcomes = acceptance.step_outcome_distribution(cond, q_rows, k, V)
    assert sum(outcomes.values()) == pytest.approx(1.0, abs=1e-12)
    assert all(1 <= len(e) <= k + 1 for e in outcomes)
    got = _complete(outcomes, cond, k + 1)
    want = _target_joint(cond, k + 1)
    err = max(abs(got.get(s, 0.0) - w) for s, w in want.items())
    assert err < 1e-12


def test_residual_is_positive_part_normalised():
    p = np.array([0.5, 0.3, 0.2, 0.0])
    q = np.array([0.1, 0.6, 0.2, 0.1])
    np.testing.assert_allclose(acceptance.residual_distribution(p, q), [1.0, 0, 0, 0])
    assert acceptance.acceptance_probability(p, q, 1) == pytest.approx(0.5)
    assert acceptance.acceptance_probability(p, q, 0) == 1.0


@pytest.mark.parametrize("k", [1, 2])
def test_philox_driven_sampler_matches_target_first_two_tokens(k):
    """The FP32 sampler that the decode step runs (accept coins and Gumbel
    redraws from Philox) reproduces the target's joint of the first two tokens
    (chi-square over 256 cells); with k=1 the second token is the bonus."""
    from scipy.stats import chisquare
    cond = _target_conditional_factory(7)
    zq = np.log(_table(107, k)).astype(np.float32)
    n = 10000
    counts = np.zeros((V, V))
    for trial in range(n):
        seq = trial & 0xFFFFFF
        cands = [acceptance.gumbel_argmax(zq[i], philox.gumbel_noise(5, seq, 1, i + 1,
                 philox.TAG_DRAFT, V)) for i in range(k)]
        xt = np.log(np.stack([cond(tuple(cands[:i])) for i in range(k + 1)])).astype(np.float32)
        coins = [philox.accept_uniform(5, seq, 1, i + 1) for i in range(k)]
        rn = [philox.gumbel_noise(5, seq, 1, i + 1, philox.TAG_RESIDUAL, V) for i in range(k)]
        bn = philox.gumbel_noise(5, seq, 1, k, philox.TAG_BONUS, V)
        em, a, _ = acceptance.rejection_accept(xt, zq, cands, coins, rn, bn, eos_id=-1)
        if len(em) == 1:                       # second token from the target itself
            p = cond((em[0],))
            g = philox.gumbel_noise(5, seq, 2, 0, philox.TAG_BONUS, V)
            em = em + [acceptance.gumbel_argmax(np.log(p).astype(np.float32), g)]
        counts[em[0], em[1]] += 1
    want = np.array([[cond(())[a] * cond((a,))[b] for b in range(V)] for a in range(V)])
    mask = want * n >= 5
    obs = np.append(counts[mask], counts[~mask].sum())
    exp = np.append(want[mask] * n, want[~mask].sum() * n)
    exp *= obs.sum() / exp.sum()
    assert chisquare(obs, exp).pvalue > 1e-3
