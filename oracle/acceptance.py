"""Acceptance rules of one speculative step (oracle side).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Sec. 3.1: the verifier keeps candidates while they agree with the target and
emits the target's own token at the first disagreement, or a bonus token when
all candidates agree.  For sampling at temperature T>0 a candidate drawn from
q_i is accepted with probability min(1, p_i(c)/q_i(c)); at the first rejection
the token is redrawn from the normalised residual (p_i - q_i)_+, and after a
fully accepted block a bonus is drawn from the target.  App. A.1: an accepted
EOS ends the transcript with no bonus.  App. A.4: draft and target logits get
the same temperature and suppression, and softmax and acceptance arithmetic is
FP32.

Index convention: candidate i (1-based, i = 1..k) is checked against target
row i-1 of the verify block [anchor, c_1, ..., c_k]; row k gives the bonus.
"""
from __future__ import annotations

import itertools

import numpy as np


# ---------------------------------------------------------------- greedy ----
def greedy_accept(candidates, target_argmax, eos_id: int):
    """Greedy verification of one block.

    candidates:    the k live candidates c_1..c_k
    target_argmax: argmax of the target logits at rows 0..k
    Returns (emitted tokens, a = number of accepted candidates, stopped)."""
    k = len(candidates)
    emitted = []
    for i in range(k):
        c = int(candidates[i])
        if c != int(target_argmax[i]):
            break
        emitted.append(c)
        if c == eos_id:                      # accepted EOS: no bonus (App. A.1)
            return emitted, i + 1, True
    a = len(emitted)
    last = int(target_argmax[a])             # correction (a < k) or bonus (a == k)
    emitted.append(last)
    return emitted, a, last == eos_id


# -------------------------------------------------------------- sampling ----
def scaled_logits_fp32(z, temperature: float, suppress=None) -> np.ndarray:
    """z / T in FP32 with suppressed ids at -inf (App. A.4)."""
    x = np.asarray(z, dtype=np.float32) / np.float32(temperature)
    if suppress is not None:
        x = np.where(suppress, np.float32(-np.inf), x)
    return x.astype(np.float32)


def log_sum_exp_fp32(x) -> np.float32:
    x = np.asarray(x, dtype=np.float32)
    m = x.max()
    return np.float32(m + np.log(np.exp(x - m, dtype=np.float32).sum(dtype=np.float32)))


def probs_fp32(x) -> np.ndarray:
    """softmax in FP32 as exp(x - logsumexp(x))."""
    x = np.asarray(x, dtype=np.float32)
    return np.exp(x - log_sum_exp_fp32(x), dtype=np.float32)


def acceptance_probability(p, q, c: int) -> float:
    """min(1, p(c) / q(c)) for a candidate c drawn from q (Sec. 3.1)."""
    return min(1.0, float(p[c]) / float(q[c]))


def residual_distribution(p, q) -> np.ndarray:
    """The normalised residual (p - q)_+ (Sec. 3.1).  If it is empty (possible
    only through rounding, never in exact arithmetic) the target p is used."""
    r = np.maximum(np.asarray(p, dtype=np.float64) - np.asarray(q, dtype=np.float64), 0.0)
    s = r.sum()
    return r / s if s > 0 else np.asarray(p, dtype=np.float64) / np.sum(p)


def gumbel_argmax(x, noise) -> int:
    """A draw from softmax(x) by the Gumbel-max trick: argmax_v (x_v + G_v);
    the lowest id wins ties."""
    return int(np.argmax(np.asarray(x, np.float32) + np.asarray(noise, np.float32)))


def rejection_accept(xt, xd, candidates, coins, residual_noise, bonus_noise, eos_id: int):
    """Speculative rejection sampling over one block, in FP32 (Sec. 3.1, App. A.4).

    xt: target logits / T at rows 0..k            [k+1, V] float32
    xd: draft logits / T at mask positions 1..k    [k, V]  float32
    candidates: c_1..c_k drawn from softmax(xd[i-1])
    coins: accept uniforms u_1..u_k in [0, 1)
    residual_noise: Gumbel noise per row for the residual redraw [k, V]
    bonus_noise: Gumbel noise for the bonus draw from row k       [V]
    Returns (emitted tokens, a, stopped)."""
    k = len(candidates)
    emitted = []
    for i in range(k):
        c = int(candidates[i])
        lse_t = log_sum_exp_fp32(xt[i])
        lse_d = log_sum_exp_fp32(xd[i])
        p_c = np.exp(np.float32(xt[i][c]) - lse_t, dtype=np.float32)
        q_c = np.exp(np.float32(xd[i][c]) - lse_d, dtype=np.float32)
        if np.float32(coins[i]) < np.float32(p_c / q_c):
            emitted.append(c)
            if c == eos_id:
                return emitted, i + 1, True
            continue
        p = np.exp(xt[i] - lse_t, dtype=np.float32)
        q = np.exp(xd[i] - lse_d, dtype=np.float32)
        r = np.maximum(p - q, np.float32(0.0))
        if r.sum(dtype=np.float32) > 0:
            with np.errstate(divide="ignore"):
                score = np.where(r > 0, np.log(r, dtype=np.float32), np.float32(-np.inf))
        else:
            score = xt[i]
        t = gumbel_argmax(score, residual_noise[i])
        emitted.append(t)
        return emitted, i, t == eos_id
    t = gumbel_argmax(xt[k], bonus_noise)
    emitted.append(t)
    return emitted, k, t == eos_id


# ------------------------------------------------- exact enumeration (toy) ---
def step_outcome_distribution(target_conditional, q_rows, k: int, vocab: int) -> dict:
    """Exact distribution of the tokens one rejection-sampling step emits.

    target_conditional(prefix tuple) -> p(. | prefix) over `vocab` ids
    q_rows: draft distributions q_1..q_k (each independent of the other
            candidates, as the parallel drafter samples every mask position
            independently, App. A.4)
    Returns {emitted tuple: probability}, enumerating every candidate tuple."""
    out: dict = {}
    for cand in itertools.product(range(vocab), repeat=k):
        w = 1.0
        for i, c in enumerate(cand):
            w *= float(q_rows[i][c])
        if w == 0.0:
            continue
        reach = w
        prefix: tuple = ()
        for i, c in enumerate(cand):
            p = target_conditional(prefix)
            acc = acceptance_probability(p, q_rows[i], c)
            rej = reach * (1.0 - acc)
            if rej > 0:
                r = residual_distribution(p, q_rows[i])
                for t in range(vocab):
                    if r[t] > 0:
                        key = prefix + (t,)
                        out[key] = out.get(key, 0.0) + rej * r[t]
            reach *= acc
            prefix = prefix + (c,)
            if reach == 0.0:
                break
        if reach > 0:
            p = target_conditional(prefix)
            for t in range(vocab):
                if p[t] > 0:
                    key = prefix + (t,)
                    out[key] = out.get(key, 0.0) + reach * float(p[t])
    return out
