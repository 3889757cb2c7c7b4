"""The accept kernel's edge cases on the GPU (App. A.1), against the oracle's
acceptance rule.

Four requests decode in one batch with teacher-forced proposals taken from
the GPU's own greedy transcripts, and the end-of-transcript id set to a token
that one transcript emits, so that within two steps:
  - slot 0 accepts the EOS in the middle of its block (no bonus follows);
  - slot 1 (the same request) emits the EOS as its correction token;
  - slot 2 reaches its budget inside a block (k = R - 1 < K live proposals);
  - the batch compacts around the finished slots while slot 3 continues.
Each step's emitted tokens, count, cache length, remaining budget and done
flag must equal, bit for bit, what the oracle's greedy acceptance rule
(oracle.acceptance.greedy_accept, with k = min(K, R - 1)) gives for the
step's proposals and the argmax of the GPU's own verify logits: the rule is
checked exactly, with no near-tie exemption.  (The weights are ten times
wider than the workloads' so that transcripts do not repeat one token; the
forward pass is held to the oracle at the workloads' scale by the other
parity tests.)"""
import numpy as np
import pytest

from oracle import acceptance
from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu


def _forced(g, t, a, K, V):
    cand = [g[t + j] if t + j < len(g) else 0 for j in range(K)]
    if a < K and t + a < len(g):
        cand[a] = (g[t + a] + 1) % V
    return cand


def _gpu_greedy(s, slots, enc, prompt, budgets):
    first = s.prefill(slots, enc, prompt, budgets).cpu().numpy()
    g = {int(sl): [int(first[i])] for i, sl in enumerate(slots)}
    while True:
        toks, cnt = s.greedy_step()
        toks, cnt = toks.cpu().numpy(), cnt.cpu().numpy()
        if cnt.sum() == 0:
            return g
        for sl in g:
            g[sl].extend(int(x) for x in toks[sl, :cnt[sl]])


def test_eos_budget_and_compaction_follow_the_acceptance_rule():
    import torch
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session, upload_weights
    cfg0 = syn.toy_config()
    ws = syn.make_weights(cfg0, seed=3, std=0.2, ln_noise=True)
    dev = upload_weights(ws)
    request = [1, 1, 0, 3]                      # slot -> request
    enc = syn.encoder_output(cfg0, 4, seed=1)[request]
    prompt = syn.prompts(cfg0, 4, length=4, seed=1)[request]
    budgets = np.array([40, 40, 12, 30], np.int32)
    slots = np.arange(4, dtype=np.int32)
    s0 = Session(cfg0, dev, max_batch=4)
    g0 = _gpu_greedy(s0, slots, enc, prompt, budgets)
    s0.close()
    # the end-of-transcript id: a token of request 1's transcript at index 4..7
    # that appears neither earlier there nor in the first 12 tokens of request 0
    idx = next(i for i in range(4, 8) if g0[0][i] not in g0[0][:i] and g0[0][i] not in g0[2][:12])
    eos = g0[0][idx]
    cfg = syn.toy_config(eos_id=eos)
    K, V = cfg.block_k, cfg.vocab
    g = {sl: (seq[:seq.index(eos) + 1] if eos in seq else seq) for sl, seq in g0.items()}
    assert len(g[0]) == idx + 1
    # accept lengths: slot 0 takes the whole block (the EOS is accepted at
    # position idx), slot 1 stops one short of the EOS and then proposes a
    # wrong token (the EOS is the correction), slot 2 accepts everything
    sched = {0: [8], 1: [idx - 2, 0], 2: [8, 8], 3: [5, 2, 8, 0, 6, 3, 8, 1, 4, 7]}

    s = Session(cfg, dev, max_batch=4, keep_logits=True)
    first = s.prefill(slots, enc, prompt, budgets).cpu().numpy()
    assert [int(x) for x in first] == [g[sl][0] for sl in range(4)]
    emitted = {sl: 1 for sl in range(4)}
    gpu_done = np.zeros(4, bool)
    events = set()
    n_active, step = 4, 0
    st = s.state()
    while n_active:
        active = [b for b in range(4) if not gpu_done[b]]     # ascending after compaction
        forced = np.zeros((4, K), np.int32)
        for b in active:
            forced[b] = _forced(g[b], emitted[b], sched[b][step % len(sched[b])], K, V)
        L0, R0 = st["len"].copy(), st["remaining"].copy()
        toks, cnt = s.step(forced=forced)
        toks, cnt = toks.cpu().numpy(), cnt.cpu().numpy()
        vl = s.view(B.WF_VIEW_TARGET_LOGITS, torch.float32, (4 * (K + 1), V)).cpu().numpy()
        st = s.state()
        for b in range(4):
            if gpu_done[b]:                     # finished and compacted away: emits nothing
                assert cnt[b] == 0 and (toks[b] == -1).all()
                continue
            r0 = active.index(b) * (K + 1)
            k = max(0, min(K, int(R0[b]) - 1))
            want, a, stop = acceptance.greedy_accept(forced[b][:k], np.argmax(vl[r0:r0 + k + 1], axis=1), eos)
            assert [int(x) for x in toks[b, :cnt[b]]] == want, (step, b)
            assert (toks[b, cnt[b]:] == -1).all()
            assert st["len"][b] == L0[b] + 1 + a, (step, b)
            assert st["remaining"][b] == R0[b] - len(want)
            assert bool(st["done"][b]) == (stop or R0[b] - len(want) <= 0)
            emitted[b] += len(want)
            if want[-1] == eos and a == len(want):
                events.add("accepted EOS, no bonus")
            if want[-1] == eos and a == len(want) - 1 and a < k:
                events.add("EOS as correction")
            if k < K and st["remaining"][b] == 0:
                events.add("budget ends inside a block")
        gpu_done = st["done"] != 0
        if gpu_done.any():
            n_active = s.compact()
            assert n_active == int((~gpu_done).sum())
            if 0 < n_active < 4:
                events.add("compacted with sequences left")
        step += 1
        assert step < 60
    assert events == {"accepted EOS, no bonus", "EOS as correction", "budget ends inside a block",
                      "compacted with sequences left"}, events
    assert s.error() == 0
    s.close()
