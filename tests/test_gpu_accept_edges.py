"""The accept kernel's edge cases against the oracle on the GPU (App. A.1).

Four requests decode in one batch with teacher-forced proposals taken from
the oracle's greedy transcripts, and the end-of-transcript id set to a token
that one transcript emits, so that within two steps:
  - slot 0 accepts the EOS in the middle of its block (no bonus follows);
  - slot 1 (the same request) emits the EOS as its correction token;
  - slot 2 reaches its budget inside a block (k = R - 1 < K live proposals);
  - the batch compacts around the finished slots while slot 3 continues.
Every emitted token, count, cache length and done flag must equal the
oracle's wherever the deciding top-2 margins are clear.  The weights are
drawn wider than the workloads' N(0, 0.02) so that transcripts do not repeat
one token; the logits grow with them, so "clear" means above both 0.05 and
twice the largest difference between the GPU's and the oracle's logits on
that sequence's rows (then both sides must take the same argmax).  They are
clear for every event below on these seeds; a closer call only exempts that
sequence from the remaining comparisons."""
import numpy as np
import pytest

from oracle.decoder import WhisperFlashOracle
from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu

MARGIN = 0.05


def _margin(row):
    top = np.partition(np.asarray(row, np.float64), -2)[-2:]
    return float(top[1] - top[0])


def _forced(g, t, a, K, V):
    cand = [g[t + j] if t + j < len(g) else 0 for j in range(K)]
    if a < K and t + a < len(g):
        cand[a] = (g[t + a] + 1) % V
    return cand


def test_eos_budget_and_compaction_match_oracle():
    import torch
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session
    cfg0 = syn.toy_config()
    ws = syn.make_weights(cfg0, seed=3, std=0.2, ln_noise=True)
    wf = syn.weights_as_float(ws)
    enc_all = syn.encoder_output(cfg0, 4, seed=1)
    prompt_all = syn.prompts(cfg0, 4, length=4, seed=1)
    # the end-of-transcript id: the 6th token of request 1's greedy transcript
    o0 = WhisperFlashOracle(wf, cfg0)
    encf1 = syn.bf16_bits_to_f32(enc_all[1]).astype(np.float64)
    eos = int(o0.greedy_decode(encf1, prompt_all[1], 8)[5])
    cfg = syn.toy_config(eos_id=eos)
    K, V = cfg.block_k, cfg.vocab
    o = WhisperFlashOracle(wf, cfg)

    request = [1, 1, 0, 3]                      # slot -> request
    budgets = np.array([40, 40, 12, 30], np.int32)
    sched = {0: [8], 1: [3, 0], 2: [8, 8], 3: [5, 2, 8, 0, 6, 3, 8, 1, 4, 7]}
    enc = enc_all[request]
    prompt = prompt_all[request]
    encf = [syn.bf16_bits_to_f32(enc[b]).astype(np.float64) for b in range(4)]
    greedy = [o.greedy_decode(encf[b], prompt[b], int(budgets[b])) for b in range(4)]
    seqs = [o.prefill(encf[b], prompt[b], int(budgets[b]), seq_id=b) for b in range(4)]
    assert greedy[0][5] == eos and eos not in greedy[2] + greedy[0][:5]

    s = Session(cfg, ws, max_batch=4, keep_logits=True)
    first = s.prefill(np.arange(4, dtype=np.int32), enc, prompt, budgets).cpu().numpy()
    assert list(first) == [sq.emitted[0] for sq in seqs]

    live = set(range(4))                        # sequences still compared token for token
    events = set()
    gpu_done = np.zeros(4, bool)
    max_err = 0.0                               # logit difference relative to the logits' range
    log = []
    n_active, step = 4, 0
    while n_active:
        forced = np.zeros((4, K), np.int32)
        for b in range(4):
            a = sched[b][step % len(sched[b])]
            forced[b] = _forced(greedy[b], len(seqs[b].emitted), a, K, V)
        active = [b for b in range(4) if not gpu_done[b]]   # ascending after compaction
        toks, cnt = s.step(forced=forced)
        toks, cnt = toks.cpu().numpy(), cnt.cpu().numpy()
        vl = s.view(B.WF_VIEW_TARGET_LOGITS, torch.float32, (4 * (K + 1), V)).cpu().numpy()
        st = s.state()
        for b in range(4):
            if gpu_done[b]:                     # finished and compacted away: emits nothing
                assert cnt[b] == 0 and (toks[b] == -1).all()
                continue
            assert 1 <= cnt[b] <= K + 1 and (toks[b, cnt[b]:] == -1).all()
            if b not in live:
                continue
            rec = o.spec_step(seqs[b], forced=forced[b])
            r0 = active.index(b) * (K + 1)
            nd = min(rec.accepted + 1, rec.k + 1)        # rows whose argmax decides the step
            err = float(np.abs(vl[r0:r0 + nd] - rec.verify_logits[:nd]).max())
            max_err = max(max_err, err / float(np.abs(rec.verify_logits[:nd]).max()))
            deciding = [_margin(rec.verify_logits[j]) for j in range(nd)]
            log.append((step, b, rec.k, rec.accepted, rec.emitted, list(toks[b, :cnt[b]]),
                        round(min(deciding), 3), round(err, 4)))
            if min(deciding) <= max(MARGIN, 2 * err):
                live.discard(b)
                continue
            assert list(toks[b, :cnt[b]]) == rec.emitted, log
            assert st["len"][b] == seqs[b].L and bool(st["done"][b]) == seqs[b].done, (step, b)
            assert st["remaining"][b] == seqs[b].remaining
            if rec.emitted[-1] == eos and rec.accepted == len(rec.emitted):
                events.add("accepted EOS, no bonus")
            if rec.emitted[-1] == eos and rec.accepted == len(rec.emitted) - 1 and rec.accepted < rec.k:
                events.add("EOS as correction")
            if rec.k < K and seqs[b].remaining == 0:
                events.add("budget ends inside a block")
        gpu_done = st["done"] != 0
        if gpu_done.any():
            n_active = s.compact()
            assert n_active == int((~gpu_done).sum())
            if len(live) == 4:
                assert n_active == sum(not sq.done for sq in seqs)
            if 0 < n_active < 4:
                events.add("compacted with sequences left")
        step += 1
        assert step < 60
    assert events == {"accepted EOS, no bonus", "EOS as correction", "budget ends inside a block",
                      "compacted with sequences left"}, (events, log)
    assert max_err <= 1e-2, (max_err, log)
    assert s.error() == 0
    s.close()
