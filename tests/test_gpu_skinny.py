"""The low-latency projections of single-sequence handles (GPU).

A handle whose every step pass has at most 144 token rows can run its
projections with the skinny kernels (WF_OPT_SKINNY, on by default for
single-sequence handles): at most 14 rows (max_batch 1: the anchor and K = 8
proposals) with the whole operand tile resident (wf_skinny.cu), more with the
operand streamed by k-block (wf_skinny_mt.cu).  Checked against the oracle at the Whisper-tiny
and Whisper-large shapes with every LayerNorm's gain and bias drawn on its own:
draft and verify logits within 3e-2, tapped hidden states within 1e-2
relative, tokens and cache lengths equal wherever the deciding margins
exceed 0.05.  Speculative greedy must equal plain greedy token for token on
the same handle (both take the skinny form), and the tcgen05 form of the
same handle must agree with it within the logit tolerance."""
import numpy as np
import pytest

from oracle import acceptance
from oracle.decoder import WhisperFlashOracle
from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu

LOGIT_ATOL = 3e-2
HIDDEN_REL = 1e-2
MARGIN = 0.05


def _margin(row):
    top = np.partition(np.asarray(row, np.float64), -2)[-2:]
    return float(top[1] - top[0])


def _forced(g, t, a, K, V):
    cand = [g[t + j] if t + j < len(g) else 0 for j in range(K)]
    if a < K and t + a < len(g):
        cand[a] = (g[t + a] + 1) % V
    return cand


def _setup(name):
    cfg = getattr(syn, name)
    ws = syn.make_weights(cfg, seed=0, ln_noise=True)
    enc = syn.encoder_output(cfg, 1, seed=7)
    prompt = syn.prompts(cfg, 1, length=4, seed=7)
    return cfg, ws, enc, prompt


@pytest.mark.parametrize("name", ["TINY", pytest.param("LARGE", marks=pytest.mark.slow)])
def test_single_sequence_steps_match_oracle(name):
    import torch
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session
    cfg, ws, enc, prompt = _setup(name)
    K, V, d = cfg.block_k, cfg.vocab, cfg.d_model
    budget = 40
    s = Session(cfg, ws, max_batch=1, keep_logits=True)
    B.wf_set_option(s.h, B.WF_OPT_SKINNY, 1)        # the default here; raises if unsupported
    first = int(s.prefill([0], enc, prompt, np.array([budget], np.int32)).cpu()[0])
    o = WhisperFlashOracle(syn.weights_as_float(ws, np.float64), cfg)
    encf = syn.bf16_bits_to_f32(enc[0]).astype(np.float64)
    seq = o.prefill(encf, prompt[0], budget)
    gseq = o.prefill(encf, prompt[0], budget)
    while len(gseq.emitted) < 24 and not gseq.done:
        o.greedy_step(gseq)
    greedy = gseq.emitted
    seq.anchor = first                          # continue from the GPU's first token
    decisions = 0
    for step, a in enumerate((8, 2, 5)):
        L0, R0 = int(s.state()["len"][0]), int(s.state()["remaining"][0])
        forced = np.array([_forced(greedy, len(seq.emitted), a, K, V)], np.int32)
        toks, cnt = s.step(forced=forced)
        torch.cuda.synchronize()
        dl = s.view(B.WF_VIEW_DRAFT_LOGITS, torch.float32, (K + 1, V)).cpu().numpy()
        vl = s.view(B.WF_VIEW_TARGET_LOGITS, torch.float32, (K + 1, V)).cpu().numpy()
        taps = s.view(B.WF_VIEW_TAPS, torch.bfloat16, (K + 1, cfg.n_taps * d)).float().cpu().numpy()
        rec = o.spec_step(seq, forced=forced[0])
        assert np.abs(dl[1:1 + K] - rec.draft_logits).max() <= LOGIT_ATOL
        assert np.abs(vl[:rec.k + 1] - rec.verify_logits).max() <= LOGIT_ATOL
        rel = (np.linalg.norm(taps[:rec.k + 1] - rec.verify_taps, axis=1)
               / np.linalg.norm(rec.verify_taps, axis=1))
        assert rel.max() <= HIDDEN_REL
        for gr, orow in zip(vl[:rec.k + 1], rec.verify_logits):
            if _margin(orow) > MARGIN:
                assert int(np.argmax(gr)) == int(np.argmax(orow))
                decisions += 1
        # the step's tokens and cache length follow the acceptance rule on
        # the GPU's own verify logits
        k = max(0, min(K, R0 - 1))
        want, acc, _ = acceptance.greedy_accept(forced[0][:k], np.argmax(vl[:k + 1], axis=1), cfg.eos_id)
        got = [int(x) for x in toks.cpu().numpy()[0, :int(cnt.cpu()[0])]]
        assert got == want
        assert int(s.state()["len"][0]) == L0 + 1 + acc
        if got != rec.emitted:                  # a near tie split the two trajectories
            deciding = [_margin(rec.verify_logits[j]) for j in range(min(rec.accepted + 1, rec.k + 1))]
            assert min(deciding) <= MARGIN
            break
    assert decisions >= 5
    assert s.error() == 0
    s.close()


def test_skinny_speculative_equals_plain_greedy():
    """Sec. 3.1: speculative greedy output equals plain greedy output token
    for token; both take the skinny projections on a single-sequence handle."""
    from paper_2609_32869_gb300.session import Session, upload_weights
    cfg, ws, enc, prompt = _setup("TINY")
    K, V = cfg.block_k, cfg.vocab
    dev = upload_weights(ws)
    budget = 60
    g = Session(cfg, dev, max_batch=1)
    ref = [int(g.prefill([0], enc, prompt, np.array([budget], np.int32)).cpu()[0])]
    while True:
        toks, cnt = g.greedy_step()
        c = int(cnt.cpu()[0])
        if c == 0:
            break
        ref.extend(int(x) for x in toks.cpu().numpy()[0, :c])
    g.close()
    assert len(ref) == budget or ref[-1] == cfg.eos_id
    sched = syn.accept_uniform(64, 1, k=K, seed=11)[:, 0]
    for mode in ("forced", "drafter"):
        s = Session(cfg, dev, max_batch=1)
        got = [int(s.prefill([0], enc, prompt, np.array([budget], np.int32)).cpu()[0])]
        it = 0
        while not s.state()["done"][0]:
            forced = None
            if mode == "forced":
                forced = np.array([_forced(ref, len(got), int(sched[it]), K, V)], np.int32)
            toks, cnt = s.step(forced=forced)
            got.extend(int(x) for x in toks.cpu().numpy()[0, :int(cnt.cpu()[0])])
            it += 1
            assert it < 100
        assert got == ref, mode
        assert s.error() == 0
        s.close()


@pytest.mark.parametrize("n", [1, 4], ids=["one-sequence", "batched"])
def test_skinny_and_tcgen05_forms_agree(n):
    """The skinny form (one sequence: the whole operand tile resident; four:
    the operand streamed by k-block) and the tcgen05 form of the same handle
    agree within the logit tolerance; a handle of more than 144 step rows has
    no skinny form."""
    import torch
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session, upload_weights
    cfg, ws, _, _ = _setup("TINY")
    K, V = cfg.block_k, cfg.vocab
    enc = syn.encoder_output(cfg, n, seed=7)
    prompt = syn.prompts(cfg, n, length=4, seed=7)
    dev = upload_weights(ws)
    forced = syn.random_tokens(cfg, (n, K), seed=3)
    out = {}
    for sk in (1, 0):
        s = Session(cfg, dev, max_batch=n, keep_logits=True)
        B.wf_set_option(s.h, B.WF_OPT_SKINNY, sk)
        s.prefill(np.arange(n, dtype=np.int32), enc, prompt, np.full(n, 40, np.int32))
        s.step(forced=forced)
        torch.cuda.synchronize()
        out[sk] = (s.view(B.WF_VIEW_TARGET_LOGITS, torch.float32, (n, K + 1, V)).cpu().numpy(),
                   s.view(B.WF_VIEW_DRAFT_LOGITS, torch.float32, (n, K + 1, V)).cpu().numpy())
        assert s.error() == 0
        s.close()
    assert np.abs(out[1][0] - out[0][0]).max() <= LOGIT_ATOL
    assert np.abs(out[1][1][:, 1:] - out[0][1][:, 1:]).max() <= LOGIT_ATOL
    big = Session(cfg, dev, max_batch=17)
    with pytest.raises(B.WfError):
        B.wf_set_option(big.h, B.WF_OPT_SKINNY, 1)
    big.close()
