"""Pins of the oracle's decoder, drafter and greedy speculative step.

Toy shapes (d=128, 2 heads, 3 layers, vocabulary 1000, 200 frames) keep the
suite fast; every property below is shape-independent."""
import copy
import json
import os

import numpy as np
import pytest

from oracle import acceptance
from oracle.decoder import WhisperFlashOracle
from paper_2609_32869_gb300 import synthetic as syn

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def toy():
    cfg = syn.toy_config()
    w = syn.weights_as_float(syn.make_weights(cfg, seed=0, std=0.05))
    enc = syn.bf16_bits_to_f32(syn.encoder_output(cfg, 2, seed=1)).astype(np.float64)
    prompt = syn.prompts(cfg, 2, length=4, seed=1)
    return cfg, w, enc, prompt


def test_first_position_attends_to_itself(toy):
    cfg, w, enc, prompt = toy
    o = WhisperFlashOracle(w, cfg)
    seq = o.prefill(enc[0], prompt[0][:1], budget=4)
    assert np.isfinite(seq._prefill_logits).all()


def test_incremental_cache_equals_full_causal_pass(toy):
    cfg, w, enc, prompt = toy
    o = WhisperFlashOracle(w, cfg)
    toks = np.concatenate([prompt[0], syn.random_tokens(cfg, (6,), seed=9)])
    full = o.prefill(enc[0], toks, budget=2)._prefill_logits
    inc = o.prefill(enc[0], toks[:4], budget=50)
    rows = [inc._prefill_logits[-1]]
    for t in toks[4:]:
        inc.anchor = int(t)                     # feed the given tokens, not the argmax
        rows.append(o.greedy_step(inc))
    np.testing.assert_allclose(np.stack(rows)[:-1], full[3:-1], atol=1e-10)
    np.testing.assert_allclose(rows[-1], full[-1], atol=1e-10)


def test_causality(toy):
    cfg, w, enc, prompt = toy
    o = WhisperFlashOracle(w, cfg)
    a = syn.random_tokens(cfg, (8,), seed=4)
    b = a.copy(); b[5:] = (b[5:] + 7) % cfg.vocab
    la = o.prefill(enc[0], a, budget=2)._prefill_logits
    lb = o.prefill(enc[0], b, budget=2)._prefill_logits
    np.testing.assert_allclose(la[:5], lb[:5], atol=1e-12)
    assert not np.allclose(la[5], lb[5])


def test_zero_blocks_copy_the_input_token(toy):
    """With every block's output projections zeroed the residual stream passes
    through unchanged, and the tied head maps a token back onto itself."""
    cfg, w, enc, prompt = toy
    w0 = copy.deepcopy(w)
    w0["target"]["pos_emb"][:] = 0
    for lw in w0["target_layers"]:
        for k in ("out_w", "out_b", "xout_w", "xout_b", "fc2_w", "fc2_b"):
            lw[k][:] = 0
    o = WhisperFlashOracle(w0, cfg)
    toks = syn.random_tokens(cfg, (12,), seed=5)
    logits = o.prefill(enc[0], toks, budget=2)._prefill_logits
    np.testing.assert_array_equal(np.argmax(logits, -1), toks)


def test_identical_frames_make_cross_attention_query_free(toy):
    cfg, w, enc, prompt = toy
    flat = np.broadcast_to(enc[0][:1], enc[0].shape).copy()
    o = WhisperFlashOracle(w, cfg)
    base = o.prefill(flat, prompt[0], budget=2)._prefill_logits
    w2 = copy.deepcopy(w)
    for lw in w2["target_layers"]:
        lw["xq_w"] *= -3.0
        lw["xq_b"] += 1.0
    other = WhisperFlashOracle(w2, cfg).prefill(flat, prompt[0], budget=2)._prefill_logits
    np.testing.assert_allclose(base, other, atol=1e-10)
    # ... but not with real (distinct) frames
    real = o.prefill(enc[0], prompt[0], budget=2)._prefill_logits
    real2 = WhisperFlashOracle(w2, cfg).prefill(enc[0], prompt[0], budget=2)._prefill_logits
    assert not np.allclose(real, real2)


def test_fig1_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "fig1_worked_example.json")))
    ids = g["vocab"]
    tok = lambda xs: [ids[x] for x in xs]
    emitted, a, stop = acceptance.greedy_accept(tok(g["proposals"]),
                                                tok(g["target_greedy_continuation"]) + [0],
                                                eos_id=ids[g["eos"]])
    assert a == g["expected_accepted"]
    assert emitted == tok(g["expected_emitted"])
    assert emitted[-1] == ids[g["expected_next_anchor"]]
    block = tok([g["anchor"]] + g["proposals"])
    assert block[:1 + a] == tok(g["expected_history_extension"])   # rows kept: anchor + accepted
    prefix = tok(g["prefix_before_round"]) + [ids[g["anchor"]]] + emitted
    assert prefix == tok(g["expected_prefix_after_round"])
    assert not stop


def test_greedy_accept_edge_cases():
    eos = 99
    # all agree: k accepted plus a bonus
    assert acceptance.greedy_accept([1, 2, 3], [1, 2, 3, 4], eos) == ([1, 2, 3, 4], 3, False)
    # first wrong: exactly one greedy step
    assert acceptance.greedy_accept([5, 2, 3], [1, 2, 3, 4], eos) == ([1], 0, False)
    # accepted EOS ends the transcript with no bonus (App. A.1)
    assert acceptance.greedy_accept([1, eos, 3], [1, eos, 7, 4], eos) == ([1, eos], 2, True)
    # EOS as the correction also ends it
    assert acceptance.greedy_accept([1, 2], [1, eos, 4], eos) == ([1, eos], 1, True)
    # no live candidate: the anchor alone is verified
    assert acceptance.greedy_accept([], [6], eos) == ([6], 0, False)


def _teacher_forced(g, t, a, K, vocab):
    """Proposals that agree with the greedy continuation g for exactly a tokens."""
    cand = [g[t + j] if t + j < len(g) else 0 for j in range(K)]
    if a < K and t + a < len(g):
        cand[a] = (g[t + a] + 1) % vocab
    return cand


@pytest.mark.parametrize("mode", ["drafter", "forced"])
def test_speculative_greedy_equals_plain_greedy(toy, mode):
    """Sec. 3.1 / Sec. 5.1: the speculative transcript is the greedy one, token
    by token, and the cache/history lengths follow L + 1 + a (App. A.1)."""
    cfg, w, enc, prompt = toy
    o = WhisperFlashOracle(w, cfg)
    budget = 40
    for b in range(2):
        g = o.greedy_decode(enc[b], prompt[b], budget, seq_id=b)
        seq = o.prefill(enc[b], prompt[b], budget, seq_id=b)
        sched = syn.accept_uniform(64, 1, k=cfg.block_k, seed=7 + b)[:, 0]
        s = 0
        while not seq.done:
            L0, n0 = seq.L, len(seq.emitted)
            forced = None
            if mode == "forced":
                forced = _teacher_forced(g, len(seq.emitted), int(sched[s]), cfg.block_k, cfg.vocab)
            rec = o.spec_step(seq, forced=forced)
            assert rec.k == min(cfg.block_k, budget - n0 - 1)
            assert seq.L == L0 + 1 + rec.accepted
            assert seq.hist.shape[0] == seq.L and all(k.shape[0] == seq.L for k in seq.self_k)
            assert seq.L == len(prompt[b]) + len(seq.emitted) - 1   # transcript one ahead
            if mode == "forced":
                assert rec.accepted == min(int(sched[s]), rec.k)
            s += 1
        assert seq.emitted == g
        assert len(g) == budget                  # no EOS here: the budget ends it


def test_speculative_greedy_stops_at_eos_like_greedy(toy):
    cfg, w, enc, prompt = toy
    g0 = WhisperFlashOracle(w, cfg).greedy_decode(enc[0], prompt[0], 30)
    eos = g0[6]                                   # make a token of the transcript the EOS
    cfg2 = syn.toy_config(eos_id=int(eos))
    o = WhisperFlashOracle(w, cfg2)
    g = o.greedy_decode(enc[0], prompt[0], 30)
    assert g[-1] == eos and len(g) <= 7
    for a in (0, 3, 8):
        seq = o.prefill(enc[0], prompt[0], 30)
        while not seq.done:
            o.spec_step(seq, forced=_teacher_forced(g, len(seq.emitted), a, cfg.block_k, cfg.vocab))
        assert seq.emitted == g


def test_budget_reserves_one_slot(toy):
    cfg, w, enc, prompt = toy
    o = WhisperFlashOracle(w, cfg)
    g = o.greedy_decode(enc[0], prompt[0], 6)
    seq = o.prefill(enc[0], prompt[0], 6)          # 1 token emitted, 5 left
    rec = o.spec_step(seq, forced=g[1:] + [0] * 8)
    assert rec.k == 4 and rec.accepted == 4 and len(rec.emitted) == 5
    assert seq.done and seq.emitted == g


def test_drafter_history_visibility_and_bidirectional_block(toy):
    cfg, w, enc, prompt = toy
    o = WhisperFlashOracle(w, cfg)
    seq = o.prefill(enc[0], prompt[0], 20)
    o.spec_step(seq)
    base = o.drafter_pass(seq)
    # the drafter reads history rows < L only: rows past L never exist in the
    # oracle's memory, and changing an earlier row changes the proposals
    s2 = copy.deepcopy(seq)
    s2.hist = s2.hist.copy(); s2.hist[0] += 1.0
    assert not np.allclose(o.drafter_pass(s2), base)
    # RoPE: shifting every text position by a constant changes nothing
    np.testing.assert_allclose(o.drafter_pass(seq, pos_shift=37), base, atol=5e-5)
    # the block is bidirectional: mask position 1 sees later mask positions,
    # so changing m moves every row, including through later copies only
    w2 = copy.deepcopy(w)
    w2["drafter"]["mask_emb"] = w2["drafter"]["mask_emb"] * 1.5
    assert not np.allclose(WhisperFlashOracle(w2, cfg).drafter_pass(seq)[0], base[0])


def _count(shapes):
    return int(sum(np.prod(s) for s in shapes))


class _Recorder(dict):
    def __init__(self, d, log, tag):
        super().__init__(d)
        self._log, self._tag = log, tag

    def __getitem__(self, k):
        self._log.add((self._tag, k))
        return super().__getitem__(k)


def test_drafter_parameter_count_matches_paper(toy):
    """Sec. 3.2 / Table 3: 60.7M trainable drafter parameters (47.5M without the
    cross-attention path, 52.5M without the history projection).  The
    parameters the oracle's drafter actually reads are recorded on the toy
    model and counted at the large shapes."""
    cfg, w, enc, prompt = toy
    log = set()
    w2 = dict(w)
    w2["drafter"] = _Recorder(w["drafter"], log, "d")
    w2["drafter_layers"] = [_Recorder(lw, log, "l") for lw in w["drafter_layers"]]
    o = WhisperFlashOracle(w2, cfg)
    seq = o.prefill(enc[0], prompt[0], 20)
    o.spec_step(seq)
    d, f, nt = 1280, 5120, 5
    layer_shapes = {"ln1_g": (d,), "ln1_b": (d,), "qkv_w": (3 * d, d), "qkv_b": (2 * d,),
                    "out_w": (d, d), "out_b": (d,), "ln2_g": (d,), "ln2_b": (d,),
                    "xq_w": (d, d), "xq_b": (d,), "xkv_w": (2 * d, d), "xkv_b": (d,),
                    "xout_w": (d, d), "xout_b": (d,), "ln3_g": (d,), "ln3_b": (d,),
                    "fc1_w": (f, d), "fc1_b": (f,), "fc2_w": (d, f), "fc2_b": (d,)}
    # (key biases are structurally zero in Whisper: q/v biases only)
    top_shapes = {"proj_w": (d, nt * d), "proj_b": (d,), "hln_g": (d,), "hln_b": (d,),
                  "mask_emb": (d,)}
    used_layer = {k for t, k in log if t == "l"}
    used_top = {k for t, k in log if t == "d"}
    assert used_layer == set(layer_shapes)
    assert used_top == set(top_shapes)
    total = 2 * _count(layer_shapes.values()) + _count(top_shapes.values())
    assert round(total / 1e6, 1) == 60.7
    cross = {"ln2_g", "ln2_b", "xq_w", "xq_b", "xkv_w", "xkv_b", "xout_w", "xout_b"}
    no_audio = total - 2 * _count(layer_shapes[k] for k in cross)
    assert round(no_audio / 1e6, 1) == 47.5
    no_hist = total - _count(top_shapes[k] for k in ("proj_w", "proj_b", "hln_g", "hln_b"))
    assert round(no_hist / 1e6, 1) == 52.5
