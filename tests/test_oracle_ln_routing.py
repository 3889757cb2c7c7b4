"""Pins of the oracle's LayerNorm routing and block order.

Every LayerNorm here carries its own non-trivial gain and bias (drawn with
`ln_noise`), so a LayerNorm applied in the wrong place changes the result.

1. A hand check: a 1-layer, 1-head, d=8 decoder (and a 1-layer drafter on
   top of it) evaluated with scalar float64 arithmetic written out from the
   Whisper block's definition (pre-LN: x += SelfAttn(LN1 x); x += CrossAttn(
   LN2 x, A); x += fc2(GELU(fc1(LN3 x))); final LN; tied head) and from the
   drafter's (Sec. 3.2, Eq. 2, App. A.2: history rows LN_h(W_p taps + b_p),
   one softmax over history and block with RoPE, the target's final LN and
   head).  This code shares nothing with the oracle's vectorised numpy.
2. Invariants that follow from pre-LN routing alone: zeroing the gain of one
   LayerNorm makes that sub-layer's input one constant row, so a row's result
   stops depending on the other rows; zeroing gain and bias makes the input
   zero, so the result stops depending on the sub-layer's input weights (and
   only on those); with every block gain zero the blocks add the same vector
   to every row, so residual streams keep their differences exactly.
"""
import copy
import math

import numpy as np
import pytest

from oracle.decoder import WhisperFlashOracle
from paper_2609_32869_gb300 import synthetic as syn


# ----------------------------------------------------------- hand check ----
def _cfg8():
    return syn.toy_config(name="d8", d_model=8, n_heads=1, d_ff=16, n_layers=1, vocab=11,
                          max_pos=16, taps=(0, 0, 0, 0, 0), eos_id=10, enc_frames=5,
                          n_draft_layers=1, block_k=2, rope_base=16.0)


def _rows(a):
    a = np.asarray(a, dtype=np.float64)
    return [list(map(float, r)) for r in a] if a.ndim == 2 else list(map(float, a))


def _ln(v, g, b, eps):
    n = len(v)
    mu = sum(v) / n
    var = sum((x - mu) * (x - mu) for x in v) / n
    r = 1.0 / math.sqrt(var + eps)
    return [(v[i] - mu) * r * g[i] + b[i] for i in range(n)]


def _mv(W, v, b=None):
    out = []
    for o in range(len(W)):
        s = 0.0
        for i in range(len(v)):
            s += W[o][i] * v[i]
        out.append(s + (b[o] if b is not None else 0.0))
    return out


def _add(a, b):
    return [a[i] + b[i] for i in range(len(a))]


def _attend(q, keys, vals):
    dh = len(q)
    s = [sum(q[i] * k[i] for i in range(dh)) / math.sqrt(dh) for k in keys]
    m = max(s)
    e = [math.exp(x - m) for x in s]
    z = sum(e)
    return [sum(e[j] * vals[j][i] for j in range(len(vals))) / z for i in range(dh)]


def _gelu(x):
    return 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0)))


def _rot(v, pos):
    # dims i and i + 4 rotate by pos * 16^(-2i/8) = pos * 2^-i (exact in FP32)
    out = list(v)
    for i in range(4):
        a = pos * 2.0 ** (-i)
        c, s = math.cos(a), math.sin(a)
        out[i] = v[i] * c - v[i + 4] * s
        out[i + 4] = v[i + 4] * c + v[i] * s
    return out


def _block(lw, xs, self_keys, self_vals, key_visible, enc, eps, rope_pos=None, hist=None):
    """One Whisper block over rows xs.  Self-attention keys/values are the
    given cache rows followed by the rows' own; key_visible(i, j) masks."""
    d = len(xs[0])
    W = {k: _rows(v) for k, v in lw.items()}
    Wq, Wk, Wv = W["qkv_w"][:d], W["qkv_w"][d:2 * d], W["qkv_w"][2 * d:]
    bq, bk, bv = W["qkv_b"][:d], W["qkv_b"][d:2 * d], W["qkv_b"][2 * d:]
    hs = [_ln(x, W["ln1_g"], W["ln1_b"], eps) for x in xs]
    qs = [_mv(Wq, h, bq) for h in hs]
    ks = [_mv(Wk, h, bk) for h in hs]
    vs = [_mv(Wv, h, bv) for h in hs]
    if hist is not None:                # drafter: history keys from the layer's own k/v rows
        self_keys = [_mv(Wk, h, bk) for h in hist]
        self_vals = [_mv(Wv, h, bv) for h in hist]
        self_keys = [_rot(k, i) for i, k in enumerate(self_keys)]
        qs = [_rot(q, rope_pos[i]) for i, q in enumerate(qs)]
        ks = [_rot(k, rope_pos[i]) for i, k in enumerate(ks)]
    keys, vals = self_keys + ks, self_vals + vs
    out = []
    for i, x in enumerate(xs):
        vis = [j for j in range(len(keys)) if key_visible(i, j)]
        a = _attend(qs[i], [keys[j] for j in vis], [vals[j] for j in vis])
        out.append(_add(x, _mv(W["out_w"], a, W["out_b"])))
    xs = out
    ck = [_mv(W["xkv_w"][:d], e, W["xkv_b"][:d]) for e in enc]
    cv = [_mv(W["xkv_w"][d:], e, W["xkv_b"][d:]) for e in enc]
    out = []
    for x in xs:
        h = _ln(x, W["ln2_g"], W["ln2_b"], eps)
        a = _attend(_mv(W["xq_w"], h, W["xq_b"]), ck, cv)
        x = _add(x, _mv(W["xout_w"], a, W["xout_b"]))
        h = _ln(x, W["ln3_g"], W["ln3_b"], eps)
        f = [_gelu(t) for t in _mv(W["fc1_w"], h, W["fc1_b"])]
        out.append(_add(x, _mv(W["fc2_w"], f, W["fc2_b"])))
    return out, ks, vs


def _head(wf, x, eps):
    h = _ln(x, _rows(wf["target"]["lnf_g"]), _rows(wf["target"]["lnf_b"]), eps)
    return _mv(_rows(wf["target"]["tok_emb"]), h)


@pytest.fixture(scope="module")
def d8():
    cfg = _cfg8()
    ws = syn.make_weights(cfg, seed=11, std=0.5, ln_noise=True)
    wf = syn.weights_as_float(ws)
    enc = syn.bf16_bits_to_f32(syn.encoder_output(cfg, 1, seed=2)[0]).astype(np.float64)
    prompt = np.array([3, 7, 1], np.int32)
    return cfg, wf, enc, prompt


def _hand_prefill(cfg, wf, enc, prompt):
    eps = cfg.ln_eps
    emb, pos = _rows(wf["target"]["tok_emb"]), _rows(wf["target"]["pos_emb"])
    xs = [_add(emb[t], pos[p]) for p, t in enumerate(prompt)]
    xs, _, _ = _block(wf["target_layers"][0], xs, [], [], lambda i, j: j <= i, _rows(enc), eps)
    return xs, [_head(wf, x, eps) for x in xs]


def test_hand_checked_target_block_d8(d8):
    cfg, wf, enc, prompt = d8
    _, want = _hand_prefill(cfg, wf, enc, prompt)
    got = WhisperFlashOracle(wf, cfg).prefill(enc, prompt, budget=4)._prefill_logits
    np.testing.assert_allclose(got, np.array(want), rtol=0, atol=1e-12)


def test_hand_checked_drafter_d8(d8):
    cfg, wf, enc, prompt = d8
    eps, d, K = cfg.ln_eps, cfg.d_model, cfg.block_k
    taps, _ = _hand_prefill(cfg, wf, enc, prompt)
    dr = wf["drafter"]
    hist = [_ln(_mv(_rows(dr["proj_w"]), t * 5, _rows(dr["proj_b"])), _rows(dr["hln_g"]),
                _rows(dr["hln_b"]), eps) for t in taps]
    o = WhisperFlashOracle(wf, cfg)
    seq = o.prefill(enc, prompt, budget=6)
    L = len(prompt)
    xs = [_rows(wf["target"]["tok_emb"])[seq.anchor]] + [_rows(dr["mask_emb"])] * K
    xs, _, _ = _block(wf["drafter_layers"][0], xs, None, None, lambda i, j: True, _rows(enc), eps,
                      rope_pos=[L + j for j in range(K + 1)], hist=hist)
    want = np.array([_head(wf, x, eps) for x in xs[1:]])
    np.testing.assert_allclose(o.drafter_pass(seq), want, rtol=0, atol=1e-10)
    assert d == 8


# ----------------------------------------------------------- invariants ----
@pytest.fixture(scope="module")
def toy_ln():
    cfg = syn.toy_config()
    w = syn.weights_as_float(syn.make_weights(cfg, seed=0, std=0.05, ln_noise=True))
    enc = syn.bf16_bits_to_f32(syn.encoder_output(cfg, 1, seed=1)[0]).astype(np.float64)
    prompt = syn.random_tokens(cfg, (7,), seed=21)
    return cfg, w, enc, prompt


def _prefill(cfg, w, enc, prompt):
    return WhisperFlashOracle(w, cfg).prefill(enc, prompt, budget=4)._prefill_logits


def _zero_gain(w, key, layers="target_layers"):
    w2 = copy.deepcopy(w)
    for lw in w2[layers]:
        lw[key] = np.zeros_like(lw[key])
    return w2


def _zero_ln(w, ln):
    return _zero_gain(_zero_gain(w, ln + "_g"), ln + "_b")


def test_ln1_gain_zero_cuts_rows_apart(toy_ln):
    """LN1 feeds only self-attention: with its gain zero every query, key and
    value is one constant row, so a row's logits no longer depend on the
    other rows' tokens."""
    cfg, w, enc, prompt = toy_ln
    other = prompt.copy()
    other[:-1] = (other[:-1] + 13) % cfg.vocab
    assert not np.allclose(_prefill(cfg, w, enc, prompt)[-1], _prefill(cfg, w, enc, other)[-1])
    w0 = _zero_gain(w, "ln1_g")
    np.testing.assert_allclose(_prefill(cfg, w0, enc, prompt)[-1], _prefill(cfg, w0, enc, other)[-1],
                               rtol=0, atol=1e-12)


@pytest.mark.parametrize("ln,weights", [("ln1", ("qkv_w",)), ("ln2", ("xq_w",)), ("ln3", ("fc1_w",))])
def test_block_ln_zero_frees_its_sublayer(toy_ln, ln, weights):
    """LN1 feeds only the self-attention projections, LN2 only the
    cross-attention query, LN3 only fc1: with that LayerNorm's gain and bias
    zero the sub-layer's input is zero, so the result no longer depends on its
    input weights, while it still depends on the other sub-layers'."""
    cfg, w, enc, prompt = toy_ln
    other_ln = {"ln1": "ln2", "ln2": "ln3", "ln3": "ln1"}[ln]
    other_w = {"ln1": "xq_w", "ln2": "fc1_w", "ln3": "qkv_w"}[ln]

    def scaled(wx, keys):
        w2 = copy.deepcopy(wx)
        for lw in w2["target_layers"]:
            for k in keys:
                lw[k] = lw[k] * -2.5
        return w2

    w0 = _zero_ln(w, ln)
    base = _prefill(cfg, w0, enc, prompt)
    np.testing.assert_allclose(_prefill(cfg, scaled(w0, weights), enc, prompt), base, rtol=0, atol=1e-12)
    assert not np.allclose(_prefill(cfg, scaled(w0, (other_w,)), enc, prompt), base)
    w1 = _zero_ln(w, other_ln)
    assert not np.allclose(_prefill(cfg, scaled(w1, weights), enc, prompt), _prefill(cfg, w1, enc, prompt))


def test_final_ln_gain_zero_gives_one_logit_row(toy_ln):
    """Logits are LN_f(x) Emb^T: with LN_f's gain zero every row is lnf_b Emb^T."""
    cfg, w, enc, prompt = toy_ln
    w0 = copy.deepcopy(w)
    w0["target"]["lnf_g"] = np.zeros_like(w0["target"]["lnf_g"])
    got = _prefill(cfg, w0, enc, prompt)
    want = w0["target"]["tok_emb"] @ w0["target"]["lnf_b"]
    np.testing.assert_allclose(got, np.broadcast_to(want, got.shape), rtol=0, atol=1e-12)


def test_history_ln_gain_zero_frees_the_history_projection(toy_ln):
    """LN_h normalises the projected history: with its gain zero every history
    row is hln_b, so the drafter no longer depends on W_p (but still on
    hln_b); the final LN is not involved."""
    cfg, w, enc, prompt = toy_ln

    def drafter_logits(wx):
        o = WhisperFlashOracle(wx, cfg)
        seq = o.prefill(enc, prompt, budget=20)
        return o.drafter_pass(seq)

    w0 = copy.deepcopy(w)
    w0["drafter"]["hln_g"] = np.zeros_like(w0["drafter"]["hln_g"])
    base = drafter_logits(w0)
    w1 = copy.deepcopy(w0)
    w1["drafter"]["proj_w"] = w1["drafter"]["proj_w"] * -3.0
    np.testing.assert_allclose(drafter_logits(w1), base, rtol=0, atol=1e-12)
    w2 = copy.deepcopy(w0)
    w2["drafter"]["hln_b"] = w2["drafter"]["hln_b"] + 0.5
    assert not np.allclose(drafter_logits(w2), base)
    w3 = copy.deepcopy(w)
    w3["drafter"]["proj_w"] = w3["drafter"]["proj_w"] * -3.0
    assert not np.allclose(drafter_logits(w3), drafter_logits(w))


def test_pre_ln_blocks_keep_row_differences(toy_ln):
    """With every block LayerNorm gain zero each sub-layer adds one constant
    row, so the tapped residual streams of two rows differ exactly by their
    input embeddings (a post-LN block would erase the difference)."""
    cfg, w, enc, prompt = toy_ln
    w0 = copy.deepcopy(w)
    for lw in w0["target_layers"]:
        for k in ("ln1_g", "ln2_g", "ln3_g"):
            lw[k] = np.zeros_like(lw[k])
    o = WhisperFlashOracle(w0, cfg)
    seq = o.prefill(enc, prompt, budget=4)
    _, taps, _, _ = o.target_pass(seq, prompt[:3], [0, 1, 2])
    x_in = w0["target"]["tok_emb"][prompt[:3]] + w0["target"]["pos_emb"][:3]
    d = cfg.d_model
    for t in range(cfg.n_taps):
        dt = taps[:, t * d:(t + 1) * d]
        np.testing.assert_allclose(dt - dt[0], x_in - x_in[0], rtol=0, atol=1e-12)
