"""Whisper-shaped target decoder, Whisper-Flash drafter and decode steps (oracle).

TEST INFRASTRUCTURE ONLY (see the package docstring).  float64 numpy
throughout, except where the paper fixes FP32 (RoPE phases, App. A.2; sampling
softmax and acceptance, App. A.4).  One sequence at a time: batching is an
implementation matter the method does not change.

Target decoder (the paper uses frozen Whisper large-v3 and does not restate
it; this is the Whisper decoder block as published with the model): token
embedding plus learned position embedding; per block
    x += SelfAttn(LN1 x)       causal, with a key/value cache
    x += CrossAttn(LN2 x, A)   over the encoder output A (keys/values
                               projected once per request, App. A.5)
    x += fc2(GELU(fc1(LN3 x)))
then a final LayerNorm and the output head tied to the token embedding.
Attention scale 1/sqrt(head_dim); GELU is the erf form.

Drafter (Sec. 3.2, Eq. 2, App. A.2): input [Emb(anchor), m, ..., m] with K=8
copies of the mask vector m and no absolute position embedding; each of its
two Whisper blocks self-attends in ONE softmax over the projected history of
accepted positions < anchor and the 9 block positions (bidirectional inside
the block), with RoPE (base 10000, FP32 phases, explicit text positions) on
queries and keys; it cross-attends to the encoder output through its own
acoustic key/value projections and runs its FFN; the frozen target's final
LayerNorm and tied output head, shared with the target, give one distribution
per mask position.  The drafter's own parameters are its two blocks, the
history projection with its LayerNorm, and m: 60.7M at the large shapes,
47.5M without the cross-attention path, 52.5M without the history projection
(Sec. 3.2, Table 3), which leaves room for exactly one extra LayerNorm.

History memory (Sec. 3.2, App. A.2): the target's residual streams after
blocks {1, 8, 15, 22, 29} (zero-based, before the final LayerNorm) at every
accepted position, concatenated and projected to the drafter width.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
from scipy.special import erf

from . import acceptance, philox


# ------------------------------------------------------------ primitives ----
def layer_norm(x, g, b, eps):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


def gelu(x):
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def linear(x, w, b=None):
    y = x @ w.T
    return y if b is None else y + b


def softmax(x, axis=-1):
    m = np.max(x, axis=axis, keepdims=True)
    e = np.exp(x - m)
    return e / e.sum(axis=axis, keepdims=True)


def multi_head_attention(q, k, v, n_heads, visible=None):
    """q [nq, d], k/v [nk, d]; visible[i, j] says whether query i sees key j."""
    nq, d = q.shape
    dh = d // n_heads
    qh = q.reshape(nq, n_heads, dh)
    kh = k.reshape(-1, n_heads, dh)
    vh = v.reshape(-1, n_heads, dh)
    s = np.einsum("qhd,khd->hqk", qh, kh) / np.sqrt(dh)
    if visible is not None:
        s = np.where(visible[None], s, -np.inf)
    p = softmax(s, axis=-1)
    return np.einsum("hqk,khd->qhd", p, vh).reshape(nq, d)


def rope(x, positions, n_heads, base):
    """Rotary embedding on every head of x [n, d]: dims i and i + dh/2 of a head
    rotate together by angle pos * base^(-2i/dh); the angle is formed in FP32
    (App. A.2), its cosine and sine in float64."""
    n, d = x.shape
    dh = d // n_heads
    half = dh // 2
    inv = (np.float32(base) ** (-(np.arange(half, dtype=np.float32) * np.float32(2.0))
                                / np.float32(dh))).astype(np.float32)
    ang = (np.asarray(positions, dtype=np.float32)[:, None] * inv[None, :]).astype(np.float64)
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    xh = x.reshape(n, n_heads, dh)
    x1, x2 = xh[..., :half], xh[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1).reshape(n, d)


# ----------------------------------------------------------------- state ----
@dataclass
class Sequence:
    """Decode state of one request.  Caches hold ACCEPTED positions only: rows
    enter when the step that produced them is kept (App. A.1)."""
    seq_id: int
    cross_k: list = field(default_factory=list)     # per target layer [T, d]
    cross_v: list = field(default_factory=list)
    dcross_k: list = field(default_factory=list)    # per drafter layer [T, d]
    dcross_v: list = field(default_factory=list)
    self_k: list = field(default_factory=list)      # per target layer [L, d]
    self_v: list = field(default_factory=list)
    hist: np.ndarray | None = None                  # drafter history memory [L, d]
    L: int = 0                                      # target cache length
    anchor: int = -1                                # latest emitted, unprocessed token
    remaining: int = 0                              # output tokens still allowed
    done: bool = False
    step: int = 0                                   # speculative-step counter
    emitted: list = field(default_factory=list)


@dataclass
class StepRecord:
    draft_logits: np.ndarray          # [K, V] drafter logits at mask positions 1..K
    candidates: np.ndarray            # [K] proposals (live ones first)
    k: int                            # live candidates
    verify_logits: np.ndarray         # [k+1, V]
    verify_taps: np.ndarray           # [k+1, n_taps*d]
    accepted: int                     # a
    emitted: list


class WhisperFlashOracle:
    def __init__(self, weights: dict, cfg):
        self.cfg = cfg
        self.t = weights["target"]
        self.tl = weights["target_layers"]
        self.d = weights["drafter"]
        self.dl = weights["drafter_layers"]
        self.nh = cfg.n_heads
        self.dm = cfg.d_model
        self.eps = cfg.ln_eps

    # ------------------------------------------------------ building blocks --
    def acoustic_kv(self, lw, enc):
        """Acoustic keys and values of one layer, projected once per request."""
        d = self.dm
        k = linear(enc, lw["xkv_w"][:d], lw["xkv_b"][:d])
        v = linear(enc, lw["xkv_w"][d:], lw["xkv_b"][d:])
        return k, v

    def _self_attn_proj(self, lw, h):
        d = self.dm
        qkv = linear(h, lw["qkv_w"], lw["qkv_b"])
        return qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]

    def _cross_ffn(self, lw, x, ck, cv):
        h = layer_norm(x, lw["ln2_g"], lw["ln2_b"], self.eps)
        qc = linear(h, lw["xq_w"], lw["xq_b"])
        x = x + linear(multi_head_attention(qc, ck, cv, self.nh), lw["xout_w"], lw["xout_b"])
        h = layer_norm(x, lw["ln3_g"], lw["ln3_b"], self.eps)
        return x + linear(gelu(linear(h, lw["fc1_w"], lw["fc1_b"])), lw["fc2_w"], lw["fc2_b"])

    def target_pass(self, seq: Sequence, tokens, positions):
        """One causal target pass over a block of tokens at the given positions,
        on top of the accepted cache.  Returns logits [n, V], history taps
        [n, n_taps*d] and the block's per-layer keys/values (not committed)."""
        tokens = np.asarray(tokens)
        positions = np.asarray(positions)
        n = len(tokens)
        L = seq.L
        x = self.t["tok_emb"][tokens] + self.t["pos_emb"][positions]
        taps = {}
        new_k, new_v = [], []
        key_pos = np.concatenate([np.arange(L), positions])
        visible = key_pos[None, :] <= positions[:, None]
        for li, lw in enumerate(self.tl):
            h = layer_norm(x, lw["ln1_g"], lw["ln1_b"], self.eps)
            q, k, v = self._self_attn_proj(lw, h)
            new_k.append(k)
            new_v.append(v)
            keys = np.concatenate([seq.self_k[li][:L], k]) if L else k
            vals = np.concatenate([seq.self_v[li][:L], v]) if L else v
            a = multi_head_attention(q, keys, vals, self.nh, visible)
            x = x + linear(a, lw["out_w"], lw["out_b"])
            x = self._cross_ffn(lw, x, seq.cross_k[li], seq.cross_v[li])
            taps[li] = x.copy()
        tap_rows = np.concatenate([taps[i] for i in self.cfg.taps], axis=-1)
        logits = self.head(layer_norm(x, self.t["lnf_g"], self.t["lnf_b"], self.eps))
        return logits, tap_rows, new_k, new_v

    def head(self, h):
        """Output head tied to the token embedding."""
        return h @ self.t["tok_emb"].T

    def history_features(self, tap_rows):
        """Concatenated tap rows projected to the drafter width (Sec. 3.2); the
        projection is followed by the drafter's history LayerNorm."""
        h = linear(tap_rows, self.d["proj_w"], self.d["proj_b"])
        return layer_norm(h, self.d["hln_g"], self.d["hln_b"], self.eps)

    def drafter_pass(self, seq: Sequence, pos_shift: int = 0):
        """Drafter logits for the K mask positions of the block anchored at L.
        `pos_shift` adds a constant to every RoPE position (a test hook: RoPE
        depends only on position differences, so it must not change the result)."""
        cfg = self.cfg
        K, L, d = cfg.block_k, seq.L, self.dm
        x = np.stack([self.t["tok_emb"][seq.anchor]] + [self.d["mask_emb"]] * K)   # Eq. 2
        pos = L + np.arange(K + 1) + pos_shift
        hist = seq.hist[:L]
        for li, lw in enumerate(self.dl):
            h = layer_norm(x, lw["ln1_g"], lw["ln1_b"], self.eps)
            q, kb, vb = self._self_attn_proj(lw, h)
            kh = linear(hist, lw["qkv_w"][d:2 * d], lw["qkv_b"][d:2 * d])
            vh = linear(hist, lw["qkv_w"][2 * d:], lw["qkv_b"][2 * d:])
            q = rope(q, pos, self.nh, cfg.rope_base)
            kb = rope(kb, pos, self.nh, cfg.rope_base)
            kh = rope(kh, np.arange(L) + pos_shift, self.nh, cfg.rope_base)
            a = multi_head_attention(q, np.concatenate([kh, kb]), np.concatenate([vh, vb]), self.nh)
            x = x + linear(a, lw["out_w"], lw["out_b"])
            x = self._cross_ffn(lw, x, seq.dcross_k[li], seq.dcross_v[li])
        h = layer_norm(x[1:], self.t["lnf_g"], self.t["lnf_b"], self.eps)
        return self.head(h)

    # ------------------------------------------------------------ requests --
    def _commit(self, seq: Sequence, new_k, new_v, tap_rows, n_keep: int):
        """Keep the first n_keep rows of a processed block in the target cache
        and in the drafter history (rollback drops the rest, App. A.1)."""
        for li in range(len(self.tl)):
            seq.self_k[li] = np.concatenate([seq.self_k[li], new_k[li][:n_keep]])
            seq.self_v[li] = np.concatenate([seq.self_v[li], new_v[li][:n_keep]])
        hist = self.history_features(tap_rows[:n_keep])
        seq.hist = np.concatenate([seq.hist, hist])
        seq.L += n_keep

    def _pick(self, logits_row, seq, temperature, seed, row, tag, suppress):
        if temperature == 0:
            z = logits_row if suppress is None else np.where(suppress, -np.inf, logits_row)
            return int(np.argmax(z))
        x = acceptance.scaled_logits_fp32(logits_row, temperature, suppress)
        g = philox.gumbel_noise(seed, seq.seq_id, seq.step, row, tag, self.cfg.vocab)
        return acceptance.gumbel_argmax(x, g)

    def prefill(self, enc, prompt, budget: int, seq_id: int = 0,
                temperature: float = 0.0, seed: int = 0, suppress=None) -> Sequence:
        """Acoustic K/V for every target and drafter layer, then one causal pass
        over the prompt; it emits the first transcript token, which becomes the
        first anchor (App. A.1)."""
        d = self.dm
        seq = Sequence(seq_id=seq_id)
        enc = np.asarray(enc, dtype=np.float64)
        for lw in self.tl:
            k, v = self.acoustic_kv(lw, enc)
            seq.cross_k.append(k)
            seq.cross_v.append(v)
        for lw in self.dl:
            k, v = self.acoustic_kv(lw, enc)
            seq.dcross_k.append(k)
            seq.dcross_v.append(v)
        seq.self_k = [np.zeros((0, d)) for _ in self.tl]
        seq.self_v = [np.zeros((0, d)) for _ in self.tl]
        seq.hist = np.zeros((0, d))
        prompt = np.asarray(prompt)
        logits, taps, nk, nv = self.target_pass(seq, prompt, np.arange(len(prompt)))
        self._commit(seq, nk, nv, taps, len(prompt))
        first = self._pick(logits[-1], seq, temperature, seed, 0, philox.TAG_BONUS, suppress)
        seq.anchor = first
        seq.emitted = [first]
        seq.remaining = int(budget) - 1
        seq.done = first == self.cfg.eos_id or seq.remaining <= 0
        seq.step = 1
        seq._prefill_logits = logits
        return seq

    def greedy_step(self, seq: Sequence, temperature: float = 0.0, seed: int = 0,
                    suppress=None):
        """One autoregressive target step (Eq. 1; with T>0, plain sampling)."""
        if seq.done:
            return None
        logits, taps, nk, nv = self.target_pass(seq, [seq.anchor], [seq.L])
        y = self._pick(logits[0], seq, temperature, seed, 0, philox.TAG_BONUS, suppress)
        self._commit(seq, nk, nv, taps, 1)
        seq.anchor = y
        seq.emitted.append(y)
        seq.remaining -= 1
        seq.done = y == self.cfg.eos_id or seq.remaining <= 0
        seq.step += 1
        return logits[0]

    def spec_step(self, seq: Sequence, forced=None, temperature: float = 0.0,
                  seed: int = 0, suppress=None, forced_q=None) -> StepRecord | None:
        """One propose-verify-advance round (Sec. 3.1, App. A.1, A.4).

        forced: optional K proposals that replace the drafter's (teacher
        forcing); the drafter still runs and its logits are returned.
        forced_q: optional [K, V] logits of the distributions the forced
        proposals were drawn from; the rejection rule then takes q from them
        (Sec. 3.1: q_i is the distribution the candidate was sampled from)."""
        if seq.done:
            return None
        cfg = self.cfg
        K = cfg.block_k
        k = max(0, min(K, seq.remaining - 1))          # reserve one slot (App. A.1)
        zd = self.drafter_pass(seq)
        if forced is not None:
            cands = np.asarray(forced, dtype=np.int64)[:K]
        else:
            cands = np.array([self._pick(zd[i], seq, temperature, seed, i + 1,
                                         philox.TAG_DRAFT, suppress) for i in range(K)])
        block = np.concatenate([[seq.anchor], cands[:k]]).astype(np.int64)
        zt, taps, nk, nv = self.target_pass(seq, block, seq.L + np.arange(k + 1))
        if temperature == 0:
            zz = zt if suppress is None else np.where(suppress[None], -np.inf, zt)
            emitted, a, stop = acceptance.greedy_accept(cands[:k], np.argmax(zz, axis=-1),
                                                        cfg.eos_id)
        else:
            xt = np.stack([acceptance.scaled_logits_fp32(r, temperature, suppress) for r in zt])
            zq = zd if forced_q is None else np.asarray(forced_q, dtype=np.float64)
            xd = np.stack([acceptance.scaled_logits_fp32(r, temperature, suppress)
                           for r in zq[:k]]) if k else np.zeros((0, cfg.vocab), np.float32)
            coins = [philox.accept_uniform(seed, seq.seq_id, seq.step, i + 1) for i in range(k)]
            rnoise = [philox.gumbel_noise(seed, seq.seq_id, seq.step, i + 1,
                                          philox.TAG_RESIDUAL, cfg.vocab) for i in range(k)]
            bnoise = philox.gumbel_noise(seed, seq.seq_id, seq.step, k, philox.TAG_BONUS,
                                         cfg.vocab)
            emitted, a, stop = acceptance.rejection_accept(xt, xd, cands[:k], coins, rnoise,
                                                           bnoise, cfg.eos_id)
        self._commit(seq, nk, nv, taps, 1 + a)
        seq.anchor = emitted[-1]
        seq.emitted.extend(emitted)
        seq.remaining -= len(emitted)
        seq.done = stop or seq.remaining <= 0
        seq.step += 1
        return StepRecord(draft_logits=zd, candidates=cands, k=k, verify_logits=zt,
                          verify_taps=taps, accepted=a, emitted=emitted)

    # ------------------------------------------------------------ decoding --
    def greedy_decode(self, enc, prompt, budget: int, seq_id: int = 0):
        """Plain greedy transcript (Eq. 1): the identity reference."""
        seq = self.prefill(enc, prompt, budget, seq_id)
        while not seq.done:
            self.greedy_step(seq)
        return seq.emitted
