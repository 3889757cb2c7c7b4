"""Mutation check of the oracle's pins.

Each case plants one plausible mistake in a copy of an oracle function (on
the CPU, for the duration of the case only: the function's source with one
edit, compiled and patched in) and requires that at least one pin of the
oracle fails.  A mistake that every pin let through would be a mistake the
oracle could carry into every parity test unseen."""
import __future__
import importlib.util
import inspect
import os
import textwrap

import numpy as np
import pytest

from oracle import acceptance, decoder
from oracle.decoder import WhisperFlashOracle
from paper_2609_32869_gb300 import synthetic as syn

HERE = os.path.dirname(os.path.abspath(__file__))


def _load(name):
    spec = importlib.util.spec_from_file_location(f"_mutation_pins_{name}", os.path.join(HERE, f"{name}.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _pins():
    """Every pin as a no-argument callable, cheapest first."""
    dec, prim = _load("test_oracle_decoder"), _load("test_oracle_primitives")
    lnr, sampling = _load("test_oracle_ln_routing"), _load("test_oracle_sampling")

    def toy():
        cfg = syn.toy_config()
        w = syn.weights_as_float(syn.make_weights(cfg, seed=0, std=0.05))
        enc = syn.bf16_bits_to_f32(syn.encoder_output(cfg, 2, seed=1)).astype(np.float64)
        return cfg, w, enc, syn.prompts(cfg, 2, length=4, seed=1)

    def toy_ln():
        cfg = syn.toy_config()
        w = syn.weights_as_float(syn.make_weights(cfg, seed=0, std=0.05, ln_noise=True))
        enc = syn.bf16_bits_to_f32(syn.encoder_output(cfg, 1, seed=1)[0]).astype(np.float64)
        return cfg, w, enc, syn.random_tokens(cfg, (7,), seed=21)

    def d8():
        cfg = lnr._cfg8()
        wf = syn.weights_as_float(syn.make_weights(cfg, seed=11, std=0.5, ln_noise=True))
        enc = syn.bf16_bits_to_f32(syn.encoder_output(cfg, 1, seed=2)[0]).astype(np.float64)
        return cfg, wf, enc, np.array([3, 7, 1], np.int32)

    pins = [
        prim.test_gelu_is_the_erf_form, prim.test_layer_norm_moments_and_affine,
        prim.test_linear_orientation_is_out_by_in, prim.test_attention_closed_forms,
        prim.test_attention_mask_hides_keys, prim.test_rope_rotation_convention,
        prim.test_rope_depends_only_on_position_difference,
        dec.test_greedy_accept_edge_cases, dec.test_fig1_worked_example,
        sampling.test_residual_is_positive_part_normalised,
        lambda: sampling.test_rejection_rule_preserves_target_distribution_exactly(1, 0),
        lambda: sampling.test_rejection_rule_preserves_target_distribution_exactly(2, 1),
        lambda: lnr.test_hand_checked_target_block_d8(d8()),
        lambda: lnr.test_hand_checked_drafter_d8(d8()),
        lambda: dec.test_first_position_attends_to_itself(toy()),
        lambda: dec.test_causality(toy()),
        lambda: dec.test_incremental_cache_equals_full_causal_pass(toy()),
        lambda: dec.test_zero_blocks_copy_the_input_token(toy()),
        lambda: dec.test_budget_reserves_one_slot(toy()),
        lambda: dec.test_speculative_greedy_equals_plain_greedy(toy(), "forced"),
        lambda: dec.test_speculative_greedy_stops_at_eos_like_greedy(toy()),
        lambda: lnr.test_pre_ln_blocks_keep_row_differences(toy_ln()),
        lambda: lnr.test_history_ln_gain_zero_frees_the_history_projection(toy_ln()),
        lambda: lnr.test_final_ln_gain_zero_gives_one_logit_row(toy_ln()),
        lambda: dec.test_drafter_history_visibility_and_bidirectional_block(toy()),
        lambda: sampling.test_philox_driven_sampler_matches_target_first_two_tokens(1),
    ]
    return pins


def _mutate(owner, name, edits):
    """owner.name recompiled from its source with the (old, new) edits applied
    in order; each `old` must occur exactly once when its edit applies."""
    fn = getattr(owner, name)
    fn = getattr(fn, "__func__", fn)
    src = textwrap.dedent(inspect.getsource(fn))
    for old, new in edits:
        assert src.count(old) == 1, (name, old)
        src = src.replace(old, new)
    scope = dict(fn.__globals__)
    code = compile(src, inspect.getsourcefile(fn), "exec",
                   flags=__future__.annotations.compiler_flag, dont_inherit=True)
    exec(code, scope)
    return scope[name]


W = WhisperFlashOracle
MUTATIONS = {
    "ln2 and ln3 swapped": (W, "_cross_ffn", [('lw["ln2_g"], lw["ln2_b"]', "LN_SWAP"),
                                              ('lw["ln3_g"], lw["ln3_b"]', 'lw["ln2_g"], lw["ln2_b"]'),
                                              ("LN_SWAP", 'lw["ln3_g"], lw["ln3_b"]')]),
    "final LN in place of the history LN": (W, "history_features",
                                            [('self.d["hln_g"], self.d["hln_b"]', 'self.t["lnf_g"], self.t["lnf_b"]')]),
    "history LN in place of the drafter's final LN": (
        W, "drafter_pass", [('layer_norm(x[1:], self.t["lnf_g"], self.t["lnf_b"]',
                             'layer_norm(x[1:], self.d["hln_g"], self.d["hln_b"]')]),
    "post-LN self-attention": (W, "target_pass", [
        ('h = layer_norm(x, lw["ln1_g"], lw["ln1_b"], self.eps)', 'h = x'),
        ('x = x + linear(a, lw["out_w"], lw["out_b"])',
         'x = layer_norm(x + linear(a, lw["out_w"], lw["out_b"]), lw["ln1_g"], lw["ln1_b"], self.eps)')]),
    "LayerNorm bias dropped": (decoder, "layer_norm", [("* g + b", "* g")]),
    "LayerNorm gain dropped": (decoder, "layer_norm", [("* g + b", "+ b")]),
    "flipped FFN residual": (W, "_cross_ffn", [("return x + linear(gelu(", "return x - linear(gelu(")]),
    "dropped self-attention residual": (W, "target_pass", [('x = x + linear(a, lw["out_w"]', 'x = linear(a, lw["out_w"]')]),
    "bonus from the wrong row": (acceptance, "greedy_accept",
                                 [("last = int(target_argmax[a])", "last = int(target_argmax[a - 1 if a == k and k else a])")]),
    "verify mask one position late": (W, "target_pass", [("key_pos[None, :] <= positions[:, None]",
                                                          "key_pos[None, :] <= positions[:, None] + 1")]),
    "RoPE rotates the wrong way": (decoder, "rope", [("x1 * c - x2 * s, x2 * c + x1 * s",
                                                      "x1 * c + x2 * s, x2 * c - x1 * s")]),
    "RoPE pairs adjacent dims": (decoder, "rope", [("x1, x2 = xh[..., :half], xh[..., half:]",
                                                    "x1, x2 = xh[..., 0::2], xh[..., 1::2]")]),
    "candidate checked against the next row": (acceptance, "greedy_accept",
                                               [("if c != int(target_argmax[i]):", "if c != int(target_argmax[i + 1]):")]),
    "cache keeps a rows instead of 1 + a": (W, "spec_step", [("self._commit(seq, nk, nv, taps, 1 + a)",
                                                              "self._commit(seq, nk, nv, taps, max(a, 1))")]),
    "bonus after an accepted EOS": (acceptance, "greedy_accept", [("return emitted, i + 1, True", "break")]),
    "history keys one position late": (W, "drafter_pass", [("kh = rope(kh, np.arange(L) + pos_shift",
                                                            "kh = rope(kh, np.arange(L) + 1 + pos_shift")]),
    "budget does not reserve a slot": (W, "spec_step", [("min(K, seq.remaining - 1)", "min(K, seq.remaining)")]),
    "inverted acceptance ratio": (acceptance, "rejection_accept", [("np.float32(p_c / q_c)", "np.float32(q_c / p_c)")]),
    "residual not clipped at zero": (acceptance, "residual_distribution",
                                     [("np.maximum(np.asarray(p, dtype=np.float64) - np.asarray(q, dtype=np.float64), 0.0)",
                                       "np.abs(np.asarray(p, dtype=np.float64) - np.asarray(q, dtype=np.float64))")]),
    "drafter block causal instead of bidirectional": (
        W, "drafter_pass", [("np.concatenate([vh, vb]), self.nh)",
                             "np.concatenate([vh, vb]), self.nh, np.tril(np.ones((K + 1, L + K + 1), bool), L))")]),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_fails_a_pin(name, monkeypatch):
    owner, attr, edits = MUTATIONS[name]
    monkeypatch.setattr(owner, attr, _mutate(owner, attr, edits))
    caught = None
    for pin in _pins():
        try:
            pin()
        except Exception as e:  # an assertion, or a crash the mistake causes
            caught = e
            break
    assert caught is not None, f"no pin fails with the mistake '{name}'"


def test_unmutated_oracle_passes_every_pin():
    for pin in _pins():
        pin()
