"""Speculative sampling at the full Whisper-large shapes (vocabulary 51866):
the first emitted token's distribution (GPU).

64 batch slots hold the same request in the same state after a greedy
prefill, so the first token every speculative step emits has the same
target distribution p1 = softmax(z / T) at the anchor row, where z are the
target's logits (the oracle's, float64).  Each of 32 repetitions rewinds the
slots and takes one step with its own seed (every slot draws from its own
Philox streams), giving 2048 draws per case.  The ids are binned into 16
bins of equal p1-mass (cut in id order; the mass each bin really holds is
taken exactly from p1) and the counts are tested with a chi-square against
the expected counts.  The same number of plain autoregressive draws from the
GPU (wf_greedy_step at the same temperature) must agree with the
speculative ones in a two-sample chi-square over the same bins.

Proposals are the drafter's own draws, or teacher-forced draws from
q = softmax((z + 0.3 eps) / T) with their logits passed to the step (the
benchmark's recipe): the first exercises the residual redraw at this
vocabulary size, the second mostly accepted proposals (Sec. 3.1, App. A.4)."""
import numpy as np
import pytest

from oracle import acceptance
from oracle.decoder import WhisperFlashOracle
from paper_2609_32869_gb300 import synthetic as syn

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

N_SLOTS, REPS, BINS = 64, 32, 16


@pytest.fixture(scope="module")
def large():
    import torch
    from paper_2609_32869_gb300.session import Session, upload_weights
    cfg = syn.LARGE
    ws = syn.make_weights(cfg, seed=0)
    dev = upload_weights(ws)
    enc1 = syn.encoder_output(cfg, 1, seed=5)
    prompt1 = syn.prompts(cfg, 1, length=4, seed=5)
    s = Session(cfg, dev, max_batch=N_SLOTS)
    enc = torch.from_numpy(enc1.view(np.int16)).view(torch.bfloat16).cuda().expand(N_SLOTS, -1, -1).contiguous()
    prompt = np.broadcast_to(prompt1, (N_SLOTS, 4)).copy()
    first = s.prefill(np.arange(N_SLOTS, dtype=np.int32), enc, prompt,
                      np.full(N_SLOTS, 50, np.int32)).cpu().numpy()
    assert (first == first[0]).all()
    # the oracle continues from the anchor the GPU chose (the greedy first
    # token may be a near tie between the two sides' roundings)
    o = WhisperFlashOracle(syn.weights_as_float(ws, np.float64), cfg)
    seq = o.prefill(syn.bf16_bits_to_f32(enc1[0]).astype(np.float64), prompt1[0], 50)
    seq.anchor = int(first[0])
    z0, _, _, _ = o.target_pass(seq, [seq.anchor], [seq.L])
    yield cfg, s, z0[0]
    s.close()


def _bins(p):
    """16 bins of (nearly) equal mass, cut in id order; returns the bin of
    every id and each bin's exact mass."""
    c = np.cumsum(p)
    mid = c - p / 2
    b = np.minimum((mid * BINS).astype(np.int64), BINS - 1)
    mass = np.bincount(b, weights=p, minlength=BINS)
    return b, mass


def _draws(s, cfg, T, proposals, plain, z0):
    import torch
    from paper_2609_32869_gb300 import binding as B
    K, V = cfg.block_k, cfg.vocab
    slots = np.arange(N_SLOTS, dtype=np.int32)
    out = []
    gen = torch.Generator(device="cuda")
    z = torch.as_tensor(z0, dtype=torch.float32, device="cuda")
    for rep in range(REPS):
        s.reset_slots(slots)
        assert s.compact() == N_SLOTS
        sp = B.sample_params(T, 9000 + rep)
        if plain:
            toks, cnt = s.greedy_step(sp=sp)
        elif proposals == "drafter":
            toks, cnt = s.step(sp=sp)
        else:
            gen.manual_seed(300 + rep)
            zq = z[None, None, :] + 0.3 * torch.randn((N_SLOTS, K, V), generator=gen, device="cuda")
            u = torch.rand((N_SLOTS, K, V), generator=gen, device="cuda").clamp_(1e-12, 1.0)
            cand = torch.argmax(zq / T - torch.log(-torch.log(u)), dim=-1).to(torch.int32)
            toks, cnt = s.step(forced=cand, sp=sp, forced_q=zq.contiguous())
        t = toks.cpu().numpy()
        assert (cnt.cpu().numpy() >= 1).all()
        out.append(t[:, 0].copy())
    assert s.error() == 0
    return np.concatenate(out)


@pytest.mark.parametrize("T", [0.7, 1.0])
@pytest.mark.parametrize("proposals", ["drafter", "forced_q"])
def test_first_token_follows_the_target_at_large_shapes(large, T, proposals):
    from scipy.stats import chi2_contingency, chisquare
    cfg, s, z0 = large
    p = acceptance.probs_fp32(acceptance.scaled_logits_fp32(z0, T)).astype(np.float64)
    p /= p.sum()
    bin_of, mass = _bins(p)
    spec = _draws(s, cfg, T, proposals, False, z0)
    plain = _draws(s, cfg, T, proposals, True, z0)
    n = len(spec)
    obs = np.bincount(bin_of[spec], minlength=BINS).astype(np.float64)
    exp = mass * n
    assert exp.min() >= 5
    assert chisquare(obs, exp).pvalue > 1e-3, (obs, exp)
    obs_plain = np.bincount(bin_of[plain], minlength=BINS).astype(np.float64)
    assert chi2_contingency(np.stack([obs, obs_plain])).pvalue > 1e-3
