"""A transcript that reaches the handle's context capacity (GPU).

App. A.1 bounds a sequence by its output budget; the cache bounds it too: a
verify block needs 9 free positions.  With max_ctx = 40 and a budget of 60
the accept kernel must freeze the sequence (done, WF_DEV_ERR_CAPACITY set)
after the last step whose block still fitted: every row it wrote lies inside
the cache, so the final length is at most max_ctx.  Up to that point the
speculative transcript must equal plain greedy decoding on a handle of the
same shape, token for token: on a single-sequence handle (skinny projections
with the attention fused into them, which attend to the short cache in
blocks of 32 positions) and on a two-slot handle, both with the batched
skinny projections (whose K/V epilogue checks each row's position) and with
the tcgen05 projections, and the separate attention kernel."""
import numpy as np
import pytest

from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu

CTX = 40
BUDGET = 60


def _run(cfg, dev, enc, prompt, max_batch, spec, skinny):
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session
    s = Session(cfg, dev, max_batch=max_batch, max_ctx=CTX)
    if skinny is not None:
        B.wf_set_option(s.h, B.WF_OPT_SKINNY, skinny)
    slots = np.arange(max_batch, dtype=np.int32)
    first = s.prefill(slots, enc, prompt, np.full(max_batch, BUDGET, np.int32)).cpu().numpy()
    out = [[int(first[b])] for b in range(max_batch)]
    for _ in range(200):
        toks, cnt = s.step() if spec else s.greedy_step()
        toks, cnt = toks.cpu().numpy(), cnt.cpu().numpy()
        if cnt.sum() == 0:
            break
        for b in range(max_batch):
            out[b].extend(int(x) for x in toks[b, :cnt[b]])
    st = s.state()
    err = s.error()
    s.close()
    return out, st, err, B


@pytest.mark.parametrize("max_batch,skinny", [(1, None), (2, 1), (2, 0)],
                         ids=["skinny-fused", "skinny-batched", "tcgen05"])
def test_capacity_freezes_the_sequence_inside_the_cache(max_batch, skinny):
    from paper_2609_32869_gb300.session import upload_weights
    cfg = syn.TINY
    dev = upload_weights(syn.make_weights(cfg, seed=0, ln_noise=True))
    enc = syn.encoder_output(cfg, max_batch, seed=3)
    prompt = syn.prompts(cfg, max_batch, length=4, seed=3)
    spec, st, err, B = _run(cfg, dev, enc, prompt, max_batch, True, skinny)
    plain, _, _, _ = _run(cfg, dev, enc, prompt, max_batch, False, skinny)
    K1 = cfg.block_k + 1
    for b in range(max_batch):
        assert st["done"][b]
        assert st["len"][b] <= CTX                # every block row stayed inside the cache
        n = min(len(spec[b]), len(plain[b]))
        assert spec[b][:n] == plain[b][:n], b
        if cfg.eos_id not in spec[b]:             # the cache, not the transcript, ended it
            assert st["len"][b] + K1 > CTX        # frozen only once the next block no longer fits
            assert len(spec[b]) < BUDGET
            assert err & B.WF_DEV_ERR_CAPACITY
    assert not (err & ~B.WF_DEV_ERR_CAPACITY)
