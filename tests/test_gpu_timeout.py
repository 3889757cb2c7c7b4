"""Failure detection: a bounded wait that runs out (GPU).

Every spin-wait in the projection kernels and the persistent pass is
bounded; when it gives up it records WF_DEV_ERR_TIMEOUT in the handle's
error word, waits (with the default limit) for its own copies and
tensor-core work in flight, and returns.  Here the limit is cut to a few
dozen clock cycles, far below any wait for data from memory, so waits give
up during one step.  The call must return, the error word must say TIMEOUT,
and after the word is cleared, the default limit restored and the slot
rewound, the same steps must give bit-identical results to a handle that
never timed out.  Nothing here faults or hangs a GPU: every wait still ends
within its limit."""
import numpy as np
import pytest

from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu


def _run(s, forced_steps):
    out = []
    for f in forced_steps:
        toks, cnt = s.step(forced=f)
        st = s.state()
        out.append((toks.cpu().numpy().copy(), cnt.cpu().numpy().copy(), st["len"].copy(),
                    st["anchor"].copy()))
    return out


@pytest.mark.parametrize("persist", [False, True], ids=["launch-by-launch", "persistent"])
def test_bounded_wait_gives_up_and_the_handle_recovers(persist):
    import torch
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session, upload_weights
    cfg = syn.TINY
    K, V = cfg.block_k, cfg.vocab
    ws = syn.make_weights(cfg, seed=0, ln_noise=True)
    dev = upload_weights(ws)
    enc = syn.encoder_output(cfg, 1, seed=1)
    prompt = syn.prompts(cfg, 1, length=4, seed=1)
    budget = np.array([60], np.int32)
    forced = [syn.random_tokens(cfg, (1, K), seed=70 + i) for i in range(2)]

    def session():
        s = Session(cfg, dev, max_batch=1)
        if persist:
            B.wf_set_option(s.h, B.WF_OPT_PERSIST, 1)
        s.prefill([0], enc, prompt, budget)
        return s

    ref_s = session()
    ref = _run(ref_s, forced)
    assert ref_s.error() == 0
    ref_s.close()

    s = session()
    assert s.error() == 0
    B.wf_set_option(s.h, B.WF_OPT_SPIN_LIMIT, 32)
    s.step(forced=forced[0])            # returns: every wait is bounded
    torch.cuda.synchronize()
    err = s.error(clear=True)
    assert err & B.WF_DEV_ERR_TIMEOUT, err
    assert s.error() == 0
    B.wf_set_option(s.h, B.WF_OPT_SPIN_LIMIT, 0)
    s.reset_slots([0])
    assert s.compact() == 1
    got = _run(s, forced)
    for (t0, c0, l0, a0), (t1, c1, l1, a1) in zip(ref, got):
        assert np.array_equal(t0, t1) and np.array_equal(c0, c1)
        assert np.array_equal(l0, l1) and np.array_equal(a0, a1)
    assert s.error() == 0
    with pytest.raises(B.WfError):
        B.wf_set_option(s.h, B.WF_OPT_SPIN_LIMIT, -1)
    s.close()
