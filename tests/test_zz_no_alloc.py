"""wf_attention_noalloc: the attention entry point that allocates nothing.

It serves callers that cannot allocate device memory; its scratch is an
array inside the library.  Checked through the C ABI against wf_attention
(which takes caller scratch) on two calls in a row, the second with a
different attention mode and size, so state left in the shared array by the
first call must not leak into the second.  Kept in a file of its own that
pytest collects last."""
import numpy as np
import pytest

from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu


def _dev(bits, torch):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def test_noalloc_attention_matches_scratch_entry_point_twice():
    """Both entry points run the same kernel on the same inputs, so their
    outputs must agree bit for bit.  The cases alternate between the path
    that merges key blocks inside a thread-block cluster and the path that
    merges them through the scratch array (partial sums and counters: more
    than 8 key blocks), changing mode and size between calls, so a partial
    or counter left in the array by one call would show in the next."""
    import torch
    from paper_2609_32869_gb300 import binding as B
    H, n_seq, n_slots = 4, 3, 4
    d = H * 64
    slots = torch.tensor([2, 0, 3], dtype=torch.int32, device="cuda")
    # (mode, rows per sequence, cache positions, RoPE): cross over 3000 frames
    # (12 key blocks: scratch merge), causal over 300 (cluster merge), drafter
    # block with RoPE, causal over 2600 positions (scratch merge, other size)
    cases = [(2, 9, 3000, 0), (0, 9, 300, 0), (1, 9, 300, 1), (0, 9, 2600, 0)]
    for call, (mode, rps, ctx, rope) in enumerate(cases):
        base = torch.tensor([100, 0, min(2200, ctx - rps), 211], dtype=torch.int32, device="cuda")
        q = _dev(syn.normal_bf16(41 + call, "naq", (n_seq * rps, d), 1.0), torch)
        kc = _dev(syn.normal_bf16(42 + call, "nak", (n_slots, H, ctx, 64), 1.0), torch)
        vc = _dev(syn.normal_bf16(43 + call, "nav", (n_slots, H, ctx, 64), 1.0), torch)
        ref = torch.empty(n_seq * rps, d, dtype=torch.bfloat16, device="cuda")
        got = torch.full_like(ref, float("nan"))
        nb = B.wf_attention_scratch_bytes(n_seq, rps, H, ctx)
        sc = torch.empty(nb, dtype=torch.uint8, device="cuda")
        B.wf_attention(q, kc, vc, slots, base, n_seq, rps, H, ctx, mode, rope, 1e4, ref, sc, nb)
        B.wf_attention_noalloc(q, kc, vc, slots, base, n_seq, rps, H, ctx, mode, rope, 1e4, got)
        torch.cuda.synchronize()
        assert torch.isfinite(ref.float()).all()
        assert torch.equal(got, ref), (call, mode, ctx)


def test_noalloc_rejects_oversize_requests():
    import torch
    from paper_2609_32869_gb300 import binding as B
    H, n_seq, rps, ctx = 20, 64, 9, 1500       # needs more than the 8 MiB array
    assert B.wf_attention_scratch_bytes(n_seq, rps, H, ctx) > 8 << 20
    q = torch.zeros(n_seq * rps, H * 64, dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros(1, dtype=torch.bfloat16, device="cuda")
    slots = torch.zeros(n_seq, dtype=torch.int32, device="cuda")
    out = torch.empty_like(q)
    with pytest.raises(B.WfError) as e:
        B.wf_attention_noalloc(q, kv, kv, slots, None, n_seq, rps, H, ctx, 2, 0, 1e4, out)
    assert e.value.status == B.WF_ERR_CAPACITY
