"""Kernel-level parity of the CUDA path with the oracle (GPU).

Each kernel family runs alone through its C entry point on seeded inputs and
is compared element by element with the oracle's float64 restatement of the
same operation."""
import numpy as np
import pytest

from oracle import decoder as od
from paper_2609_32869_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu


def _dev(bits_u16, shape=None):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits_u16).view(np.int16)).view(torch.bfloat16)
    if shape is not None:
        t = t.reshape(shape)
    return t.cuda()


def _f64(bits):
    return syn.bf16_bits_to_f32(bits).astype(np.float64)


GEMM_CASES = [
    # (M, N, K): split-K and single-split shapes, ragged N and M tails, several token tiles
    (1, 1280, 1280), (9, 1280, 1280), (9, 3840, 1280), (17, 5120, 1280), (9, 1280, 5120),
    (9, 1280, 6400), (144, 2560, 1280), (300, 1000, 128), (9, 51866, 1280), (1500, 2560, 1280),
    # token tiles of 48 and 64 rows (split-K rows pushed to their owner CTA)
    # and just past them (rows reduced by pulling partials), 16 and 10 splits
    (40, 1280, 5120), (64, 1280, 5120), (65, 1280, 5120), (64, 1280, 1280), (97, 1280, 1280),
]


@pytest.mark.parametrize("M,N,K", GEMM_CASES)
def test_gemm_matches_oracle(M, N, K):
    import torch
    from paper_2609_32869_gb300 import binding as B
    x = syn.normal_bf16(11, f"x{M}", (M, K), 1.0)
    w = syn.normal_bf16(12, f"w{N}", (N, K), 0.02)
    b = syn.normal_bf16(13, f"b{N}", (N,), 0.02)
    y = torch.empty(M, N, dtype=torch.float32, device="cuda")
    nbytes = B.wf_gemm_scratch_bytes(M, N, K)
    scratch = torch.empty(max(nbytes, 256), dtype=torch.uint8, device="cuda")
    B.wf_gemm_bf16(_dev(x), _dev(w), _dev(b), y, M, N, K, scratch, nbytes)
    torch.cuda.synchronize()
    got = y.cpu().numpy().astype(np.float64)
    want = od.linear(_f64(x), _f64(w), _f64(b))
    # fp32 accumulation of K exact bf16 products: |err| <= K * 2^-23 * sum|x w|
    bound = K * 2.0 ** -23 * (np.abs(_f64(x)) @ np.abs(_f64(w)).T) + 1e-6
    err = np.abs(got - want)
    assert (err <= bound).all(), f"max err {err.max():.3e}, worst ratio {(err / bound).max():.2f}"


def test_gemm_rows_do_not_depend_on_batch():
    """A row's result is bit-identical whether it runs alone, among 9 rows, or
    among 300 or 1000 (fixed split-K and token-tile-independent reduction
    order; at 1000 rows the 10 splits of a tile run in one CTA and are added
    in the same order as the cluster reduction of the smaller launches)."""
    import torch
    from paper_2609_32869_gb300 import binding as B
    N, K = 1280, 1280
    x = syn.normal_bf16(21, "xb", (1000, K), 1.0)
    w = _dev(syn.normal_bf16(22, "wb", (N, K), 0.02))
    outs = {}
    for M in (1, 9, 64, 65, 300, 1000):
        y = torch.empty(M, N, dtype=torch.float32, device="cuda")
        nb = B.wf_gemm_scratch_bytes(M, N, K)
        sc = torch.empty(max(nb, 256), dtype=torch.uint8, device="cuda")
        B.wf_gemm_bf16(_dev(x[:M]), w, None, y, M, N, K, sc, nb)
        outs[M] = y.cpu().numpy()
    np.testing.assert_array_equal(outs[1][0], outs[300][0])
    np.testing.assert_array_equal(outs[9], outs[300][:9])
    np.testing.assert_array_equal(outs[64], outs[300][:64])
    np.testing.assert_array_equal(outs[65], outs[300][:65])
    np.testing.assert_array_equal(outs[300], outs[1000][:300])


def _cache(n_slots, H, ctx, seed, name, std=1.0):
    return syn.normal_bf16(seed, name, (n_slots, H, ctx, 64), std)


@pytest.mark.parametrize("mode,rps,ctx,rope", [(0, 9, 300, 0), (0, 1, 300, 0), (0, 40, 300, 0),
                                                (1, 9, 300, 1), (2, 9, 1500, 0)])
def test_attention_matches_oracle(mode, rps, ctx, rope):
    import torch
    from paper_2609_32869_gb300 import binding as B
    H, n_seq, n_slots = 3, 3, 4
    d = H * 64
    slots = np.array([2, 0, 3], np.int32)
    base = np.array([100, 0, 57, 211], np.int32)       # cache length L per slot
    q = syn.normal_bf16(31, f"q{mode}{rps}", (n_seq * rps, d), 1.0)
    kc = _cache(n_slots, H, ctx, 32, f"k{ctx}")
    vc = _cache(n_slots, H, ctx, 33, f"v{ctx}")
    out = torch.empty(n_seq * rps, d, dtype=torch.bfloat16, device="cuda")
    nb = B.wf_attention_scratch_bytes(n_seq, rps, H, ctx)
    sc = torch.empty(nb, dtype=torch.uint8, device="cuda")
    B.wf_attention(_dev(q), _dev(kc), _dev(vc), torch.from_numpy(slots).cuda(),
                   torch.from_numpy(base).cuda(), n_seq, rps, H, ctx, mode, rope, 10000.0, out,
                   sc, nb)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy().astype(np.float64)
    qf, kf, vf = _f64(q), _f64(kc), _f64(vc)
    for i, slot in enumerate(slots):
        L = base[slot]
        qi = qf[i * rps:(i + 1) * rps]
        if mode == 2:
            n_keys = ctx
        else:
            n_keys = L + rps
        keys = kf[slot][:, :n_keys].transpose(1, 0, 2).reshape(n_keys, d)
        vals = vf[slot][:, :n_keys].transpose(1, 0, 2).reshape(n_keys, d)
        vis = None
        if mode == 0:
            vis = np.arange(n_keys)[None, :] <= (L + np.arange(rps))[:, None]
        if rope:
            qi = od.rope(qi, L + np.arange(rps), H, 10000.0)
            keys = od.rope(keys, np.arange(n_keys), H, 10000.0)
        want = od.multi_head_attention(qi, keys, vals, H, vis)
        g = got[i * rps:(i + 1) * rps]
        # bf16 output rounding (2^-8 relative) dominates the fp32 arithmetic
        np.testing.assert_allclose(g, want, atol=2e-2, rtol=1e-2)
        assert np.abs(g - want).max() < 3 * 2.0 ** -8 * max(1.0, np.abs(want).max())


@pytest.mark.parametrize("mode,ctx", [(2, 1500), (0, 448)])
def test_attention_one_cta_per_group_equals_split_blocks(mode, ctx):
    """A launch with at least two (sequence, head, query group)s per SM runs
    one CTA per group that walks its 256-key blocks in order; it leaves the
    split form's partials and merges them in block order itself, so each
    sequence's rows equal, bit for bit, those of a launch of that sequence
    alone (split blocks, merged over a cluster), and the oracle within the
    attention tolerance.  Whisper-large heads, 16 sequences, 9 query rows."""
    import torch
    from paper_2609_32869_gb300 import binding as B
    H, n_seq, rps = 20, 16, 9
    d = H * 64
    slots = np.array([(5 * i + 3) % n_seq for i in range(n_seq)], np.int32)
    base = np.array([(37 * s + 11) % (ctx - rps) for s in range(n_seq)], np.int32)
    q = syn.normal_bf16(41, f"ql{mode}", (n_seq * rps, d), 1.0)
    kc = _cache(n_seq, H, ctx, 42, f"kl{ctx}")
    vc = _cache(n_seq, H, ctx, 43, f"vl{ctx}")
    dk, dv, db = _dev(kc), _dev(vc), torch.from_numpy(base).cuda()

    def run(rows, sl):
        n = len(sl)
        out = torch.empty(n * rps, d, dtype=torch.bfloat16, device="cuda")
        nb = B.wf_attention_scratch_bytes(n, rps, H, ctx)
        sc = torch.empty(nb, dtype=torch.uint8, device="cuda")
        B.wf_attention(_dev(rows), dk, dv, torch.from_numpy(np.asarray(sl, np.int32)).cuda(), db, n, rps,
                       H, ctx, mode, 0, 10000.0, out, sc, nb)
        torch.cuda.synchronize()
        return out.float().cpu().numpy()

    big = run(q, slots)
    qf, kf, vf = _f64(q), _f64(kc), _f64(vc)
    for i in (0, 7, 15):
        one = run(q[i * rps:(i + 1) * rps], slots[i:i + 1])
        np.testing.assert_array_equal(big[i * rps:(i + 1) * rps], one)
        slot = slots[i]
        L = base[slot]
        n_keys = ctx if mode == 2 else L + rps
        keys = kf[slot][:, :n_keys].transpose(1, 0, 2).reshape(n_keys, d)
        vals = vf[slot][:, :n_keys].transpose(1, 0, 2).reshape(n_keys, d)
        vis = None if mode == 2 else np.arange(n_keys)[None, :] <= (L + np.arange(rps))[:, None]
        want = od.multi_head_attention(qf[i * rps:(i + 1) * rps], keys, vals, H, vis)
        g = big[i * rps:(i + 1) * rps].astype(np.float64)
        np.testing.assert_allclose(g, want, atol=2e-2, rtol=1e-2)
