"""Seeded synthetic inputs for the Whisper-Flash decode step.

This module is shared by the CUDA path's harness (tests, bench) and by the CPU
oracle's tests.  It holds NO arithmetic of the method: it only draws numbers.

Every draw is a pure function of (seed, tensor name, element index): a
splitmix64 hash of the index gives two 32-bit uniforms, Box-Muller turns them
into a standard normal, and the value is rounded to bfloat16 with
round-to-nearest-even on the float32 bit pattern.  Integer draws (token ids,
lengths, accept lengths) reduce the same hash modulo the range.  Nothing here
depends on the machine, the thread count or the numpy/torch version beyond
IEEE arithmetic, so the x86 development box and the Arm GPU host draw the same
bits.

Workload shapes follow the paper's setting: a Whisper-large-shaped decoder
(d=1280, 20 heads, FFN 5120, 32 layers, vocabulary 51866, 448 learned
positions) and 1500 encoder frames per 30 s window (Sec. 4, Sec. 5.1,
App. A.2); the tiny shape is Whisper-tiny's (d=384, 6 heads, FFN 1536,
4 layers, vocabulary 51865).  Weights are N(0, 0.02) bf16, LayerNorm gains 1
and biases 0; encoder outputs are N(0, 1) bf16.  With `ln_noise` every
LayerNorm gain is drawn from N(1, 0.1) and every LayerNorm bias from
N(0, 0.05) instead (bf16), so that a test can tell the LayerNorms apart.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 21


# ----------------------------------------------------------------------------
# configurations
# ----------------------------------------------------------------------------
@dataclass(frozen=True)
class ModelConfig:
    """Decoder + drafter shape.  `taps` are the zero-based target blocks whose
    output residual streams form the drafter's history features."""
    name: str
    d_model: int
    n_heads: int
    d_ff: int
    n_layers: int
    vocab: int
    max_pos: int = 448
    n_draft_layers: int = 2
    block_k: int = 8
    taps: tuple = (1, 8, 15, 22, 29)
    eos_id: int = 50257
    rope_base: float = 10000.0
    ln_eps: float = 1e-5
    enc_frames: int = 1500
    # which target layers seed the drafter's blocks (None: independent draws)
    draft_init_from: tuple | None = None

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads

    @property
    def n_taps(self) -> int:
        return len(self.taps)


TINY = ModelConfig(name="tiny", d_model=384, n_heads=6, d_ff=1536, n_layers=4,
                   vocab=51865, taps=(0, 1, 2, 3, 3))
LARGE = ModelConfig(name="large", d_model=1280, n_heads=20, d_ff=5120, n_layers=32,
                    vocab=51866, taps=(1, 8, 15, 22, 29), draft_init_from=(0, 31))


def toy_config(**kw) -> ModelConfig:
    """A very small decoder for oracle pins and quick GPU checks (several
    tiles and a ragged tail still appear: d=128, vocab 1000)."""
    base = dict(name="toy", d_model=128, n_heads=2, d_ff=512, n_layers=3, vocab=1000,
                max_pos=128, taps=(0, 1, 2, 2, 1), eos_id=999, enc_frames=200)
    base.update(kw)
    return ModelConfig(**base)


# ----------------------------------------------------------------------------
# hashing and draws
# ----------------------------------------------------------------------------
def _fnv1a64(text: str) -> int:
    h = 0xCBF29CE484222325
    for byte in text.encode():
        h ^= byte
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def _stream_key(seed: int, name: str) -> np.uint64:
    return np.uint64((_fnv1a64(name) ^ ((seed * 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF))
                     & 0xFFFFFFFFFFFFFFFF)


def _mix(x: np.ndarray) -> np.ndarray:
    x = x ^ (x >> np.uint64(30))
    x = x * _M1
    x = x ^ (x >> np.uint64(27))
    x = x * _M2
    return x ^ (x >> np.uint64(31))


def _hash_range(key: np.uint64, start: int, stop: int) -> np.ndarray:
    idx = np.arange(start, stop, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(idx * _GOLDEN + key)


def _normal_chunk(key, start, stop, std) -> np.ndarray:
    h = _hash_range(key, start, stop)
    u1 = ((h >> np.uint64(32)).astype(np.float64) + 0.5) * (1.0 / 4294967296.0)
    u2 = ((h & np.uint64(0xFFFFFFFF)).astype(np.float64) + 0.5) * (1.0 / 4294967296.0)
    z = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)
    return f32_to_bf16_bits((z * std).astype(np.float32))


def _threads() -> int:
    try:
        return max(1, min(16, len(os.sched_getaffinity(0))))
    except AttributeError:  # pragma: no cover
        return max(1, min(16, os.cpu_count() or 1))


def normal_bf16(seed: int, name: str, shape, std: float) -> np.ndarray:
    """N(0, std^2) drawn per element, rounded to bf16; returned as uint16 bits."""
    n = int(np.prod(shape))
    key = _stream_key(seed, name)
    out = np.empty(n, dtype=np.uint16)
    spans = [(s, min(n, s + _CHUNK)) for s in range(0, n, _CHUNK)]

    def work(span):
        out[span[0]:span[1]] = _normal_chunk(key, span[0], span[1], std)

    if len(spans) > 1:
        with ThreadPoolExecutor(_threads()) as ex:
            list(ex.map(work, spans))
    elif spans:
        work(spans[0])
    return out.reshape(shape)


def uniform_int(seed: int, name: str, shape, lo: int, hi: int) -> np.ndarray:
    """Integers uniform on [lo, hi] inclusive (int64)."""
    n = int(np.prod(shape))
    h = _hash_range(_stream_key(seed, name), 0, n)
    span = np.uint64(hi - lo + 1)
    return ((h >> np.uint64(11)) % span).astype(np.int64).reshape(shape) + lo


def uniform_01(seed: int, name: str, shape) -> np.ndarray:
    n = int(np.prod(shape))
    h = _hash_range(_stream_key(seed, name), 0, n)
    return ((h >> np.uint64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)).reshape(shape)


# ----------------------------------------------------------------------------
# bf16 bit helpers (pure data conversion)
# ----------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest-even), returning the 16-bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _const_bf16(shape, value: float) -> np.ndarray:
    return np.full(shape, f32_to_bf16_bits(np.array([value], np.float32))[0], dtype=np.uint16)


# ----------------------------------------------------------------------------
# parameter sets (uint16 bf16 bit patterns)
# ----------------------------------------------------------------------------
LAYER_KEYS = ("ln1_g", "ln1_b", "qkv_w", "qkv_b", "out_w", "out_b",
              "ln2_g", "ln2_b", "xq_w", "xq_b", "xkv_w", "xkv_b", "xout_w", "xout_b",
              "ln3_g", "ln3_b", "fc1_w", "fc1_b", "fc2_w", "fc2_b")


def _ln_pair(seed: int, name: str, d: int, noise: bool):
    """LayerNorm gain and bias: 1 and 0, or N(1, 0.1) and N(0, 0.05) draws."""
    if not noise:
        return _const_bf16((d,), 1.0), _const_bf16((d,), 0.0)
    dev = bf16_bits_to_f32(normal_bf16(seed, name + "_g", (d,), 0.1))
    g = f32_to_bf16_bits((dev + np.float32(1.0)).astype(np.float32))
    return g, normal_bf16(seed, name + "_b", (d,), 0.05)


def _layer(seed: int, prefix: str, cfg: ModelConfig, std: float, ln_noise: bool = False) -> dict:
    d, f = cfg.d_model, cfg.d_ff
    w = {}
    for nm in ("ln1", "ln2", "ln3"):
        w[nm + "_g"], w[nm + "_b"] = _ln_pair(seed, prefix + nm, d, ln_noise)
    w["qkv_w"] = normal_bf16(seed, prefix + "qkv_w", (3 * d, d), std)
    qkv_b = normal_bf16(seed, prefix + "qkv_b", (3 * d,), std)
    qkv_b[d:2 * d] = 0          # the key projection carries no bias in Whisper
    w["qkv_b"] = qkv_b
    w["out_w"] = normal_bf16(seed, prefix + "out_w", (d, d), std)
    w["out_b"] = normal_bf16(seed, prefix + "out_b", (d,), std)
    w["xq_w"] = normal_bf16(seed, prefix + "xq_w", (d, d), std)
    w["xq_b"] = normal_bf16(seed, prefix + "xq_b", (d,), std)
    w["xkv_w"] = normal_bf16(seed, prefix + "xkv_w", (2 * d, d), std)
    xkv_b = normal_bf16(seed, prefix + "xkv_b", (2 * d,), std)
    xkv_b[:d] = 0
    w["xkv_b"] = xkv_b
    w["xout_w"] = normal_bf16(seed, prefix + "xout_w", (d, d), std)
    w["xout_b"] = normal_bf16(seed, prefix + "xout_b", (d,), std)
    w["fc1_w"] = normal_bf16(seed, prefix + "fc1_w", (f, d), std)
    w["fc1_b"] = normal_bf16(seed, prefix + "fc1_b", (f,), std)
    w["fc2_w"] = normal_bf16(seed, prefix + "fc2_w", (d, f), std)
    w["fc2_b"] = normal_bf16(seed, prefix + "fc2_b", (d,), std)
    return w


@dataclass
class WeightSet:
    """All parameters as bf16 bit patterns (numpy uint16).

    Matrices are [out, in] row-major.  `qkv_w` stacks the query, key and value
    projections ([3d, d]); `xkv_w` stacks the acoustic key and value
    projections ([2d, d]); the key biases are zero."""
    cfg: ModelConfig
    target: dict = field(default_factory=dict)
    target_layers: list = field(default_factory=list)
    drafter: dict = field(default_factory=dict)
    drafter_layers: list = field(default_factory=list)


def make_weights(cfg: ModelConfig, seed: int = 0, std: float = 0.02,
                 ln_noise: bool = False) -> WeightSet:
    """Seeded parameters.  ln_noise: LayerNorm gains N(1, 0.1) and biases
    N(0, 0.05) (every LayerNorm its own draw) instead of 1 and 0."""
    d = cfg.d_model
    ws = WeightSet(cfg=cfg)
    ws.target["tok_emb"] = normal_bf16(seed, "tok_emb", (cfg.vocab, d), std)
    ws.target["pos_emb"] = normal_bf16(seed, "pos_emb", (cfg.max_pos, d), std)
    ws.target["lnf_g"], ws.target["lnf_b"] = _ln_pair(seed, "lnf", d, ln_noise)
    ws.target_layers = [_layer(seed, f"t{i}.", cfg, std, ln_noise) for i in range(cfg.n_layers)]
    if cfg.draft_init_from is not None:
        ws.drafter_layers = [{k: v.copy() for k, v in ws.target_layers[i].items()}
                             for i in cfg.draft_init_from]
    else:
        ws.drafter_layers = [_layer(seed, f"d{i}.", cfg, std, ln_noise)
                             for i in range(cfg.n_draft_layers)]
    ws.drafter["proj_w"] = normal_bf16(seed, "d.proj_w", (d, cfg.n_taps * d), std)
    ws.drafter["proj_b"] = normal_bf16(seed, "d.proj_b", (d,), std)
    ws.drafter["hln_g"], ws.drafter["hln_b"] = _ln_pair(seed, "d.hln", d, ln_noise)
    ws.drafter["mask_emb"] = normal_bf16(seed, "d.mask_emb", (d,), std)
    return ws


def weights_as_float(ws: WeightSet, dtype=np.float64) -> dict:
    """The same parameter values as float arrays (exact: bf16 embeds in fp32/fp64)."""
    conv = lambda a: bf16_bits_to_f32(a).astype(dtype, copy=False)
    return {
        "cfg": ws.cfg,
        "target": {k: conv(v) for k, v in ws.target.items()},
        "target_layers": [{k: conv(v) for k, v in lw.items()} for lw in ws.target_layers],
        "drafter": {k: conv(v) for k, v in ws.drafter.items()},
        "drafter_layers": [{k: conv(v) for k, v in lw.items()} for lw in ws.drafter_layers],
    }


# ----------------------------------------------------------------------------
# per-request inputs
# ----------------------------------------------------------------------------
def encoder_output(cfg: ModelConfig, n: int, seed: int = 1) -> np.ndarray:
    """Stand-in for the Whisper encoder output: [n, frames, d] bf16 bits, N(0,1)."""
    return normal_bf16(seed, "enc", (n, cfg.enc_frames, cfg.d_model), 1.0)


def prompts(cfg: ModelConfig, n: int, length: int = 4, seed: int = 1) -> np.ndarray:
    """Seeded token ids standing in for the language/task prompt, never EOS."""
    ids = uniform_int(seed, f"prompt{length}", (n, length), 0, cfg.vocab - 2)
    return np.where(ids >= cfg.eos_id, ids + 1, ids).astype(np.int32)


def budgets(n: int, lo: int, hi: int, seed: int = 2) -> np.ndarray:
    """Per-sequence output token budgets, uniform on [lo, hi]."""
    return uniform_int(seed, f"budget{lo}_{hi}", (n,), lo, hi).astype(np.int32)


def accept_uniform(n_steps: int, n: int, k: int = 8, seed: int = 3) -> np.ndarray:
    """Teacher-forced accept lengths, uniform on 0..k: [n_steps, n]."""
    return uniform_int(seed, "accept_u", (n_steps, n), 0, k).astype(np.int32)


def accept_geometric(n_steps: int, n: int, mean: float = 4.0, k: int = 8,
                     seed: int = 3) -> np.ndarray:
    """Teacher-forced accept lengths: successes before the first failure with
    success probability mean/(1+mean), clipped to k: [n_steps, n]."""
    p = mean / (1.0 + mean)
    u = uniform_01(seed, "accept_g", (n_steps, n, k))
    ok = u < p
    run = np.cumprod(ok, axis=-1)
    return run.sum(axis=-1).astype(np.int32)


def random_tokens(cfg: ModelConfig, shape, seed: int, name: str = "tok") -> np.ndarray:
    return uniform_int(seed, name, shape, 0, cfg.vocab - 1).astype(np.int32)
