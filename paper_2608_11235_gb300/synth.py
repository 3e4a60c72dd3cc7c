"""Seeded synthetic inputs: weights, prompts and gate-isolation logits.

This module is the ONE place that both the CUDA path's callers and the CPU
oracle's callers take their inputs from. It holds none of the decoding
method's arithmetic: only a counter-based random generator and the recipes
that turn its bits into tensors of the paper's workload shapes.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast Splittable Pseudorandom
Number Generators", OOPSLA 2014).  The i-th output (0-based) of a stream with
state ``key`` is ``mix64(key + (i + 1) * GOLDEN)`` with

    mix64(z): z ^= z >> 30; z *= 0xBF58476D1CE4E5B9
              z ^= z >> 27; z *= 0x94D049BB133111EB
              z ^= z >> 31

(all arithmetic mod 2**64).  Every tensor has its own stream key, so element
``i`` of any tensor can be produced independently; the CUDA library carries a
second implementation of the same generator (``cora_synth_normal_bf16``) so the
8B-parameter weights can be written straight into device memory, and a test
checks the two bit for bit.

An approximate N(0, sigma) sample is the Irwin-Hall sum of the four 16-bit
fields of one 64-bit output: ``X = 2*(u0+u1+u2+u3) - 4*65535`` (an odd
integer, |X| <= 262140, exact in fp32), scaled by the fp32 constant
``sigma / SD_X`` with one IEEE fp32 multiply.  A workload whose weights are
bf16 (``weight_dtype`` "bf16", the default) rounds that product to bf16
(round to nearest even), so both sides see identical values; a workload with
fp32 weights (``weight_dtype`` "f32", the tiny model) keeps the fp32 product,
which in general is not bf16-representable: the oracle computes with it and
the library rounds it to bf16 on the device.  Integer fields, one fp32
multiply and an integer rounding step give the same bits on any IEEE machine.
"""

from __future__ import annotations

import math

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB

# Standard deviation of X = 2*(u0+u1+u2+u3) - 4*65535 with u_j uniform on
# {0..65535}: var(u) = (65536**2 - 1)/12, var(X) = 4 * 4 * var(u).
SD_X = math.sqrt(16.0 * (65536.0 ** 2 - 1.0) / 12.0)


def mix64_int(z: int) -> int:
    """SplitMix64 output function on a Python int (mod 2**64)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, stream: int) -> int:
    """Key of stream ``stream`` under ``seed``: mix64(mix64(seed) + stream)."""
    return mix64_int((mix64_int(seed) + stream) & MASK64)


def _mix64(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(MIX1)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(MIX2)
    return z ^ (z >> np.uint64(31))


def bits64(key: int, start: int, count: int) -> np.ndarray:
    """Outputs ``start .. start+count-1`` of the SplitMix64 stream ``key``."""
    with np.errstate(over="ignore"):
        idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
        z = np.uint64(key) + idx * np.uint64(GOLDEN)
        return _mix64(z)


def normal_scale_f32(sigma: float) -> np.float32:
    """fp32 multiplier that maps X to an approximate N(0, sigma) sample."""
    return np.float32(sigma / SD_X)


def f32_to_bf16_bits(f: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest, ties to even); returns uint16 bit patterns.

    Inputs here are finite, so no NaN handling is needed.
    """
    u = np.ascontiguousarray(f, dtype=np.float32).view(np.uint32)
    bias = np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to fp32 values (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_f32(key: int, start: int, count: int, sigma: float) -> np.ndarray:
    """Approximate N(0, sigma) samples in fp32: X times the fp32 scale (see module doc)."""
    b = bits64(key, start, count)
    m = np.uint64(0xFFFF)
    s = (b & m) + ((b >> np.uint64(16)) & m) + ((b >> np.uint64(32)) & m) + (b >> np.uint64(48))
    x = (2 * s.astype(np.int64) - 4 * 65535).astype(np.float32)
    return x * normal_scale_f32(sigma)


def normal_bf16_bits(key: int, start: int, count: int, sigma: float) -> np.ndarray:
    """Approximate N(0, sigma) samples as bf16 bit patterns (see module doc)."""
    return f32_to_bf16_bits(normal_f32(key, start, count, sigma))


def uniform_int(key: int, start: int, count: int, n: int) -> np.ndarray:
    """Integers uniform on [0, n): high 32 bits times n, shifted down 32."""
    assert 0 < n < (1 << 32)
    b = bits64(key, start, count)
    return ((b >> np.uint64(32)) * np.uint64(n) >> np.uint64(32)).astype(np.int64)


def uniform01(key: int, start: int, count: int) -> np.ndarray:
    """Doubles uniform on the open interval (0, 1): ((bits >> 11) + 0.5) / 2**53."""
    b = bits64(key, start, count)
    return ((b >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)


# ---------------------------------------------------------------------------
# Model weights.  Tensor stream ids: global tensors use small ids, per-layer
# tensors use ((layer + 1) << 8) | kind.  Norm weights are all ones.
# ---------------------------------------------------------------------------
EMBED, LM_HEAD = 1, 2
WQ, WK, WV, WO, WGATE, WUP, WDOWN = 3, 4, 5, 6, 7, 8, 9


def tensor_stream(layer: int, kind: int) -> int:
    return kind if layer < 0 else (((layer + 1) << 8) | kind)


def weight_shapes(cfg: dict) -> dict:
    """Shapes (nn.Linear layout: [out_features, in_features]) of every tensor."""
    d, hd, hq, hkv, f, v = (cfg["d_model"], cfg["head_dim"], cfg["n_heads"],
                            cfg["n_kv_heads"], cfg["ffn"], cfg["vocab"])
    return {
        EMBED: (v, d), LM_HEAD: (v, d),
        WQ: (hq * hd, d), WK: (hkv * hd, d), WV: (hkv * hd, d), WO: (d, hq * hd),
        WGATE: (f, d), WUP: (f, d), WDOWN: (d, f),
    }


def weight_sigma(cfg: dict, kind: int) -> float:
    return float(cfg["head_sigma"]) if kind == LM_HEAD else float(cfg["init_sigma"])


def weight_bf16_bits(cfg: dict, layer: int, kind: int, rows: slice | None = None) -> np.ndarray:
    """bf16 bits of one weight tensor (optionally a row range), shape [rows, cols]."""
    shp = weight_shapes(cfg)[kind]
    r0, r1 = (0, shp[0]) if rows is None else (rows.start or 0, rows.stop)
    key = stream_key(cfg["seed"], tensor_stream(layer, kind))
    out = normal_bf16_bits(key, r0 * shp[1], (r1 - r0) * shp[1], weight_sigma(cfg, kind))
    return out.reshape(r1 - r0, shp[1])


def weight_f32(cfg: dict, layer: int, kind: int, rows: slice | None = None) -> np.ndarray:
    """fp32 values of one weight tensor of an fp32-weight workload (not rounded to bf16)."""
    shp = weight_shapes(cfg)[kind]
    r0, r1 = (0, shp[0]) if rows is None else (rows.start or 0, rows.stop)
    key = stream_key(cfg["seed"], tensor_stream(layer, kind))
    return normal_f32(key, r0 * shp[1], (r1 - r0) * shp[1], weight_sigma(cfg, kind)).reshape(r1 - r0, shp[1])


def is_f32_weights(cfg: dict) -> bool:
    return cfg.get("weight_dtype", "bf16") == "f32"


def weight_f64(cfg: dict, layer: int, kind: int, rows: slice | None = None) -> np.ndarray:
    """The workload's weight values widened to float64: the fp32 originals of an
    fp32-weight workload, else the bf16 values."""
    if is_f32_weights(cfg):
        return weight_f32(cfg, layer, kind, rows).astype(np.float64)
    return bf16_bits_to_f32(weight_bf16_bits(cfg, layer, kind, rows)).astype(np.float64)


def model_weights_f64(cfg: dict) -> dict:
    """All weights widened to float64, in the layout the oracle reads."""
    L = cfg["n_layers"]
    d = cfg["d_model"]
    w = {
        "embed": weight_f64(cfg, -1, EMBED),
        "lm_head": weight_f64(cfg, -1, LM_HEAD),
        "final_norm": np.ones(d),
        "layers": [],
    }
    for l in range(L):
        w["layers"].append({
            "attn_norm": np.ones(d), "ffn_norm": np.ones(d),
            "wq": weight_f64(cfg, l, WQ), "wk": weight_f64(cfg, l, WK),
            "wv": weight_f64(cfg, l, WV), "wo": weight_f64(cfg, l, WO),
            "w_gate": weight_f64(cfg, l, WGATE), "w_up": weight_f64(cfg, l, WUP),
            "w_down": weight_f64(cfg, l, WDOWN),
        })
    return w


def layer_weights_f64(cfg: dict, l: int) -> dict:
    d = cfg["d_model"]
    return {
        "attn_norm": np.ones(d), "ffn_norm": np.ones(d),
        "wq": weight_f64(cfg, l, WQ), "wk": weight_f64(cfg, l, WK),
        "wv": weight_f64(cfg, l, WV), "wo": weight_f64(cfg, l, WO),
        "w_gate": weight_f64(cfg, l, WGATE), "w_up": weight_f64(cfg, l, WUP),
        "w_down": weight_f64(cfg, l, WDOWN),
    }


# ---------------------------------------------------------------------------
# Prompts: ids uniform on [0, mask_id), one stream per (seed, sequence).
# ---------------------------------------------------------------------------
PROMPT_STREAM = 0x50524F4D  # "PROM"


def prompts(seed: int, batch: int, length: int, mask_id: int) -> np.ndarray:
    out = np.empty((batch, length), dtype=np.int32)
    for b in range(batch):
        key = stream_key(seed, PROMPT_STREAM + b)
        out[b] = uniform_int(key, 0, length, mask_id)
    return out


# ---------------------------------------------------------------------------
# Mid-decode canvases (full-size parity at later blocks): prompt, then every
# block before `block` committed to uniform ids on [0, mask_id), the active
# block with each position committed with probability `frac_resolved`, and
# the later blocks masked.  State codes: 0 unresolved, 1 transferred.
# ---------------------------------------------------------------------------
CANVAS_STREAM = 0x43414E56  # "CANV"


def mid_decode_canvas(cfg: dict, seed: int, block: int, frac_resolved: float) -> tuple:
    """(tokens int32 [P + G], state uint8 [G]) for sequence 0 of `cfg`."""
    P, G, BL, mask_id = cfg["prompt_len"], cfg["gen_len"], cfg["block_len"], cfg["mask_id"]
    key = stream_key(seed, CANVAS_STREAM + block)
    prompt = prompts(cfg["prompt_seed"], 1, P, mask_id)[0]
    ids = uniform_int(key, 0, G, mask_id)
    pos = np.arange(G)
    committed = pos < block * BL
    active = (pos >= block * BL) & (pos < (block + 1) * BL)
    committed |= active & (uniform01(key, G, G) < frac_resolved)
    gen = np.where(committed, ids, mask_id).astype(np.int32)
    return np.concatenate([prompt.astype(np.int32), gen]), committed.astype(np.uint8)


# ---------------------------------------------------------------------------
# Gate-isolation inputs: bf16 logits [B, R, V] = Gumbel(0,1) + Delta * onehot
# (Delta ~ U[0, 12]) plus a history of prior-step argmax tensors and a mask
# state.  The boosted target of a row is its last history id with prob 0.8,
# else a fresh uniform id; each history step keeps the previous id with
# prob 0.8, else draws a new uniform id.
# ---------------------------------------------------------------------------
HIST_STREAM, STATE_STREAM, TARGET_STREAM, GUMBEL_STREAM = 0x48495354, 0x53544154, 0x54415247, 0x47554D42


def gate_history(seed: int, B: int, R: int, V: int, n_hist: int = 8, keep: float = 0.8) -> np.ndarray:
    """[n_hist, B, R] int32 argmax history."""
    n = B * R
    h = np.empty((n_hist, n), dtype=np.int64)
    h[0] = uniform_int(stream_key(seed, HIST_STREAM), 0, n, V)
    for t in range(1, n_hist):
        k = stream_key(seed, HIST_STREAM + t)
        stay = uniform01(k, 0, n) < keep
        fresh = uniform_int(k, n, n, V)
        h[t] = np.where(stay, h[t - 1], fresh)
    return h.reshape(n_hist, B, R).astype(np.int32)


def gate_unresolved(seed: int, B: int, R: int, frac: float = 0.5) -> np.ndarray:
    """[B, R] bool: True where the position is still masked (unresolved)."""
    return (uniform01(stream_key(seed, STATE_STREAM), 0, B * R) < frac).reshape(B, R)


def gate_logits_bf16(seed: int, B: int, R: int, V: int, last_hist: np.ndarray,
                     keep: float = 0.8, delta_max: float = 12.0) -> np.ndarray:
    """[B, R, V] uint16 bf16 logits; generated row by row to bound memory."""
    n = B * R
    kt = stream_key(seed, TARGET_STREAM)
    stay = uniform01(kt, 0, n) < keep
    fresh = uniform_int(kt, n, n, V)
    target = np.where(stay, last_hist.reshape(-1), fresh)
    delta = uniform01(kt, 2 * n, n) * delta_max
    out = np.empty((n, V), dtype=np.uint16)
    kg = stream_key(seed, GUMBEL_STREAM)
    for r in range(n):
        u = uniform01(kg, r * V, V)
        g = -np.log(-np.log(u))
        g[target[r]] += delta[r]
        out[r] = f32_to_bf16_bits(g.astype(np.float32))
    return out.reshape(B, R, V)
