"""Writes the oracle's first-step results for the 8B-class workloads.

For each workload, sequence 0's first executed step (block 0, step 0: canvas
= prompt + all masks) is computed by the CPU oracle in float64, one layer at
a time (weights regenerated per layer by the seeded generator), then Eq. 1 on
the 32 active rows for two LM heads: the workload's own head and the
gate-exercising head N(0, 8/sqrt(d)).  Only oracle/ and the seeded input
generator are called.

    python tests/golden/make_fullsize_golden.py [preset ...]

Output: tests/golden/fullsize_<preset>.json (conf, argmax, top-1/top-2
probability margin and logit gap per row, for each head).

    python tests/golden/make_fullsize_golden.py --blocks [preset ...]

Later blocks: the same pass on seeded mid-decode canvases of sequence 0
(synth.mid_decode_canvas), per workload in BLOCK_CASES: first passes of
later blocks and passes inside a block with part of it already resolved.
Output: tests/golden/fullsize_<preset>_blocks.json (cases already there are
kept, so new cases can be added without recomputing the others).

    python tests/golden/make_fullsize_golden.py --cached [preset ...]

Prefix-cache step (a decoding variant), per workload in CACHED_CASES: the
dense pass on the canvas with the active block fully masked keeps every
layer's keys/values; the pass on the same canvas with part of the block
resolved recomputes the rows from the block's start on, the positions before
it contributing their kept keys/values (the oracle's layer_forward_prefix,
layer by layer for both canvases, as forward_hidden_kv and
forward_hidden_cached compose it).  Output: tests/golden/fullsize_<preset>_cached.json.
"""

from __future__ import annotations

import json
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import cora_oracle as O  # noqa: E402
from paper_2608_11235_gb300 import configs, synth  # noqa: E402

PRESETS = ["llada8b-shape-256+256", "dream7b-shape-256+512-b4", "llada8b-shape-512+1024-b8"]


def head_eq1(cfg, rows, v_chunk=16384):
    V = cfg["vocab"]
    logits = np.empty((rows.shape[0], V))
    for v0 in range(0, V, v_chunk):
        v1 = min(V, v0 + v_chunk)
        head = {"final_norm": np.ones(cfg["d_model"]),
                "lm_head": synth.weight_f64(cfg, -1, synth.LM_HEAD, slice(v0, v1))}
        logits[:, v0:v1] = O.lm_logits(cfg, head, rows)
    c, a = O.top1(logits)
    srt = np.sort(logits, axis=-1)
    return {"conf": c.tolist(), "argmax": a.tolist(), "margin": O.top2_margin(logits).tolist(),
            "logit_gap": (srt[:, -1] - srt[:, -2]).tolist()}


CANVAS_SEED = 500
# (active block, fraction of it already resolved) per workload
BLOCK_CASES = {
    "llada8b-shape-256+256": [(1, 0.0), (4, 0.0), (7, 0.0), (3, 0.5), (6, 0.75), (2, 0.0), (3, 0.0), (5, 0.0),
                              (6, 0.0)],
    "dream7b-shape-256+512-b4": [(5, 0.0), (15, 0.0), (10, 0.5)] + [(b, 0.0) for b in (1, 2, 3, 4, 6, 7, 8, 9, 11, 12,
                                                                                 13, 14)] + [(3, 0.25), (12, 0.75)],
    "llada8b-shape-512+1024-b8": [(15, 0.0), (31, 0.0), (7, 0.5), (23, 0.75)],
}


def run_blocks(preset: str) -> None:
    """Cases already in the output file (same canvas seed) are kept, not recomputed.
    The missing cases go through the layers together: each layer's weights are
    generated once and applied to every canvas (generating them is most of the
    time), and the LM heads run once over all their active rows."""
    cfg = dict(configs.PRESETS[preset])
    P, BL = cfg["prompt_len"], cfg["block_len"]
    path = os.path.join(HERE, f"fullsize_{preset}_blocks.json")
    done = {}
    if os.path.exists(path):
        with open(path) as f:
            for c in json.load(f)["cases"]:
                if c["canvas_seed"] == CANVAS_SEED:
                    done[(c["block"], c["frac_resolved"])] = c
    todo = [(b, fr) for b, fr in BLOCK_CASES[preset] if (b, fr) not in done]
    if todo:
        hs, pos = [], None
        for block, frac in todo:
            tokens, _ = synth.mid_decode_canvas(cfg, CANVAS_SEED, block, frac)
            hs.append(np.stack([synth.weight_f64(cfg, -1, synth.EMBED, slice(int(t), int(t) + 1))[0]
                                for t in tokens]))
            pos = np.arange(len(tokens))
        t0 = time.time()
        for l in range(cfg["n_layers"]):
            lw = synth.layer_weights_f64(cfg, l)
            hs = [O.layer_forward(cfg, lw, h, pos) for h in hs]
            print(f"{preset}: {len(todo)} canvases, layer {l} done at {time.time() - t0:.0f} s", flush=True)
        rows = np.concatenate([h[P + b * BL: P + (b + 1) * BL] for h, (b, _) in zip(hs, todo)])
        heads = {"workload": head_eq1(cfg, rows), "gate_exercising": head_eq1(configs.gate_exercising(cfg), rows)}
        for i, (block, frac) in enumerate(todo):
            per = {name: {k: v[i * BL: (i + 1) * BL] for k, v in res.items()} for name, res in heads.items()}
            done[(block, frac)] = {"block": block, "frac_resolved": frac, "canvas_seed": CANVAS_SEED, "heads": per}
    out = {"preset": preset, "sequence": 0,
           "source": "oracle/cora_oracle.py (layer_forward, lm_logits, top1, top2_margin), float64",
           "cases": [done[c] for c in BLOCK_CASES[preset]]}
    with open(path, "w") as f:
        json.dump(out, f)


CACHED_CASES = {"llada8b-shape-256+256": [(3, 0.5), (6, 0.75)]}  # (block, fraction resolved at the cached pass)


def run_cached(preset: str) -> None:
    """Cases already in the output file (same canvas seed) are kept, not
    recomputed; the missing ones go through the layers together, each layer's
    weights generated once for all of them."""
    cfg = dict(configs.PRESETS[preset])
    P, BL = cfg["prompt_len"], cfg["block_len"]
    hkv, hd = cfg["n_kv_heads"], cfg["head_dim"]
    path = os.path.join(HERE, f"fullsize_{preset}_cached.json")
    done = {}
    if os.path.exists(path):
        with open(path) as f:
            for c in json.load(f)["cases"]:
                if c["canvas_seed"] == CANVAS_SEED:
                    done[(c["block"], c["frac_resolved"])] = c
    todo = [(b, fr) for b, fr in CACHED_CASES[preset] if (b, fr) not in done]
    if todo:
        embed = lambda toks: np.stack([synth.weight_f64(cfg, -1, synth.EMBED, slice(int(t), int(t) + 1))[0]
                                       for t in toks])
        has, hbs, los, pos = [], [], [], None
        for block, frac in todo:
            tok_a, _ = synth.mid_decode_canvas(cfg, CANVAS_SEED, block, 0.0)   # the block's first pass
            tok_b, _ = synth.mid_decode_canvas(cfg, CANVAS_SEED, block, frac)  # a later pass of the block
            lo = P + block * BL
            assert np.array_equal(tok_a[:lo], tok_b[:lo])
            has.append(embed(tok_a))
            hbs.append(embed(tok_b[lo:]))
            los.append(lo)
            pos = np.arange(len(tok_a))
        empty = np.zeros((0, hkv, hd))
        t0 = time.time()
        for l in range(cfg["n_layers"]):
            lw = synth.layer_weights_f64(cfg, l)
            for i, lo in enumerate(los):
                has[i], k, v = O.layer_forward_prefix(cfg, lw, has[i], pos, empty, empty)
                hbs[i], _, _ = O.layer_forward_prefix(cfg, lw, hbs[i], pos[lo:], k[:lo], v[:lo])
            print(f"{preset} cached: {len(todo)} cases, layer {l} done at {time.time() - t0:.0f} s", flush=True)
        rows = np.concatenate([hb[:BL] for hb in hbs])
        heads = {"workload": head_eq1(cfg, rows), "gate_exercising": head_eq1(configs.gate_exercising(cfg), rows)}
        for i, (block, frac) in enumerate(todo):
            per = {name: {k: v[i * BL: (i + 1) * BL] for k, v in res.items()} for name, res in heads.items()}
            done[(block, frac)] = {"block": block, "frac_resolved": frac, "canvas_seed": CANVAS_SEED, "heads": per}
    out = {"preset": preset, "sequence": 0,
           "source": "oracle/cora_oracle.py (layer_forward_prefix, lm_logits, top1, top2_margin), float64",
           "cases": [done[c] for c in CACHED_CASES[preset]]}
    with open(path, "w") as f:
        json.dump(out, f)


def run(preset: str) -> None:
    cfg = dict(configs.PRESETS[preset])
    P, G, BL = cfg["prompt_len"], cfg["gen_len"], cfg["block_len"]
    prompt = synth.prompts(cfg["prompt_seed"], cfg["batch"], P, cfg["mask_id"])[0]
    x = np.concatenate([prompt, np.full(G, cfg["mask_id"])])
    h = np.stack([synth.weight_f64(cfg, -1, synth.EMBED, slice(int(t), int(t) + 1))[0] for t in x])
    pos = np.arange(len(x))
    t0 = time.time()
    for l in range(cfg["n_layers"]):
        h = O.layer_forward(cfg, synth.layer_weights_f64(cfg, l), h, pos)
        print(f"{preset}: layer {l} done at {time.time() - t0:.0f} s", flush=True)
    rows = h[P: P + BL]
    out = {"preset": preset, "sequence": 0, "block": 0, "step": 0,
           "source": "oracle/cora_oracle.py (layer_forward, lm_logits, top1, top2_margin), float64",
           "heads": {"workload": head_eq1(cfg, rows),
                     "gate_exercising": head_eq1(configs.gate_exercising(cfg), rows)}}
    with open(os.path.join(HERE, f"fullsize_{preset}.json"), "w") as f:
        json.dump(out, f)


if __name__ == "__main__":
    args = sys.argv[1:]
    if args and args[0] == "--blocks":
        for p in (args[1:] or PRESETS[:1]):
            run_blocks(p)
    elif args and args[0] == "--cached":
        for p in (args[1:] or PRESETS[:1]):
            run_cached(p)
    else:
        for p in (args or PRESETS):
            run(p)
