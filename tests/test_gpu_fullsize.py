"""Full-size parity: one denoising step of each 8B-class workload, in the
session configuration bench.py times, against the oracle on sampled outputs.

The GPU runs the whole batch (every sequence, every layer, all kernels as in
the timed decode).  The oracle recomputes sequence 0's first executed step in
float64, one layer at a time (weights regenerated per layer from the seeded
generator, so host memory stays bounded), then the LM head and Eq. 1 on the
active block's 32 rows.  The LM head is the gate-exercising variant
(N(0, 8/sqrt(d))), so confidences span (0, 1) and the argmax check is not
vacuous; the body weights and every kernel launch are those of the workload.
"""

import numpy as np
import pytest
import torch

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import build, configs, cora, model, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available()
    build.build()
    cora.lib()


def oracle_first_step(cfg, prompt):
    """Sequence 0, block 0, step 0: conf, x_hat and logits of the 32 active rows."""
    P, G, BL = cfg["prompt_len"], cfg["gen_len"], cfg["block_len"]
    x = np.concatenate([prompt, np.full(G, cfg["mask_id"])])
    h = np.stack([synth.weight_f64(cfg, -1, synth.EMBED, slice(int(t), int(t) + 1))[0] for t in x])
    pos = np.arange(len(x))
    for l in range(cfg["n_layers"]):
        h = O.layer_forward(cfg, synth.layer_weights_f64(cfg, l), h, pos)
    V = cfg["vocab"]
    logits = np.empty((BL, V))
    for v0 in range(0, V, 16384):        # the head in vocabulary slices (independent columns)
        v1 = min(V, v0 + 16384)
        head = {"final_norm": np.ones(cfg["d_model"]),
                "lm_head": synth.weight_f64(cfg, -1, synth.LM_HEAD, slice(v0, v1))}
        logits[:, v0:v1] = O.lm_logits(cfg, head, h[P: P + BL])
    c, a = O.top1(logits)
    return c, a, logits


@pytest.mark.parametrize("preset", ["llada8b-shape-256+256", "dream7b-shape-256+512-b4",
                                    "llada8b-shape-512+1024-b8"])
def test_first_step_parity_full_size(preset):
    cfg = configs.gate_exercising(configs.PRESETS[preset])
    B, P, G, BL, T = cfg["batch"], cfg["prompt_len"], cfg["gen_len"], cfg["block_len"], cfg["steps_per_block"]
    prompts = synth.prompts(cfg["prompt_seed"], B, P, cfg["mask_id"])
    m = model.create_model(cfg)
    try:
        s = cora.cora_session_create(m, B, prompts, P, G, BL, T, cfg["tau"], cfg["K"])
        try:
            cora.cora_denoise_step(s)
            out = cora.cora_session_read(s, B, P + G, G, BL)
        finally:
            cora.cora_session_destroy(s)
        assert cora.cora_device_error() == 0
    finally:
        cora.cora_model_destroy(m)
        torch.cuda.empty_cache()
    c_ref, a_ref, logits = oracle_first_step(cfg, prompts[0])
    c, a = out["conf"][0], out["argmax"][0]
    dc = np.abs(c - c_ref)
    assert dc.max() <= 2e-2, dc.max()
    sel = O.top2_margin(logits) > 2e-2
    assert sel.sum() >= 8, "too few rows with a clear top-1 to check the argmax"
    assert np.array_equal(a[sel], a_ref[sel])
    # The first step fixes exactly one position per sequence (k_0 = 1) and accepts none (m = 1).
    assert np.all(out["unmask"].sum(1) == 1) and np.all(out["accept"].sum(1) == 0)
    assert np.all(out["ctrl"][:, 2] == 1)
    print(f"{preset}: max|dc| = {dc.max():.2e}, argmax checked on {int(sel.sum())}/32 rows")
