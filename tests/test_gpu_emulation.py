"""The full-size dense pass against a float32 reference with the kernels' bf16
rounding points (tests/bf16_emulation.py), per row, with a bar measured on
the reference itself.

Against the float64 oracle, bf16 rounding alone moves the gate-exercising
head's confidences by up to ~0.19 on these random models, so the oracle-side
bars of tests/test_gpu_fullsize.py are that wide.  Here the kernels are
compared with a reference that rounds to bf16 where they do (normalised
activations, Q/K/V after RoPE, softmax probabilities, attention output,
SwiGLU product, final rows) and computes the rest in float32.  That leaves
accumulation order, and on these models even that is not small: the bf16
roundings make the 32-layer pass chaotic, so two references that differ only
in accumulation order (every projection summed over the whole K, or in two or
four K slices) disagree by up to ~0.09 in the gate-exercising head's
confidences (final rows ~1 % apart).  Each case therefore computes the
reference and two alternatives, and holds the kernels to the reference:
  max |dc| <= max(floor, 3 x the largest max |dc| of an alternative)
  mean |dc| <= max(floor, 2 x the largest mean |dc| of an alternative)
  (floors: the stated 2e-2 / 5e-3 for the gate-exercising head; 1e-5 / 1e-6
  for the workload head, whose confidences are ~1e-3)
  argmax equal on every row where all references agree and the reference's
  top-1/top-2 logit gap exceeds 0.25 + 2 x the largest gap difference between
  them (at least 4 such rows for the gate-exercising head, 1 for the workload head),
for both LM heads, on the first step and on seeded mid-decode canvases set
into the batch the bench times (sequence 0), and on the prefix-cache pass,
including one whose attention runs the two-query-tile kernel on a query
range (more (sequence, head, query tile) items than SMs).
"""

import numpy as np
import pytest
import torch

import bf16_emulation as E
from paper_2608_11235_gb300 import build, configs, cora, model, synth

pytestmark = pytest.mark.gpu

# (block, fraction of the block resolved) of sequence 0's canvases; (0, None): the first step
CASES = {
    "llada8b-shape-256+256": [(0, None), (3, 0.5), (6, 0.75)],
    "dream7b-shape-256+512-b4": [(0, None), (10, 0.5)],
    "llada8b-shape-512+1024-b8": [(0, None), (23, 0.75)],
}
CANVAS_SEED = 500


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available()
    build.build()
    cora.lib()


def test_torch_generator_matches_synth_on_gpu():
    key = synth.stream_key(2, synth.tensor_stream(5, synth.WGATE))
    got = E.normal_bf16(key, 123_456_789, 100_000, 0.02, "cuda").view(torch.int16).cpu().numpy().view(np.uint16)
    assert np.array_equal(got, synth.normal_bf16_bits(key, 123_456_789, 100_000, 0.02))


def canvas(cfg, blk, frac):
    P, G, mask = cfg["prompt_len"], cfg["gen_len"], cfg["mask_id"]
    if frac is None:
        prompt = synth.prompts(cfg["prompt_seed"], 1, P, mask)[0].astype(np.int32)
        return np.concatenate([prompt, np.full(G, mask, np.int32)]), np.zeros(G, np.uint8)
    return synth.mid_decode_canvas(cfg, CANVAS_SEED, blk, frac)


# Floors of the bars (max, mean): the stated |dc| <= 2e-2 for the
# gate-exercising head (confidences across (0, 1)); for the workload head
# (confidences ~1e-3) only the measured spread counts.
FLOORS = {"gate_exercising": (2e-2, 5e-3), "workload": (1e-5, 1e-6)}
K_SPLITS = (2, 4)  # accumulation orders of the alternative references


def check_rows(label, head, c, a, ref, alts):
    """Kernel (c, a) against reference ``ref``; ``alts`` are the same reference
    in other accumulation orders, whose distance from ``ref`` sets the bar."""
    c_e, a_e, gap_e = ref
    spread_max = max(np.abs(c_e - alt[0]).max() for alt in alts)
    spread_mean = max(np.abs(c_e - alt[0]).mean() for alt in alts)
    gap_dev = max(np.abs(gap_e - alt[2]).max() for alt in alts)
    agree = np.all([a_e == alt[1] for alt in alts], axis=0)
    dc = np.abs(c - c_e)
    fmax, fmean = FLOORS[head]
    bar_max, bar_mean = max(fmax, 3 * spread_max), max(fmean, 2 * spread_mean)
    sel = agree & (gap_e > 0.25 + 2 * gap_dev)
    print(f"{label}: kernel vs bf16-point reference max|dc| {dc.max():.2e} mean {dc.mean():.2e}; "
          f"references max {spread_max:.2e} mean {spread_mean:.2e}; argmax on {int(sel.sum())}/{len(c)}")
    assert dc.max() <= bar_max and dc.mean() <= bar_mean, (label, dc.max(), dc.mean(), bar_max, bar_mean)
    assert sel.sum() >= (4 if head == "gate_exercising" else 1), label
    assert np.array_equal(a[sel], a_e[sel]), (label, np.flatnonzero(a[sel] != a_e[sel]))


@pytest.mark.parametrize("preset", list(CASES))
def test_dense_pass_against_bf16_point_reference(preset):
    base = configs.PRESETS[preset]
    B, P, G, BL, T = base["batch"], base["prompt_len"], base["gen_len"], base["block_len"], base["steps_per_block"]
    W = E.Weights(base)
    refs = {}
    heads = {"workload": W.head(base), "gate_exercising": W.head(configs.gate_exercising(base))}
    for blk, frac in CASES[preset]:
        tokens, _ = canvas(base, blk, frac)
        rows = slice(P + blk * BL, P + (blk + 1) * BL)
        xf = E.final_rows(W, tokens, rows)
        xalt = [E.final_rows(W, tokens, rows, k_split=ks) for ks in K_SPLITS]
        for head, hw in heads.items():
            refs[(blk, frac, head)] = (E.eq1(xf, hw), [E.eq1(x, hw) for x in xalt])
    del W
    torch.cuda.empty_cache()
    for head, cfg in (("workload", base), ("gate_exercising", configs.gate_exercising(base))):
        m = model.create_model(cfg)
        try:
            prompts = synth.prompts(cfg["prompt_seed"], B, P, cfg["mask_id"])
            fresh = np.concatenate([prompts, np.full((B, G), cfg["mask_id"], np.int32)], axis=1)
            s = cora.cora_session_create(m, B, prompts, P, G, BL, T, cfg["tau"], cfg["K"])
            try:
                for blk, frac in CASES[preset]:
                    tokens, state = canvas(cfg, blk, frac)
                    tok = fresh.copy()
                    tok[0] = tokens
                    st = np.zeros((B, G), np.uint8)
                    st[0] = state
                    ctrl = np.zeros((B, 4), np.int32)
                    ctrl[0] = [blk, min(int(state[blk * BL:(blk + 1) * BL].sum()), T - 1), 0, 0]
                    cora.cora_session_write(s, tokens=tok, state=st, persist=np.zeros((B, BL), np.int32),
                                            prev=np.full((B, BL), -1, np.int32), ctrl=ctrl)
                    c = np.zeros((B, BL), np.float32)
                    a = np.zeros((B, BL), np.int32)
                    cora.cora_denoise_step(s, -1, -1, c, a)
                    check_rows(f"{preset} block {blk} frac {frac} [{head}]", head, c[0], a[0],
                               *refs[(blk, frac, head)])
            finally:
                cora.cora_session_destroy(s)
            assert cora.cora_device_error() == 0
        finally:
            cora.cora_model_destroy(m)
            torch.cuda.empty_cache()


CACHED_CASES = {
    "llada8b-shape-256+256": [(3, 0.5), (6, 0.75)],
    # 288 recomputed rows x 32 heads x 8 sequences = 768 (sequence, head,
    # query tile) items: the persistent attention kernel, queries from an offset
    "llada8b-shape-512+1024-b8": [(23, 0.75)],
}


@pytest.mark.parametrize("preset", list(CACHED_CASES))
def test_prefix_cache_pass_against_bf16_point_reference(preset):
    """The cached pass (rows from the active block on, attending to the keys
    and values the block's dense first pass kept) in the batch the bench
    times, sequence 0 on a seeded mid-decode canvas, against the same
    reference computed the cached way."""
    base = configs.PRESETS[preset]
    B, P, G, BL, T = base["batch"], base["prompt_len"], base["gen_len"], base["block_len"], base["steps_per_block"]
    cases = CACHED_CASES[preset]
    W = E.Weights(base)
    refs = {}
    heads = {"workload": W.head(base), "gate_exercising": W.head(configs.gate_exercising(base))}
    for blk, frac in cases:
        first, _ = synth.mid_decode_canvas(base, CANVAS_SEED, blk, 0.0)
        tokens, _ = synth.mid_decode_canvas(base, CANVAS_SEED, blk, frac)
        lo = P + blk * BL
        xf = E.cached_final_rows(W, first, tokens, lo, slice(lo, lo + BL))
        xalt = [E.cached_final_rows(W, first, tokens, lo, slice(lo, lo + BL), k_split=ks) for ks in K_SPLITS]
        for head, hw in heads.items():
            refs[(blk, head)] = (E.eq1(xf, hw), [E.eq1(x, hw) for x in xalt])
    del W
    torch.cuda.empty_cache()
    for head, cfg in (("workload", base), ("gate_exercising", configs.gate_exercising(base))):
        m = model.create_model(cfg)
        try:
            prompts = synth.prompts(cfg["prompt_seed"], B, P, cfg["mask_id"])
            fresh = np.concatenate([prompts, np.full((B, G), cfg["mask_id"], np.int32)], axis=1)
            s = cora.cora_session_create(m, B, prompts, P, G, BL, T, cfg["tau"], cfg["K"],
                                         options=cora.decode_options(cache=cora.CACHE_PREFIX))
            try:
                for blk, frac in cases:
                    for f, step in ((0.0, 0), (frac, 1)):    # step 0: the dense first pass; then a cached one
                        tokens, state = synth.mid_decode_canvas(cfg, CANVAS_SEED, blk, f)
                        tok = fresh.copy()
                        tok[0] = tokens
                        st = np.zeros((B, G), np.uint8)
                        st[0] = state
                        ctrl = np.tile(np.array([[blk, step, 0, 0]], np.int32), (B, 1))
                        cora.cora_session_write(s, tokens=tok, state=st, persist=np.zeros((B, BL), np.int32),
                                                prev=np.full((B, BL), -1, np.int32), ctrl=ctrl)
                        c = np.zeros((B, BL), np.float32)
                        a = np.zeros((B, BL), np.int32)
                        cora.cora_denoise_step(s, blk, step, c, a)
                    check_rows(f"{preset} cached pass block {blk} frac {frac} [{head}]", head, c[0], a[0],
                               *refs[(blk, head)])
            finally:
                cora.cora_session_destroy(s)
            assert cora.cora_device_error() == 0
        finally:
            cora.cora_model_destroy(m)
            torch.cuda.empty_cache()
