"""Pins for the decoding variants (ablations of Sec. 3): the remaining-steps
transfer schedule and the EOS-aware stop.

remaining_step_count fixes ceil(|U| / (T - s)) positions at step s.  Pinned by
its defining properties: it resolves any block within the horizon, equals the
fixed schedule when nothing is accepted and T divides the block length, and
the decode loop applies it step by step (recorded traces).
"""

import numpy as np
import pytest

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import synth

G, T = 8, 4


@pytest.fixture(scope="module")
def model(micro_cfg):
    return micro_cfg, synth.model_weights_f64(micro_cfg)


@pytest.fixture(scope="module")
def prompt(micro_cfg):
    return synth.prompts(3, 1, 6, micro_cfg["mask_id"])[0]


def test_remaining_count_values():
    assert O.remaining_step_count(8, 4, 0) == 2
    assert O.remaining_step_count(3, 4, 1) == 1      # after acceptances: fewer than the fixed schedule's 2
    assert O.remaining_step_count(5, 4, 3) == 5      # the last step fixes everything left
    assert O.remaining_step_count(0, 4, 2) == 0


@pytest.mark.parametrize("Tn", [1, 2, 3, 4, 7])
def test_remaining_schedule_resolves_within_horizon(Tn):
    for n in range(0, 3 * Tn + 1):
        rem = n
        for s in range(Tn):
            k = O.remaining_step_count(rem, Tn, s)
            assert (k >= 1) == (rem > 0)
            rem -= min(k, rem)
        assert rem == 0
        if n % Tn == 0:                                  # dense and divisible: the fixed schedule
            rem, ks = n, []
            for s in range(Tn):
                ks.append(O.remaining_step_count(rem, Tn, s))
                rem -= ks[-1]
            assert ks == O.transfer_schedule(n, Tn)


@pytest.mark.parametrize("BL", [4, 8])
def test_remaining_equals_fixed_with_the_gate_off(model, prompt, BL):
    cfg, w = model
    a = O.generate(cfg, w, prompt, G, BL, T, 2.0, 1)
    b = O.generate(cfg, w, prompt, G, BL, T, 2.0, 1, schedule="remaining")
    assert np.array_equal(a.tokens, b.tokens) and a.passes_per_block == b.passes_per_block


@pytest.mark.parametrize("tau,K", [(0.3, 1), (0.5, 0), (0.2, 2)])
def test_remaining_schedule_trace(model, prompt, tau, K):
    cfg, w = model
    BL = 8
    tr = O.generate(cfg, w, prompt, G, BL, T, tau, K, record=True, schedule="remaining")
    per_block = {}
    for s in tr.steps:
        U0 = s["before"].state == O.UNRESOLVED
        k = O.remaining_step_count(int(U0.sum()), T, s["step"])
        assert sorted(s["result"].transferred) == O.transfer_set(s["conf"], U0, k)
        per_block[s["block"]] = per_block.get(s["block"], 0) + len(s["result"].transferred) + len(s["result"].accepted)
    assert all(v == BL for v in per_block.values())
    assert all(1 <= p <= T for p in tr.passes_per_block)


def test_eos_stop_after_the_block_that_commits_it(model, prompt):
    """EOS-aware stop: with eos_id = a token the plain decode commits in
    block b (and none earlier), the decode is identical through block b, then
    every later position is the EOS id and the later blocks run no pass; an
    EOS id that is never committed changes nothing."""
    cfg, w = model
    BL = 4
    base = O.generate(cfg, w, prompt, G, BL, T, 0.3, 1)
    nb = G // BL
    first = {}
    for b in range(nb):
        for t in base.tokens[b * BL:(b + 1) * BL]:
            first.setdefault(int(t), b)
    for eos, b in sorted(first.items(), key=lambda kv: kv[1]):
        tr = O.generate(cfg, w, prompt, G, BL, T, 0.3, 1, eos_id=eos)
        assert np.array_equal(tr.tokens[:(b + 1) * BL], base.tokens[:(b + 1) * BL])
        assert np.all(tr.tokens[(b + 1) * BL:] == eos)
        assert tr.passes_per_block == base.passes_per_block[:b + 1] + [0] * (nb - b - 1)
    unused = next(v for v in range(cfg["vocab"]) if v not in first)
    tr = O.generate(cfg, w, prompt, G, BL, T, 0.3, 1, eos_id=unused)
    assert np.array_equal(tr.tokens, base.tokens) and tr.passes_per_block == base.passes_per_block


def test_disagreement_definitions():
    tok = np.array([5, 1, 2, 3, 9, 9])
    ref = np.array([5, 1, 7, 3, 9, 0])
    st = np.array([O.TRANSFERRED, O.ACCEPTED, O.ACCEPTED, O.TRANSFERRED, O.ACCEPTED, O.TRANSFERRED])
    l_acc, l_out = O.disagreement(tok, st, ref)
    assert l_acc == 1 / 3 and l_out == 2 / 6               # accepted 1, 2, 4: only 2 differs; 2 and 5 differ overall
    assert O.disagreement(tok, np.zeros(6, np.uint8), ref) == (0.0, 2 / 6)   # nothing accepted: L_acc = 0


def test_disagreement_gate_off_is_zero(model, prompt):
    cfg, w = model
    dense, _ = O.dense_decode(cfg, w, prompt, G, 4, T)
    tr = O.generate(cfg, w, prompt, G, 4, T, 2.0, 1, record=True)
    st = np.zeros(G, np.uint8)
    for s in tr.steps:
        st[s["block"] * 4:(s["block"] + 1) * 4] = s["after"].state
    assert O.disagreement(tr.tokens, st, dense) == (0.0, 0.0)


@pytest.mark.parametrize("K", [0, -1])
def test_carry_equals_block_when_persistence_cannot_matter(model, prompt, K):
    """K = 0 accepts whatever the count, K = inf never accepts: the counters'
    starting point cannot change the decode."""
    cfg, w = model
    a = O.generate(cfg, w, prompt, G, 4, T, 0.3, K)
    b = O.generate(cfg, w, prompt, G, 4, T, 0.3, K, persistence="carry")
    assert np.array_equal(a.tokens, b.tokens) and a.passes_per_block == b.passes_per_block


@pytest.mark.parametrize("tau,K", [(0.3, 1), (0.2, 2), (0.0, 1)])
def test_carry_counters_brute_force(model, prompt, tau, K):
    """Carry mode: after every executed step the counter of each position of
    the active block that was unresolved equals the trailing run length - 1 of
    its top-1 predictions over ALL executed passes so far (recomputed here by
    replaying the recorded canvases through the forward)."""
    cfg, w = model
    BL, P = 4, len(prompt)
    tr = O.generate(cfg, w, prompt, G, BL, T, tau, K, record=True, persistence="carry")
    hist = []
    for s in tr.steps:
        h = O.forward_hidden(cfg, w, s["canvas"])
        hist.append(O.top1(O.lm_logits(cfg, w, h[P:]))[1])
        H = np.array(hist)                                   # [passes so far, G]
        U0 = s["before"].state == O.UNRESOLVED
        for i in np.flatnonzero(U0):
            j = s["block"] * BL + i
            run = 1
            while run < len(H) and H[-1 - run, j] == H[-1, j]:
                run += 1
            assert s["after"].persist[i] == run - 1, (s["block"], s["step"], i)
    assert any(s["step"] == 0 and s["result"].accepted for s in tr.steps) or K != 1 or tau > 0.0


def test_prefix_layer_with_empty_prefix_is_the_dense_layer(model):
    cfg, w = model
    rng = np.random.default_rng(0)
    h = rng.normal(size=(7, cfg["d_model"]))
    e = np.zeros((0, cfg["n_kv_heads"], cfg["head_dim"]))
    out, _, _ = O.layer_forward_prefix(cfg, w["layers"][0], h, np.arange(7), e, e)
    assert np.allclose(out, O.layer_forward(cfg, w["layers"][0], h, np.arange(7)), rtol=0, atol=1e-12)


@pytest.mark.parametrize("lo", [0, 3, 6, 13])
def test_cache_of_the_same_canvas_reproduces_the_dense_rows(model, prompt, lo):
    """Keys/values cached from a canvas, reused for that same canvas, give the
    dense pass's rows exactly (the approximation only enters once the canvas
    changes after the cache was taken)."""
    cfg, w = model
    x = np.concatenate([prompt, np.full(G, cfg["mask_id"])])
    x[8:10] = [2, 5]
    h_dense = O.forward_hidden(cfg, w, x)
    h_kv, cache = O.forward_hidden_kv(cfg, w, x)
    assert np.allclose(h_kv, h_dense, rtol=0, atol=1e-12)
    assert np.allclose(O.forward_hidden_cached(cfg, w, x, cache, lo), h_dense[lo:], rtol=0, atol=1e-12)


def test_prefix_cache_decode(model, prompt):
    """Cached decode: every block's first pass is the dense pass of its canvas;
    with no prompt and a single block every pass recomputes every row, so the
    decode equals the uncached one; trace invariants hold."""
    cfg, w = model
    BL = 4
    tr = O.generate(cfg, w, prompt, G, BL, T, 0.3, 1, record=True, cache="prefix")
    for s in tr.steps:
        if s["step"] == 0:
            lo = len(prompt) + s["block"] * BL
            ref = O.lm_logits(cfg, w, O.forward_hidden(cfg, w, s["canvas"])[lo: lo + BL])
            assert np.allclose(s["logits"], ref, rtol=0, atol=1e-10)
    per_block = {}
    for s in tr.steps:
        per_block[s["block"]] = per_block.get(s["block"], 0) + len(s["result"].transferred) + len(s["result"].accepted)
    assert all(v == BL for v in per_block.values())
    a = O.generate(cfg, w, prompt[:0], 8, 8, T, 0.3, 1)
    b = O.generate(cfg, w, prompt[:0], 8, 8, T, 0.3, 1, cache="prefix")
    assert np.array_equal(a.tokens, b.tokens) and a.passes_per_block == b.passes_per_block
