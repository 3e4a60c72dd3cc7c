"""End-to-end decode on the GPU against the oracle (tiny two-layer model).

Replay parity: the oracle decodes with the tiny model's operating point
(tau = 0.9, K = 2); before each of its executed steps the GPU session is set
to the oracle's pre-step state (canvas, position states, persistence) and runs
one cora_denoise_step.  Eq. 1 must agree (|dc| <= 2e-2, argmax equal where
the oracle's top-1/top-2 probability margin exceeds 2e-2); the gate's output
must equal the oracle's wherever the measured confidence error cannot flip a
decision, and must follow the rule on the GPU's own confidences everywhere.

Closed forms on the GPU: the gate switched off gives the full horizon; an
accept-everything gate ends every block after one pass (K = 0) or two (K = 1).
"""

import numpy as np
import pytest
import torch

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import build, configs, cora, model, synth

pytestmark = pytest.mark.gpu
CFG = dict(configs.TINY)
P, G, BL, T = CFG["prompt_len"], CFG["gen_len"], CFG["block_len"], CFG["steps_per_block"]
TAU, K = CFG["tau"], CFG["K"]


@pytest.fixture(scope="module")
def tiny():
    assert torch.cuda.is_available()
    build.build()
    m = model.create_model(CFG, on_device_fill=False)
    w = synth.model_weights_f64(CFG)
    prompt = synth.prompts(CFG["prompt_seed"], 3, P, CFG["mask_id"])
    yield m, w, prompt
    cora.cora_model_destroy(m)
    assert cora.cora_device_error(clear=True) == 0


def rule_holds(before_state, persist_before, prev_before, conf, arg, k, tau, Kp, after):
    """The gate's output follows Eq. 2-4 on the GPU's own conf/argmax."""
    U = before_state == 0
    persist = np.where(U, np.where(prev_before == arg, persist_before + 1, 0), persist_before)
    idx = [i for i in np.argsort(-conf.astype(np.float64), kind="stable") if U[i]]
    Tm = np.zeros(len(U), bool)
    Tm[idx[:min(k, len(idx))]] = True
    A = U & ~Tm & (conf >= np.float32(tau)) & (persist >= Kp) & (Kp >= 0)
    return np.array_equal(after["unmask"].astype(bool), Tm) and np.array_equal(after["accept"].astype(bool), A)


def test_replay_parity_every_step(tiny):
    m, w, prompt = tiny
    tr = O.generate(CFG, w, prompt[0], G, BL, T, TAU, K, record=True)
    assert sum(len(s["result"].accepted) for s in tr.steps) > 0, "the gate should fire on the tiny model"
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, K)
    robust_steps = 0
    max_dc = 0.0
    try:
        for st in tr.steps:
            b0 = st["before"]
            ctrl = np.array([[st["block"], st["step"], st["passes_before"], 0]], np.int32)
            cora.cora_session_write(s, tokens=st["canvas"][None], state=st["gen_state"][None],
                                    persist=b0.persist[None], prev=b0.prev[None], ctrl=ctrl)
            c_step = np.full((1, BL), -1.0, np.float32)
            a_step = np.full((1, BL), -1, np.int32)
            d_step = np.full(1, 7, np.uint8)
            cora.cora_denoise_step(s, st["block"], st["step"], c_step, a_step, d_step)
            out = cora.cora_session_read(s, 1, P + G, G, BL)
            c, a = out["conf"][0], out["argmax"][0]
            # the step's own outputs are the session's Eq. 1 state and the gate's block-done flag
            assert np.array_equal(c_step[0], c) and np.array_equal(a_step[0], a)
            assert d_step[0] == int(not np.any(out["state"][0][st["block"] * BL:(st["block"] + 1) * BL] == 0))
            dc = np.abs(c - st["conf"])
            max_dc = max(max_dc, float(dc.max()))
            assert dc.max() <= 2e-2, (st["block"], st["step"], dc.max())
            sel = O.top2_margin(st["logits"]) > 2e-2
            assert np.array_equal(a[sel], st["x_hat"][sel])
            k = O.transfer_schedule(BL, T)[st["step"]]
            after = dict(unmask=out["unmask"][0], accept=out["accept"][0])
            assert rule_holds(b0.state, b0.persist, b0.prev, c, a, k, TAU, K, after)
            # Decisions the measured error cannot flip must equal the oracle's.
            eps = float(dc.max()) + 1e-6
            U = b0.state == O.UNRESOLVED
            cu = np.sort(st["conf"][U])[::-1]
            robust = np.array_equal(a[U], st["x_hat"][U])
            robust &= len(cu) <= k or k == 0 or (cu[k - 1] - cu[k]) > 2 * eps
            robust &= bool(np.all(np.abs(st["conf"][U] - TAU) > eps))
            if robust:
                robust_steps += 1
                r = st["result"]
                assert sorted(np.flatnonzero(out["unmask"][0])) == r.transferred
                assert sorted(np.flatnonzero(out["accept"][0])) == r.accepted
                lo = P + st["block"] * BL
                assert np.array_equal(out["tokens"][0][lo: lo + BL], st["after"].tokens)
                assert np.array_equal(out["state"][0][st["block"] * BL:(st["block"] + 1) * BL], st["after"].state)
                if not r.done:
                    assert np.array_equal(out["persist"][0], st["after"].persist)
                    assert out["ctrl"][0, 1] == st["step"] + 1
                else:
                    assert out["ctrl"][0, 0] == st["block"] + 1 and out["ctrl"][0, 1] == 0
    finally:
        cora.cora_session_destroy(s)
    print(f"replayed {len(tr.steps)} steps, {robust_steps} with flip-proof decisions, max|dc| = {max_dc:.2e}")


def test_batched_replay_on_the_2sm_gemm(tiny):
    """Three sequences at once: 3 x 96 = 288 rows, so every projection runs
    on the 2-CTA GEMM (the single-sequence replays use the 1-CTA and few-row
    kernels).  Step i of every sequence's oracle trace is replayed in one
    batched step, each sequence at its own block and step: Eq. 1 within 2e-2,
    argmax equal above the margin, the gate's rule on the GPU's own outputs."""
    m, w, prompt = tiny
    B = 3
    trs = [O.generate(CFG, w, prompt[b], G, BL, T, TAU, K, record=True) for b in range(B)]
    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, TAU, K)
    try:
        n = min(12, *(len(tr.steps) for tr in trs))
        max_dc = 0.0
        for i in range(n):
            sts = [tr.steps[i] for tr in trs]
            ctrl = np.array([[st["block"], st["step"], st["passes_before"], 0] for st in sts], np.int32)
            cora.cora_session_write(s, tokens=np.stack([st["canvas"] for st in sts]),
                                    state=np.stack([st["gen_state"] for st in sts]),
                                    persist=np.stack([st["before"].persist for st in sts]),
                                    prev=np.stack([st["before"].prev for st in sts]), ctrl=ctrl)
            cora.cora_denoise_step(s)
            out = cora.cora_session_read(s, B, P + G, G, BL)
            for b, st in enumerate(sts):
                c, a = out["conf"][b], out["argmax"][b]
                dc = np.abs(c - st["conf"])
                max_dc = max(max_dc, float(dc.max()))
                assert dc.max() <= 2e-2, (b, i, dc.max())
                sel = O.top2_margin(st["logits"]) > 2e-2
                assert np.array_equal(a[sel], st["x_hat"][sel]), (b, i)
                k = O.transfer_schedule(BL, T)[st["step"]]
                b0 = st["before"]
                assert rule_holds(b0.state, b0.persist, b0.prev, c, a, k, TAU, K,
                                  dict(unmask=out["unmask"][b], accept=out["accept"][b]))
    finally:
        cora.cora_session_destroy(s)
    print(f"batched replay: {n} steps x {B} sequences, max|dc| = {max_dc:.2e}")


def test_denoise_step_rejects_a_wrong_block_or_step(tiny):
    """cora_denoise_step(s, block, step, ...) checks the caller's (block, step)
    against the session before launching: a mismatch is CORA_ESTATE and
    leaves the state untouched; -1 skips the check."""
    m, _, prompt = tiny
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, K)
    try:
        cora.cora_denoise_step(s, 0, 0)
        before = cora.cora_session_read(s, 1, P + G, G, BL)
        assert before["ctrl"][0, :3].tolist() == [0, 1, 1]
        for blk, stp in ((1, 1), (0, 0), (0, 2)):
            with pytest.raises(cora.CoraError) as e:
                cora.cora_denoise_step(s, blk, stp)
            assert e.value.code == cora.CORA_ESTATE
        after = cora.cora_session_read(s, 1, P + G, G, BL)
        assert all(np.array_equal(before[k], after[k]) for k in before)
        cora.cora_denoise_step(s, 0, -1)
        cora.cora_denoise_step(s, -1, 2)
        assert cora.cora_session_read(s, 1, P + G, G, BL)["ctrl"][0, 2] == 3
    finally:
        cora.cora_session_destroy(s)


def test_fp32_weights_equal_their_bf16_rounding(tiny):
    """The tiny model's weights are fp32; the library rounds them to bf16 on
    the device (round to nearest even).  A model built from the host-rounded
    bf16 bits decodes to the same tokens and passes, and so does one built
    from device-resident fp32 tensors (read in place, no staging)."""
    m, _, prompt = tiny
    bits = {"embed": synth.f32_to_bf16_bits(synth.weight_f32(CFG, -1, synth.EMBED)),
            "lm_head": synth.f32_to_bf16_bits(synth.weight_f32(CFG, -1, synth.LM_HEAD))}
    for name, kind in model.KINDS.items():
        bits[name] = [synth.f32_to_bf16_bits(synth.weight_f32(CFG, l, kind)) for l in range(CFG["n_layers"])]
    m16 = cora.cora_model_create(CFG, bits)
    m32d = model.create_model(CFG, on_device_fill=True)
    try:
        ref = cora.cora_generate(m, prompt[:2], G, BL, T, TAU, K)
        for other in (m16, m32d):
            got = cora.cora_generate(other, prompt[:2], G, BL, T, TAU, K)
            assert np.array_equal(got[0], ref[0]) and np.array_equal(got[1], ref[1])
    finally:
        cora.cora_model_destroy(m16)
        cora.cora_model_destroy(m32d)


def test_gate_off_runs_full_horizon(tiny):
    m, _, prompt = tiny
    toks, passes, batched = cora.cora_generate(m, prompt[:1], G, BL, T, 2.0, 1)
    assert passes[0] == (G // BL) * T and batched == (G // BL) * T
    toks2, passes2, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 1.0, -1)
    assert passes2[0] == (G // BL) * T and np.array_equal(toks, toks2)


def test_accept_all_gate_closed_form(tiny):
    m, _, prompt = tiny
    _, passes, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 0.0, 0)      # every position on the first pass
    assert passes[0] == G // BL
    _, passes, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 0.0, 1)      # one persistence check: >= 2 passes
    assert 2 * (G // BL) <= passes[0] <= (G // BL) * T


@pytest.fixture(scope="module")
def sharp():
    cfg = dict(configs.TINY_SHARP)
    m = model.create_model(cfg)
    prompt = synth.prompts(cfg["prompt_seed"], 3, P, cfg["mask_id"])
    yield m, prompt
    cora.cora_model_destroy(m)


def test_sharp_model_decision_logic(sharp):
    """Sharp-attention variant: every executed step's gate output follows the
    rule on the GPU's own confidences, counts per block sum to the block
    length, and the special cases hold."""
    m, prompt = sharp
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, K)
    try:
        per_block = {}
        accepted = 0
        done = False
        while not done:
            before = cora.cora_session_read(s, 1, P + G, G, BL)
            done = cora.cora_denoise_step(s)
            out = cora.cora_session_read(s, 1, P + G, G, BL)
            blk, step = before["ctrl"][0, 0], before["ctrl"][0, 1]
            gstate = before["state"][0][blk * BL:(blk + 1) * BL]
            k = O.transfer_schedule(BL, T)[step]
            assert rule_holds(gstate, before["persist"][0], before["prev"][0], out["conf"][0], out["argmax"][0], k,
                              TAU, K, dict(unmask=out["unmask"][0], accept=out["accept"][0]))
            per_block[blk] = per_block.get(blk, 0) + int(out["unmask"][0].sum() + out["accept"][0].sum())
            accepted += int(out["accept"][0].sum())
        assert all(v == BL for v in per_block.values()) and len(per_block) == G // BL
        assert accepted > 0
    finally:
        cora.cora_session_destroy(s)
    _, passes, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 2.0, 1)
    assert passes[0] == (G // BL) * T
    _, passes, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 0.0, 0)
    assert passes[0] == G // BL


def test_free_running_decode_invariants(tiny):
    m, w, prompt = tiny
    toks, passes, batched = cora.cora_generate(m, prompt[:1], G, BL, T, TAU, K)
    assert 3 * (G // BL) <= passes[0] <= (G // BL) * T     # K = 2: no acceptance before a block's third pass
    assert np.all((toks >= 0) & (toks < CFG["vocab"]))
    tr = O.generate(CFG, w, prompt[0], G, BL, T, TAU, K)
    agree = float(np.mean(toks[0] == tr.tokens))
    print(f"free-running GPU vs oracle: {agree:.3f} token agreement, passes {passes[0]} vs {sum(tr.passes_per_block)}")


def test_batch_sequences_are_independent(tiny):
    m, _, prompt = tiny
    toks3, passes3, batched = cora.cora_generate(m, prompt, G, BL, T, TAU, K)
    assert batched == passes3.max()
    for b in range(3):
        toks1, passes1, _ = cora.cora_generate(m, prompt[b: b + 1], G, BL, T, TAU, K)
        assert passes1[0] == passes3[b]
        assert np.array_equal(toks1[0], toks3[b])


def test_device_loop_matches_host_steps(sharp):
    """cora_session_run (the whole decode as one graph launch with a WHILE
    node) executes exactly the steps of a host loop over cora_denoise_step,
    with identical results; it can run again after a reset."""
    m, prompt = sharp
    B = 3
    s_dev = cora.cora_session_create(m, B, prompt, P, G, BL, T, TAU, K)
    s_host = cora.cora_session_create(m, B, prompt, P, G, BL, T, TAU, K)
    try:
        steps, on_device = cora.cora_session_run(s_dev)
        assert on_device, "the decode should run as one device-side loop"
        host_steps, done = 0, False
        while not done:
            done = cora.cora_denoise_step(s_host)
            host_steps += 1
        assert steps == host_steps == cora.cora_session_batched_passes(s_dev)
        a = cora.cora_session_read(s_dev, B, P + G, G, BL)
        b = cora.cora_session_read(s_host, B, P + G, G, BL)
        for key in ("tokens", "state", "ctrl"):
            assert np.array_equal(a[key], b[key]), key
        assert np.all(a["ctrl"][:, 3] == 1) and a["ctrl"][:, 2].max() == steps
        with pytest.raises(cora.CoraError) as e:
            cora.cora_session_run(s_dev)
        assert e.value.code == cora.CORA_ESTATE
        cora.cora_session_reset(s_dev, prompt)
        steps2, _ = cora.cora_session_run(s_dev)
        assert steps2 == steps
        assert np.array_equal(cora.cora_session_read(s_dev, B, P + G, G, BL)["tokens"], a["tokens"])
    finally:
        cora.cora_session_destroy(s_dev)
        cora.cora_session_destroy(s_host)


def test_remaining_schedule_on_gpu(sharp):
    """Decoding option CORA_SCHEDULE_REMAINING: with the gate off it gives the
    fixed schedule's tokens (block length = horizon); with the gate on every
    executed step transfers ceil(|U| / (T - s)) positions and accepts by the
    rule, on the GPU's own confidences."""
    m, prompt = sharp
    rem = cora.decode_options(schedule=cora.SCHEDULE_REMAINING)
    t_fix, p_fix, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 2.0, 1)
    t_rem, p_rem, _ = cora.cora_generate(m, prompt[:1], G, BL, T, 2.0, 1, options=rem)
    assert np.array_equal(t_fix, t_rem) and np.array_equal(p_fix, p_rem)
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, K, options=rem)
    try:
        per_block, done = {}, False
        while not done:
            before = cora.cora_session_read(s, 1, P + G, G, BL)
            done = cora.cora_denoise_step(s)
            out = cora.cora_session_read(s, 1, P + G, G, BL)
            blk, step = before["ctrl"][0, 0], before["ctrl"][0, 1]
            gstate = before["state"][0][blk * BL:(blk + 1) * BL]
            k = O.remaining_step_count(int((gstate == 0).sum()), T, int(step))
            assert rule_holds(gstate, before["persist"][0], before["prev"][0], out["conf"][0], out["argmax"][0], k,
                              TAU, K, dict(unmask=out["unmask"][0], accept=out["accept"][0]))
            per_block[blk] = per_block.get(blk, 0) + int(out["unmask"][0].sum() + out["accept"][0].sum())
        assert all(v == BL for v in per_block.values()) and len(per_block) == G // BL
    finally:
        cora.cora_session_destroy(s)


def test_eos_stop_on_gpu(sharp):
    """Decoding option eos_id (EOS-aware stop), per sequence of a batch."""
    m, prompt = sharp
    B = prompt.shape[0]
    base, p_base, _ = cora.cora_generate(m, prompt, G, BL, T, TAU, K)
    eos = int(base[0, 0])                                   # committed by sequence 0 in its first block
    toks, passes, batched = cora.cora_generate(m, prompt, G, BL, T, TAU, K, options=cora.decode_options(eos_id=eos))
    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, TAU, K, options=cora.decode_options(eos_id=eos))
    try:
        cora.cora_session_run(s)
        st = cora.cora_session_read(s, B, P + G, G, BL)["state"]
    finally:
        cora.cora_session_destroy(s)
    stopped = 0
    for b in range(B):
        blocks = [i for i in range(G // BL) if np.any(base[b, i * BL:(i + 1) * BL] == eos)]
        if not blocks or blocks[0] == G // BL - 1:
            assert np.array_equal(toks[b], base[b]) and passes[b] == p_base[b]
            continue
        fb = blocks[0]
        end = (fb + 1) * BL
        assert np.array_equal(toks[b, :end], base[b, :end])
        assert np.all(toks[b, end:] == eos) and np.all(st[b, end:] == 3)
        assert passes[b] < p_base[b]
        stopped += 1
    assert stopped >= 1 and batched == passes.max()


def test_disagreement_counts_on_gpu(sharp):
    """cora_session_disagreement against the definitions (Sec. 4) applied to
    the two sessions' canvases on the host; integer counts, so exact."""
    m, prompt = sharp
    B = prompt.shape[0]
    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, TAU, K)
    d = cora.cora_session_create(m, B, prompt, P, G, BL, T, 2.0, 1)     # gate off: the dense endpoint
    try:
        cora.cora_session_run(s)
        cora.cora_session_run(d)
        n_acc, n_ad, n_od = cora.cora_session_disagreement(s, d, B)
        a = cora.cora_session_read(s, B, P + G, G, BL)
        ref = cora.cora_session_read(d, B, P + G, G, BL)["tokens"][:, P:]
        for b in range(B):
            tok, st = a["tokens"][b, P:], a["state"][b]
            l_acc, l_out = O.disagreement(tok, st, ref[b])
            assert n_acc[b] == int((st == O.ACCEPTED).sum()) > 0
            assert l_acc == n_ad[b] / max(1, n_acc[b]) and l_out == n_od[b] / G
        z = cora.cora_session_disagreement(d, d, B)
        assert all(int(v.sum()) == 0 for v in z)
    finally:
        cora.cora_session_destroy(s)
        cora.cora_session_destroy(d)


@pytest.mark.parametrize("Kp", [0, -1])
def test_carry_equals_block_when_persistence_cannot_matter_gpu(sharp, Kp):
    m, prompt = sharp
    carry = cora.decode_options(persistence=cora.PERSIST_CARRY)
    a = cora.cora_generate(m, prompt, G, BL, T, TAU, Kp)
    b = cora.cora_generate(m, prompt, G, BL, T, TAU, Kp, options=carry)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_carry_persistence_on_gpu(sharp):
    """CORA_PERSIST_CARRY: Eq. 1 runs on every generation row; every executed
    step updates Eq. 2 for every unresolved position (the active block through
    the gate, which follows the rule on the carried counters), and counters
    are never reset at a block's end."""
    m, prompt = sharp
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, 1,
                                 options=cora.decode_options(persistence=cora.PERSIST_CARRY))
    try:
        done, first_pass_accepts = False, 0
        while not done:
            bf = cora.cora_session_read(s, 1, P + G, G, BL, eq1_rows=G)
            done = cora.cora_denoise_step(s)
            af = cora.cora_session_read(s, 1, P + G, G, BL, eq1_rows=G)
            blk, step = bf["ctrl"][0, 0], bf["ctrl"][0, 1]
            lo, hi = blk * BL, (blk + 1) * BL
            st0 = bf["state"][0]
            k = O.transfer_schedule(BL, T)[step]
            assert rule_holds(st0[lo:hi], bf["persist"][0, lo:hi], bf["prev"][0, lo:hi], af["conf"][0, lo:hi],
                              af["argmax"][0, lo:hi], k, TAU, 1, dict(unmask=af["unmask"][0], accept=af["accept"][0]))
            if step == 0:
                first_pass_accepts += int(af["accept"][0].sum())
            out = np.ones(G, bool)
            out[lo:hi] = False
            U = out & (st0 == 0)
            want = np.where(bf["prev"][0] == af["argmax"][0], bf["persist"][0] + 1, 0)
            assert np.array_equal(af["persist"][0][U], want[U]) and np.array_equal(af["prev"][0][U], af["argmax"][0][U])
            keep = out & (st0 != 0)
            assert np.array_equal(af["persist"][0][keep], bf["persist"][0][keep])
            # active block: carried, never reset
            Ub = st0[lo:hi] == 0
            assert np.array_equal(af["prev"][0, lo:hi][Ub], af["argmax"][0, lo:hi][Ub])
        print(f"carry: {first_pass_accepts} positions accepted on a block's first pass")
    finally:
        cora.cora_session_destroy(s)


def replay_compare(m, cfg, w, prompt, options, label):
    """Replay the oracle's prefix-cache decode step by step: the GPU session is
    set to the oracle's pre-step state (a block's step 0 makes the pass dense,
    which keeps the keys/values; later steps reuse them), then Eq. 1 and the
    gate must agree."""
    tr = O.generate(cfg, w, prompt[0], G, BL, T, TAU, K, record=True, cache="prefix")
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, K, options=options)
    max_dc, cached = 0.0, 0
    try:
        for st in tr.steps:
            b0 = st["before"]
            ctrl = np.array([[st["block"], st["step"], st["passes_before"], 0]], np.int32)
            cora.cora_session_write(s, tokens=st["canvas"][None], state=st["gen_state"][None],
                                    persist=b0.persist[None], prev=b0.prev[None], ctrl=ctrl)
            cora.cora_denoise_step(s)
            out = cora.cora_session_read(s, 1, P + G, G, BL)
            c, a = out["conf"][0], out["argmax"][0]
            dc = np.abs(c.astype(np.float64) - st["conf"])
            max_dc = max(max_dc, float(dc.max()))
            assert dc.max() <= 2e-2, (label, st["block"], st["step"], dc.max())
            sel = O.top2_margin(st["logits"]) > 2e-2
            assert np.array_equal(a[sel], st["x_hat"][sel]), (label, st["block"], st["step"])
            k = O.transfer_schedule(BL, T)[st["step"]]
            assert rule_holds(b0.state, b0.persist, b0.prev, c, a, k, TAU, K,
                              dict(unmask=out["unmask"][0], accept=out["accept"][0]))
            cached += st["step"] > 0
    finally:
        cora.cora_session_destroy(s)
    blocks = {st["block"] for st in tr.steps}
    print(f"{label}: replayed {len(tr.steps)} steps ({cached} cached passes, blocks {sorted(blocks)}), "
          f"max|dc| = {max_dc:.2e}")
    assert cached >= 2 and len(blocks) == G // BL


def test_prefix_cache_matches_oracle(tiny):
    m, w, prompt = tiny
    replay_compare(m, CFG, w, prompt, cora.decode_options(cache=cora.CACHE_PREFIX), "prefix cache, hd 64")


def test_prefix_cache_matches_oracle_hd128():
    cfg = dict(CFG, name="tiny-hd128", n_heads=2, n_kv_heads=2, head_dim=128)
    m = model.create_model(cfg, on_device_fill=False)
    try:
        w = synth.model_weights_f64(cfg)
        prompt = synth.prompts(cfg["prompt_seed"], 1, P, cfg["mask_id"])
        replay_compare(m, cfg, w, prompt, cora.decode_options(cache=cora.CACHE_PREFIX), "prefix cache, hd 128")
    finally:
        cora.cora_model_destroy(m)


def test_profile_step_runs_the_cached_pass(tiny):
    """cora_session_profile_step runs the pass the next step would run: on a
    prefix-cache session after a block's dense first pass, the pass over the
    rows from the block on.  Same pre-step state through the profiled eager
    pass and through cora_denoise_step: identical Eq. 1 outputs and state."""
    m, _, prompt = tiny
    s = cora.cora_session_create(m, 1, prompt[:1], P, G, BL, T, TAU, K,
                                 options=cora.decode_options(cache=cora.CACHE_PREFIX))
    try:
        cora.cora_denoise_step(s, 0, 0)                       # block 0's dense first pass
        st = cora.cora_session_read(s, 1, P + G, G, BL)
        prof = cora.cora_session_profile_step(s, CFG["n_layers"])
        assert len(prof) == 4 + 7 * CFG["n_layers"]
        a = cora.cora_session_read(s, 1, P + G, G, BL)
        cora.cora_session_write(s, tokens=st["tokens"], state=st["state"], persist=st["persist"], prev=st["prev"],
                                ctrl=st["ctrl"])
        cora.cora_denoise_step(s, 0, 1)                       # the same cached pass through the graph
        b = cora.cora_session_read(s, 1, P + G, G, BL)
        for key in ("conf", "argmax", "tokens", "state", "persist", "prev", "unmask", "accept"):
            assert np.array_equal(a[key], b[key]), key
        assert a["ctrl"][0, :2].tolist() == b["ctrl"][0, :2].tolist()
    finally:
        cora.cora_session_destroy(s)


def test_prefix_cache_batch_moves_blocks_together(sharp):
    """Prefix-cache sessions move a batch's sequences to the next block
    together: unfinished sequences always share the block index, a sequence
    whose block has ended waits with its canvas untouched, its executed-pass
    count grows only while it works, and the decode ends fully resolved."""
    m, prompt = sharp
    B = prompt.shape[0]
    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, TAU, K,
                                 options=cora.decode_options(cache=cora.CACHE_PREFIX))
    try:
        active_steps = np.zeros(B, np.int64)
        waited = 0
        done = False
        while not done:
            bf = cora.cora_session_read(s, B, P + G, G, BL)
            done = cora.cora_denoise_step(s)
            af = cora.cora_session_read(s, B, P + G, G, BL)
            live = bf["ctrl"][:, 3] == 0
            assert len(set(bf["ctrl"][live, 0])) <= 1                      # one block for the batch
            for b in np.flatnonzero(live):
                if bf["ctrl"][b, 1] < 0:                                   # waiting: nothing changes
                    waited += 1
                    assert np.array_equal(af["tokens"][b], bf["tokens"][b])
                    assert np.array_equal(af["state"][b], bf["state"][b])
                    assert af["ctrl"][b, 2] == bf["ctrl"][b, 2]
                else:
                    active_steps[b] += 1
        out = cora.cora_session_read(s, B, P + G, G, BL)
        assert np.array_equal(out["ctrl"][:, 2], active_steps)
        assert np.all(out["state"] != 0) and np.all(out["ctrl"][:, 3] == 1)
        print(f"prefix-cache batch: {waited} waiting sequence-steps, passes {active_steps.tolist()}")
    finally:
        cora.cora_session_destroy(s)


@pytest.mark.parametrize("frac", [0.05, 0.5, 0.9])
def test_checkpoint_and_resume_in_a_new_session(sharp, frac):
    """Checkpoint/resume at step granularity: a decode stopped after some
    steps, its state read out (canvas, position states, persistence, previous
    predictions, block/step/pass counters) and written into a fresh session
    continues to the same tokens and pass counts as an uninterrupted decode
    (the kernels are deterministic, so equality is exact)."""
    m, prompt = sharp
    B = prompt.shape[0]
    cfg = dict(configs.TINY_SHARP)
    tau, Kp = cfg["tau"], cfg["K"]

    def run_to_end(s):
        n = 1
        while not cora.cora_denoise_step(s):
            n += 1
            assert n <= (G // BL) * T
        return cora.cora_session_read(s, B, P + G, G, BL), n

    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, tau, Kp)
    try:
        ref, n_steps = run_to_end(s)
    finally:
        cora.cora_session_destroy(s)
    stop_after = max(1, min(n_steps - 1, int(frac * n_steps)))
    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, tau, Kp)
    try:
        for _ in range(stop_after):
            assert not cora.cora_denoise_step(s)
        ck = cora.cora_session_read(s, B, P + G, G, BL)
    finally:
        cora.cora_session_destroy(s)
    s = cora.cora_session_create(m, B, prompt, P, G, BL, T, tau, Kp)
    try:
        cora.cora_session_write(s, tokens=ck["tokens"], state=ck["state"], persist=ck["persist"], prev=ck["prev"],
                                ctrl=ck["ctrl"])
        out, n_rest = run_to_end(s)
    finally:
        cora.cora_session_destroy(s)
    assert stop_after + n_rest == n_steps
    assert np.array_equal(out["tokens"], ref["tokens"])
    assert np.array_equal(out["state"], ref["state"])
    assert np.array_equal(out["ctrl"], ref["ctrl"])  # block, step, passes executed, finished
    assert cora.cora_device_error() == 0
