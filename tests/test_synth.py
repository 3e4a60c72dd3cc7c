"""Pins for the seeded input generator (shared by both sides; no method arithmetic)."""

import numpy as np
import torch

from paper_2608_11235_gb300 import synth


def test_splitmix64_reference_outputs():
    """First outputs of SplitMix64 from state 0, as published with the generator."""
    assert [int(x) for x in synth.bits64(0, 0, 3)] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    assert int(synth.bits64(0, 2, 1)[0]) == 0x06C45D188009454F        # counter access = sequential access


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    f = np.concatenate([rng.normal(scale=s, size=20000) for s in (1e-3, 0.02, 1.0, 300.0)]).astype(np.float32)
    f = np.concatenate([f, np.array([1.00390625, 1.01171875, -1.00390625], np.float32)])   # exact ties
    ours = synth.f32_to_bf16_bits(f)
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_normal_moments_and_range():
    x = synth.bf16_bits_to_f32(synth.normal_bf16_bits(synth.stream_key(5, 9), 0, 400000, 0.02))
    assert abs(x.mean()) < 1e-4 and abs(x.std() - 0.02) < 2e-4
    assert np.abs(x).max() <= 0.02 * 262140 / synth.SD_X * 1.01


def test_uniform_int_range_and_prompts():
    p = synth.prompts(1, 3, 500, 2047)
    assert p.min() >= 0 and p.max() <= 2046 and not np.array_equal(p[0], p[1])
    u = synth.uniform01(synth.stream_key(2, 2), 0, 10000)
    assert 0 < u.min() and u.max() < 1 and abs(u.mean() - 0.5) < 0.02


def test_gate_inputs_shapes():
    h = synth.gate_history(1, 2, 32, 1000)
    assert h.shape == (8, 2, 32)
    keep = (h[1:] == h[:-1]).mean()
    assert 0.75 < keep < 0.86
    lg = synth.gate_logits_bf16(1, 2, 32, 1000, h[-1])
    assert lg.shape == (2, 32, 1000) and lg.dtype == np.uint16
