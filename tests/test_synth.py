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


def test_fp32_weights_are_the_unrounded_product():
    """fp32-weight workloads keep X * scale; the bf16 workloads' values are its rounding."""
    key = synth.stream_key(0, synth.tensor_stream(0, synth.WQ))
    f = synth.normal_f32(key, 0, 50000, 0.02)
    assert f.dtype == np.float32
    assert np.array_equal(synth.normal_bf16_bits(key, 0, 50000, 0.02), synth.f32_to_bf16_bits(f))
    b = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(f))
    assert np.mean(b != f) > 0.95                       # almost none is bf16-representable
    rel = np.abs(b - f) / np.abs(f)
    assert rel.max() <= 2.0 ** -8 + 1e-12                # bf16 rounding: half an ulp, 8 significand bits
    cfg = dict(n_layers=1, d_model=8, n_heads=2, n_kv_heads=1, head_dim=4, ffn=12, vocab=16, mask_id=15,
               init_sigma=0.5, head_sigma=1.5, seed=7)
    w16 = synth.weight_f64(cfg, 0, synth.WQ)
    w32 = synth.weight_f64(dict(cfg, weight_dtype="f32"), 0, synth.WQ)
    assert np.array_equal(synth.f32_to_bf16_bits(w32.astype(np.float32)),
                          synth.f32_to_bf16_bits(w16.astype(np.float32)))
    assert not np.array_equal(w16, w32)


def test_torch_restatement_of_the_generator_matches():
    """The float32 bf16-point reference's torch generator (int64 wrap-around
    arithmetic) gives synth's bits, on the CPU here and on the GPU in its own test."""
    import bf16_emulation as E
    for seed, stream, start, n, sigma in ((2, 0x103, 0, 5000, 0.02), (11, 2, 7_777_777_777, 3000, 8 / 64.0),
                                          (0, 1, (1 << 40) + 3, 2000, 0.5)):
        key = synth.stream_key(seed, stream)
        got = E.normal_bf16(key, start, n, sigma, "cpu").view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(got, synth.normal_bf16_bits(key, start, n, sigma))
