"""GPU parity of each kernel of the path against the CPU oracle's definitions.

All inputs come from the seeded generator; expected values come from the
oracle (float64) on the same inputs.  Tolerances follow from the arithmetic:
bf16 outputs carry a relative rounding error of 2^-9, fp32 accumulation over
K <= 4096 adds ~1e-6 relative.
"""

import math

import numpy as np
import pytest
import torch

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import build, cora, synth

pytestmark = pytest.mark.gpu

BF16_RTOL = 2.0 ** -8


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    build.build()
    cora.lib()
    yield
    assert cora.cora_device_error(clear=True) == 0


def bits(seed, stream, shape, sigma):
    n = int(np.prod(shape))
    return synth.normal_bf16_bits(synth.stream_key(seed, stream), 0, n, sigma).reshape(shape)


def dev(b):
    return torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).cuda()


def f64(b):
    return synth.bf16_bits_to_f32(b).astype(np.float64)


def from_dev_bf16(t):
    return synth.bf16_bits_to_f32(t.cpu().numpy().view(np.uint16)).astype(np.float64)


def close_bf16(got, ref, atol_frac=1e-3):
    atol = atol_frac * float(np.sqrt(np.mean(ref ** 2)) + 1e-30)
    err = np.abs(got - ref) - (BF16_RTOL * np.abs(ref) + atol)
    assert err.max() <= 0, f"max excess {err.max():.3e} at {np.unravel_index(err.argmax(), err.shape)}"


# ------------------------------------------------------------------- synth
@pytest.mark.parametrize("seed,stream,sigma,start", [(0, 3, 0.02, 0), (2, 0x2107, 0.5, 12345), (11, 9, 0.0125, 7)])
def test_device_generator_bit_exact(seed, stream, sigma, start):
    n = 1 << 20
    key = synth.stream_key(seed, stream)
    t = torch.empty(n, dtype=torch.int16, device="cuda")
    cora.cora_synth_normal_bf16(t, n, key, start, float(synth.normal_scale_f32(sigma)))
    want = synth.normal_bf16_bits(key, start, n, sigma)
    assert np.array_equal(t.cpu().numpy().view(np.uint16), want)


# ----------------------------------------------------------------- RMSNorm
@pytest.mark.parametrize("M,d", [(1, 256), (97, 4096), (33, 3584), (5, 8192), (512, 4096), (607, 3584), (1000, 4096)])
def test_rmsnorm(M, d):
    x = f64(bits(1, 1, (M, d), 0.7)).astype(np.float32)
    w = bits(1, 2, (d,), 1.0)
    out = torch.empty((M, d), dtype=torch.int16, device="cuda")
    cora.cora_op_rmsnorm(torch.from_numpy(x).cuda(), dev(w), out, M, d, 1e-5)
    ref = O.rms_norm(x.astype(np.float64), f64(w), 1e-5)
    close_bf16(from_dev_bf16(out), ref)


# -------------------------------------------------------------------- GEMM
def run_gemm(A, Bm, M, N, K, epi, out_cols, out_dtype=torch.int16, C0=None, **kw):
    if C0 is not None:
        Ct = torch.from_numpy(C0.copy()).cuda()
    else:
        Ct = torch.zeros((M, out_cols), dtype=out_dtype, device="cuda")
    cora.cora_op_gemm(dev(A), dev(Bm), Ct, M, N, K, out_cols, epi, **kw)
    torch.cuda.synchronize()
    return Ct


@pytest.mark.parametrize("M,N,K", [(300, 512, 320), (128, 384, 64), (2048, 4096, 256), (256, 256, 4096),
                                   (96, 768, 256), (1, 256, 128), (512, 4096, 4096), (512, 12288, 1024),
                                   (96, 768, 2048), (128, 16384, 512),
                                   (64, 12288, 1024), (16, 4096, 4096), (5, 384, 640),    # few-row kernel
                                   (256, 12288, 1024),   # one row block, 48 pair-tiles: whole tiles on 48 pairs
                                   (2048, 12288, 256),   # 384 pair-tiles: stream-K + 4 data-parallel waves
                                   (1800, 10240, 192)])  # 320 pair-tiles, ragged last row block, 3 waves
def test_gemm_store(M, N, K):
    A = bits(2, 10, (M, K), 1.0)
    Bm = bits(2, 11, (N, K), 1.0 / math.sqrt(K))
    Ct = run_gemm(A, Bm, M, N, K, cora.EPI_STORE_BF16, N)
    close_bf16(from_dev_bf16(Ct), f64(A) @ f64(Bm).T)


@pytest.mark.parametrize("M,N,K", [(512, 4096, 4096),    # 32 pair-tiles: two k-pieces sharing the fix-up
                                   (96, 4096, 12288),    # 1-CTA: four skewed k-pieces, three partials per finisher
                                   (512, 12288, 4096),   # 96 pair-tiles over the SM pairs: stream-K
                                   (2048, 12288, 1024)])  # 384 pair-tiles: stream-K + data-parallel waves
def test_gemm_split_tiles_are_deterministic(M, N, K):
    A = bits(2, 20, (M, K), 1.0)
    Bm = bits(2, 21, (N, K), 1.0 / math.sqrt(K))
    c1 = run_gemm(A, Bm, M, N, K, cora.EPI_STORE_BF16, N).cpu().numpy()
    c2 = run_gemm(A, Bm, M, N, K, cora.EPI_STORE_BF16, N).cpu().numpy()
    assert np.array_equal(c1, c2)


@pytest.mark.parametrize("M,N,K", [(300, 512, 320), (130, 256, 1024), (512, 4096, 12288), (100, 16384, 512),
                                   (40, 4096, 12288), (64, 16384, 512),
                                   (256, 4096, 4096),    # one row block of 16 pair-tiles: two pieces sharing the fix-up
                                   (96, 4096, 4096),     # 1-CTA, 16 tiles: two pieces sharing the fix-up
                                   (96, 4096, 12288),    # 1-CTA, 16 tiles, K of 192 k-blocks: four skewed pieces
                                   (1536, 8192, 512)])  # 192 pair-tiles: stream-K + one data-parallel wave
def test_gemm_residual(M, N, K):
    A = bits(3, 10, (M, K), 1.0)
    Bm = bits(3, 11, (N, K), 1.0 / math.sqrt(K))
    H = f64(bits(3, 12, (M, N), 0.5)).astype(np.float32)
    Ct = run_gemm(A, Bm, M, N, K, cora.EPI_RESID_F32, N, C0=H)
    ref = H.astype(np.float64) + f64(A) @ f64(Bm).T
    assert np.abs(Ct.cpu().numpy() - ref).max() <= 1e-5 * np.abs(ref).max() + 1e-6


@pytest.mark.parametrize("M,F,K", [(300, 256, 256), (96, 768, 256), (48, 4096, 4096), (7, 768, 256),
                                   (1100, 10240, 128)])  # 400 pair-tiles, ragged: stream-K + 4 waves
def test_gemm_swiglu(M, F, K):
    A = bits(4, 10, (M, K), 1.0)
    g = bits(4, 11, (F, K), 1.0 / math.sqrt(K))
    u = bits(4, 12, (F, K), 1.0 / math.sqrt(K))
    il = np.empty((2 * F, K), np.uint16)          # [gate 128 | up 128] per group of 128 features
    for g0 in range(0, F, 128):
        il[2 * g0: 2 * g0 + 128] = g[g0: g0 + 128]
        il[2 * g0 + 128: 2 * g0 + 256] = u[g0: g0 + 128]
    Ct = run_gemm(A, il, M, 2 * F, K, cora.EPI_SWIGLU, F)
    ref = O.silu(f64(A) @ f64(g).T) * (f64(A) @ f64(u).T)
    close_bf16(from_dev_bf16(Ct), ref, atol_frac=2e-3)


def rope_table(seq, hd, theta):
    ang = O.rope_angles(np.arange(seq), hd, theta)
    return torch.from_numpy(np.stack([np.cos(ang), np.sin(ang)], -1).astype(np.float32)).cuda()


@pytest.mark.parametrize("B,S,H,Hkv,hd,theta", [(2, 96, 4, 4, 64, 1e4), (1, 300, 2, 1, 128, 5e5),
                                                  (1, 96, 4, 4, 64, 1e4), (1, 100, 2, 1, 128, 5e5),
                                                  (1, 48, 4, 4, 64, 1e4), (1, 60, 2, 1, 128, 5e5),
                                                  (1, 224, 32, 8, 128, 5e5)])  # one row block, 24 whole pair-tiles
def test_gemm_rope(B, S, H, Hkv, hd, theta):
    d = 256
    N = (H + 2 * Hkv) * hd
    M = B * S
    A = bits(5, 10, (M, d), 1.0)
    Wt = bits(5, 11, (N, d), 1.0 / math.sqrt(d))
    rope_cols = (H + Hkv) * hd
    Ct = run_gemm(A, Wt, M, N, d, cora.EPI_ROPE_BF16, N, rope=rope_table(S, hd, theta), seq=S, head_dim=hd,
                  rope_cols=rope_cols)
    y = (f64(A) @ f64(Wt).T).reshape(B, S, H + 2 * Hkv, hd)
    ref = np.empty_like(y)
    for b in range(B):
        ref[b, :, : H + Hkv] = O.rope(y[b, :, : H + Hkv], np.arange(S), theta)
        ref[b, :, H + Hkv:] = y[b, :, H + Hkv:]
    close_bf16(from_dev_bf16(Ct), ref.reshape(M, N))


# --------------------------------------------------------------- attention
# The last three head_dim-128 cases have more (sequence, head, query tile)
# items than a GB300 has SMs, so persistent CTAs run several items each
# (many key tiles per item; ragged; one key tile per item).
@pytest.mark.parametrize("B,S,Hq,Hkv,hd", [(2, 96, 4, 4, 64), (1, 200, 8, 2, 128), (1, 512, 2, 2, 128),
                                          (2, 130, 4, 2, 128), (1, 1, 2, 2, 128), (2, 300, 4, 4, 128),
                                          (3, 1, 2, 1, 64), (4, 768, 28, 4, 128), (2, 1000, 16, 4, 128),
                                          (40, 100, 8, 8, 128)])
def test_attention(B, S, Hq, Hkv, hd):
    W = (Hq + 2 * Hkv) * hd
    qkv = bits(6, 10, (B * S, W), 1.0)
    out = torch.zeros((B * S, Hq * hd), dtype=torch.int16, device="cuda")
    cora.cora_op_attention(dev(qkv), out, B, S, Hq, Hkv, hd)
    x = f64(qkv).reshape(B, S, Hq + 2 * Hkv, hd)
    ref = np.stack([O.attention(x[b, :, :Hq], x[b, :, Hq: Hq + Hkv], x[b, :, Hq + Hkv:]) for b in range(B)])
    got = from_dev_bf16(out).reshape(B, S, Hq, hd)
    # P is rounded to bf16 before the PV product (flash-attention style): 1e-2 relative budget.
    atol = 1e-2 * np.sqrt(np.mean(ref ** 2))
    assert np.abs(got - ref).max() <= atol + 1e-2 * np.abs(ref).max()


# Scores that jump far above everything seen earlier in a row: every even
# query row of every head is 2u (u a random +-1 vector), keys 40, 300 and S-1
# are 3u, 4u and 8u, so after the 1/sqrt(hd) scale those rows' scores rise by
# ~98, ~131 and ~261 (log2 units, hd 128) over the first keys' ~N(0, 1): the softmax
# reference must be raised inside the first key tile and in the last one
# (where O is rescaled).  One CTA per item (first and last case) and two
# query tiles per CTA (items > SMs); the last key tile is ragged.
@pytest.mark.parametrize("B,S,Hq,hd", [(1, 600, 2, 128), (2, 1000, 96, 128), (1, 300, 2, 64)])
def test_attention_score_jumps(B, S, Hq, hd):
    Hkv = Hq
    x = f64(bits(6, 13, (B, S, 3 * Hq, hd), 0.3))
    rng = np.random.default_rng(7)
    for b in range(B):
        for h in range(Hq):
            u = rng.choice([-1.0, 1.0], size=hd)
            x[b, 0::2, h] = 2.0 * u
            for key, scale in ((40, 3.0), (300 % S, 4.0), (S - 1, 8.0)):
                x[b, key, Hq + h] = scale * u
    qkv = (x.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)  # exact: every value is bf16
    assert np.array_equal(f64(qkv), x)
    out = torch.zeros((B * S, Hq * hd), dtype=torch.int16, device="cuda")
    cora.cora_op_attention(dev(qkv.reshape(B * S, 3 * Hq * hd)), out, B, S, Hq, Hkv, hd)
    ref = np.stack([O.attention(x[b, :, :Hq], x[b, :, Hq: 2 * Hq], x[b, :, 2 * Hq:]) for b in range(B)])
    got = from_dev_bf16(out).reshape(B, S, Hq, hd)
    assert np.all(np.isfinite(got))
    atol = 1e-2 * np.sqrt(np.mean(ref ** 2))
    assert np.abs(got - ref).max() <= atol + 1e-2 * np.abs(ref).max()


# Queries from an offset on (the rows a prefix-cache pass recomputes) against
# every key, with enough (sequence, head, query tile) items to run the
# persistent kernel (more items than SMs: 256, 320 and 448 here), a query
# start that is not a multiple of the tile, and ragged last tiles.
@pytest.mark.parametrize("B,S,Hq,Hkv,q_start", [(2, 1000, 32, 8, 488), (2, 1000, 32, 32, 480),
                                                (4, 544, 28, 4, 96), (1, 600, 8, 2, 32)])
def test_attention_query_rows(B, S, Hq, Hkv, q_start):
    hd = 128
    q_len = S - q_start
    W = (Hq + 2 * Hkv) * hd
    qkv = bits(6, 12, (B * S, W), 1.0)
    out = torch.zeros((B * q_len, Hq * hd), dtype=torch.int16, device="cuda")
    cora.cora_op_attention_rows(dev(qkv), out, B, S, Hq, Hkv, hd, q_start, q_len)
    x = f64(qkv).reshape(B, S, Hq + 2 * Hkv, hd)
    ref = np.stack([O.attention(x[b, :, :Hq], x[b, :, Hq: Hq + Hkv], x[b, :, Hq + Hkv:])[q_start:]
                    for b in range(B)])
    got = from_dev_bf16(out).reshape(B, q_len, Hq, hd)
    atol = 1e-2 * np.sqrt(np.mean(ref ** 2))
    assert np.abs(got - ref).max() <= atol + 1e-2 * np.abs(ref).max()


# ---------------------------------------------------------------- LM head
@pytest.mark.parametrize("R,V,d", [(32, 2048, 256), (5, 1000, 128), (256, 4096, 512), (128, 1088, 256),
                                   (32, 40000, 4096)])
def test_lm_head_top1(R, V, d):
    x = bits(7, 10, (R, d), 1.0)
    W = bits(7, 11, (V, d), 6.0 / math.sqrt(d))
    conf = torch.empty(R, dtype=torch.float32, device="cuda")
    arg = torch.empty(R, dtype=torch.int32, device="cuda")
    cora.cora_op_lm_head_top1(dev(x), dev(W), R, V, d, conf, arg)
    logits = f64(x) @ f64(W).T
    c_ref, a_ref = O.top1(logits)
    c, a = conf.cpu().numpy(), arg.cpu().numpy()
    assert np.abs(c - c_ref).max() <= 1e-4
    srt = np.sort(logits, -1)
    robust = (srt[:, -1] - srt[:, -2]) > 1e-3          # fp32 accumulation cannot swap these
    assert robust.mean() > 0.9
    assert np.array_equal(a[robust], a_ref[robust])
    assert np.all(a >= 0) and np.all(a < V)


# --------------------------------------------------- Eq. 1 from logits
@pytest.mark.parametrize("rows,V", [(64, 126464), (1, 126464), (300, 20000), (7, 1000), (3, 1001), (1, 1)])
def test_reduce_top1(rows, V):
    hist = synth.gate_history(5, 1, rows, V)
    lg = synth.gate_logits_bf16(5, 1, rows, V, hist[-1]).reshape(rows, V)
    conf = torch.empty(rows, dtype=torch.float32, device="cuda")
    arg = torch.empty(rows, dtype=torch.int32, device="cuda")
    lg_dev = dev(lg)
    cora.cora_reduce_top1(lg_dev, rows, V, conf, arg)
    c_ref, a_ref = O.top1(f64(lg))
    c, a = conf.cpu().numpy(), arg.cpu().numpy()
    assert np.all(np.abs(c - c_ref) <= 1e-4 * c_ref + 1e-7)
    assert np.array_equal(a, a_ref)      # bf16 logits compare exactly on both sides; lowest id wins ties
    conf.zero_()
    arg.zero_()
    cora.cora_reduce_top1(lg_dev, rows, V, conf, arg)   # second call: completion counters were left at zero
    assert np.array_equal(conf.cpu().numpy(), c) and np.array_equal(arg.cpu().numpy(), a)


# ----------------------------------------------------------- failure detection
@pytest.mark.parametrize("which,code", [(0, 0x102), (1, 0x104)])
def test_bounded_wait_reports_and_context_survives(which, code):
    """A wait that nothing completes (an mbarrier nobody arrives at, a flag
    nobody sets) gives up after the kernels' limit and reports its code; the
    context then runs a normal kernel."""
    assert cora.cora_check_wait_timeout(which) == code
    x = f64(bits(9, 1, (4, 256), 1.0)).astype(np.float32)
    out = torch.empty((4, 256), dtype=torch.int16, device="cuda")
    cora.cora_op_rmsnorm(torch.from_numpy(x).cuda(), None, out, 4, 256, 1e-5)
    close_bf16(from_dev_bf16(out), O.rms_norm(x.astype(np.float64), np.ones(256), 1e-5))
    assert cora.cora_device_error() == 0
