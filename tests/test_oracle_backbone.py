"""Pins for the oracle's backbone and Eq. 1, each against something other than itself.

RMSNorm, RoPE, attention and SwiGLU are checked against closed forms,
invariants and the complex-rotation form of RoPE; the whole layer stack is
checked against a scalar brute-force forward written with Python loops and
the math module on a micro model.
"""

import cmath
import math

import numpy as np
import pytest
from scipy.special import expit, softmax

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import synth


# --------------------------------------------------------------------- RMSNorm
def test_rmsnorm_closed_form_and_invariants():
    x = np.array([[3.0, 4.0]])
    y = O.rms_norm(x, np.ones(2), 0.0)
    r = math.sqrt((9 + 16) / 2)
    assert np.allclose(y, [[3 / r, 4 / r]], rtol=0, atol=1e-15)
    rng = np.random.default_rng(0)
    x = rng.normal(size=(5, 64))
    y = O.rms_norm(x, np.ones(64), 0.0)
    assert np.allclose(np.sqrt((y ** 2).mean(-1)), 1.0, atol=1e-12)          # unit RMS
    assert np.allclose(O.rms_norm(7.5 * x, np.ones(64), 0.0), y, atol=1e-12)  # scale invariance
    w = rng.normal(size=64)
    assert np.allclose(O.rms_norm(x, w, 0.0), y * w, atol=1e-12)              # weight is a per-channel gain


# ------------------------------------------------------------------------ RoPE
def test_rope_is_complex_rotation():
    """RoPE (Su et al.) multiplies (x_j + i x_{j+hd/2}) by exp(i pos theta^(-2j/hd))."""
    rng = np.random.default_rng(1)
    hd, theta = 8, 10000.0
    x = rng.normal(size=(5, 1, hd))
    pos = np.array([0, 1, 2, 17, 300])
    y = O.rope(x, pos, theta)
    for s in range(5):
        for j in range(hd // 2):
            z = complex(x[s, 0, j], x[s, 0, j + hd // 2]) * cmath.exp(1j * pos[s] * theta ** (-2 * j / hd))
            assert abs(y[s, 0, j] - z.real) < 1e-12 and abs(y[s, 0, j + hd // 2] - z.imag) < 1e-12


def test_rope_relative_position_property():
    rng = np.random.default_rng(2)
    q, k = rng.normal(size=(1, 1, 16)), rng.normal(size=(1, 1, 16))
    def dot(m, n):
        return float((O.rope(q, np.array([m]), 500.0) * O.rope(k, np.array([n]), 500.0)).sum())
    assert abs(dot(3, 10) - dot(103, 110)) < 1e-10
    assert abs(dot(0, 0) - float((q * k).sum())) < 1e-12
    assert np.allclose(O.rope(q, np.array([0]), 500.0), q)                     # identity at position 0


# ------------------------------------------------------------------- attention
def test_attention_special_cases():
    rng = np.random.default_rng(3)
    S, H, hd = 6, 2, 4
    v = rng.normal(size=(S, H, hd))
    k = rng.normal(size=(S, H, hd))
    out = O.attention(np.zeros((S, H, hd)), k, v)      # zero query -> uniform weights -> mean of v
    assert np.allclose(out, v.mean(0, keepdims=True).repeat(S, 0), atol=1e-12)
    q = rng.normal(size=(S, H, hd))
    perm = rng.permutation(S)                          # bidirectional: keys form a set
    assert np.allclose(O.attention(q, k[perm], v[perm]), O.attention(q, k, v), atol=1e-12)
    k2 = k.copy(); k2[-1] += 1.0                       # non-causal: the last key moves the first query
    assert not np.allclose(O.attention(q, k2, v)[0], O.attention(q, k, v)[0])


def test_attention_gqa_equals_repeated_heads():
    rng = np.random.default_rng(4)
    S, Hq, Hkv, hd = 5, 6, 2, 4
    q = rng.normal(size=(S, Hq, hd)); k = rng.normal(size=(S, Hkv, hd)); v = rng.normal(size=(S, Hkv, hd))
    rep = Hq // Hkv
    assert np.allclose(O.attention(q, k, v), O.attention(q, np.repeat(k, rep, 1), np.repeat(v, rep, 1)), atol=1e-12)


def test_attention_brute_force():
    rng = np.random.default_rng(5)
    S, H, hd = 4, 1, 3
    q, k, v = (rng.normal(size=(S, H, hd)) for _ in range(3))
    out = O.attention(q, k, v)
    for i in range(S):
        e = [math.exp(sum(q[i, 0, t] * k[j, 0, t] for t in range(hd)) / math.sqrt(hd)) for j in range(S)]
        z = sum(e)
        for t in range(hd):
            assert abs(out[i, 0, t] - sum(e[j] * v[j, 0, t] for j in range(S)) / z) < 1e-12


def test_silu():
    x = np.linspace(-30, 30, 101)
    assert np.allclose(O.silu(x), x * expit(x), atol=1e-12)
    assert O.silu(np.array([0.0]))[0] == 0.0


# ----------------------------------------------------- scalar brute-force forward
def _brute_forward(cfg, w, tokens):
    """Scalar-loop restatement of a pre-norm bidirectional Transformer."""
    S, d = len(tokens), cfg["d_model"]
    hq, hkv, hd, F = cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"], cfg["ffn"]
    eps, theta = cfg["norm_eps"], cfg["rope_theta"]
    h = [[float(w["embed"][t][c]) for c in range(d)] for t in tokens]

    def norm(row):
        r = math.sqrt(sum(a * a for a in row) / len(row) + eps)
        return [a / r for a in row]

    def lin(row, W):
        return [sum(row[c] * W[o][c] for c in range(len(row))) for o in range(len(W))]

    def rot(vec, pos):
        out = list(vec)
        for j in range(hd // 2):
            z = complex(vec[j], vec[j + hd // 2]) * cmath.exp(1j * pos * theta ** (-2 * j / hd))
            out[j], out[j + hd // 2] = z.real, z.imag
        return out

    for lw in w["layers"]:
        xs = [norm(r) for r in h]
        Q = [lin(x, lw["wq"]) for x in xs]; Kk = [lin(x, lw["wk"]) for x in xs]; Vv = [lin(x, lw["wv"]) for x in xs]
        att = [[0.0] * (hq * hd) for _ in range(S)]
        for head in range(hq):
            g = head // (hq // hkv)
            qs = [rot(Q[i][head * hd:(head + 1) * hd], i) for i in range(S)]
            ks = [rot(Kk[j][g * hd:(g + 1) * hd], j) for j in range(S)]
            for i in range(S):
                sc = [sum(qs[i][t] * ks[j][t] for t in range(hd)) / math.sqrt(hd) for j in range(S)]
                mx = max(sc)
                e = [math.exp(s - mx) for s in sc]
                z = sum(e)
                for t in range(hd):
                    att[i][head * hd + t] = sum(e[j] * Vv[j][g * hd + t] for j in range(S)) / z
        h = [[h[i][c] + y for c, y in enumerate(lin(att[i], lw["wo"]))] for i in range(S)]
        xs = [norm(r) for r in h]
        for i in range(S):
            gt, up = lin(xs[i], lw["w_gate"]), lin(xs[i], lw["w_up"])
            a = [gt[f] / (1 + math.exp(-gt[f])) * up[f] for f in range(F)]
            h[i] = [h[i][c] + y for c, y in enumerate(lin(a, lw["w_down"]))]
    logits = [lin(norm(r), w["lm_head"]) for r in h]
    return np.array(h), np.array(logits)


def test_forward_matches_scalar_brute_force(micro_cfg):
    cfg = dict(micro_cfg, n_layers=2)
    w = synth.model_weights_f64(cfg)
    tokens = np.array([3, 15, 15, 7, 0, 15, 11, 2, 15, 9])
    h = O.forward_hidden(cfg, w, tokens)
    hb, lb = _brute_forward(cfg, w, tokens)
    assert np.allclose(h, hb, rtol=0, atol=1e-10)
    assert np.allclose(O.lm_logits(cfg, w, h), lb, rtol=0, atol=1e-10)


def test_forward_is_bidirectional(micro_cfg):
    w = synth.model_weights_f64(micro_cfg)
    t1 = np.array([1, 2, 3, 4, 5, 6])
    t2 = t1.copy(); t2[-1] = 9
    assert not np.allclose(O.forward_hidden(micro_cfg, w, t1)[0], O.forward_hidden(micro_cfg, w, t2)[0])


# --------------------------------------------------------------------- Eq. 1
def test_top1_closed_forms():
    V = 64
    c, a = O.top1(np.zeros((1, V)))
    assert abs(c[0] - 1 / V) < 1e-15 and a[0] == 0          # uniform: c = 1/V, lowest id wins the tie
    for g in (0.5, 3.0, 12.0):
        l = np.zeros((1, V)); l[0, 17] = g
        c, a = O.top1(l)
        assert abs(c[0] - math.exp(g) / (math.exp(g) + V - 1)) < 1e-14 and a[0] == 17
    l = np.zeros((1, V)); l[0, 40] = 2.0; l[0, 9] = 2.0       # two-way tie: lowest id
    assert O.top1(l)[1][0] == 9
    rng = np.random.default_rng(6)
    l = rng.normal(scale=4, size=(20, 300))
    c, a = O.top1(l)
    p = softmax(l, axis=-1)
    assert np.allclose(c, p.max(-1), atol=1e-14) and np.array_equal(a, p.argmax(-1))
    c2, a2 = O.top1(l + 123.0)                                # shift invariance
    assert np.allclose(c, c2, atol=1e-13) and np.array_equal(a, a2)


def test_prop1_margin_bound_and_endpoint_preservation():
    """Prop. 1: c > 1/2 implies gamma >= log(c/(1-c)); a perturbation below gamma/2 keeps the top-1."""
    rng = np.random.default_rng(7)
    n_checked = 0
    for _ in range(400):
        V = int(rng.integers(2, 40))
        l = rng.normal(scale=3, size=V)
        l[rng.integers(V)] += rng.uniform(0, 8)
        c, a = O.top1(l[None])
        c, a = float(c[0]), int(a[0])
        srt = np.sort(l)
        gamma = srt[-1] - srt[-2]
        if c > 0.5:
            n_checked += 1
            assert gamma >= math.log(c / (1 - c)) - 1e-12
        delta = rng.uniform(-1, 1, size=V) * (0.499 * gamma)
        assert O.top1((l + delta)[None])[1][0] == a
    assert n_checked > 50


def test_drift_threshold_value_printed_in_paper():
    """Sec. 3.3 prints g(delta_p) = (1/2) log(delta_p / (1 - delta_p)) ~ 0.310 at delta_p = 0.65."""
    fixture = dict(line.split("=", 1) for line in open(
        __import__("os").path.join(__import__("os").path.dirname(__file__), "golden", "paper_values.txt"))
        .read().split("\n") if line and not line.startswith("#"))
    assert abs(0.5 * math.log(0.65 / 0.35) - float(fixture["g_at_0.65"])) < 5e-4
    # Table 1: the measured 1024/1024 GSM8K speedup is 92.7-99.5 % of the ideal 1/ratio.
    frac = float(fixture["gsm8k_1024_speedup"]) * float(fixture["gsm8k_1024_ratio"])
    assert 0.927 <= frac <= 0.995


def test_top2_margin_closed_forms():
    """p1 - p2 of softmax(l) (Eq. 1's distribution) against closed forms.

    A margin taken on logits, or from the third-largest probability, or
    without the softmax's normalisation, fails one of these."""
    V = 50
    assert abs(O.top2_margin(np.zeros((1, V)))[0]) < 1e-14                    # uniform: 0
    l = np.zeros((1, V)); l[0, 3] = 4.0; l[0, 31] = 4.0                        # exact two-way top tie: 0
    assert abs(O.top2_margin(l)[0]) < 1e-14
    for g in (0.25, 2.0, 9.0):                                                 # one boosted id over V-1 zeros
        l = np.zeros((1, V)); l[0, 11] = g
        want = (math.exp(g) - 1.0) / (math.exp(g) + V - 1)
        assert abs(O.top2_margin(l)[0] - want) < 1e-14
    for a, b in ((3.0, 1.0), (6.0, 5.5), (0.7, 0.2)):                          # two boosted ids a > b
        l = np.zeros((1, V)); l[0, 40] = a; l[0, 2] = b
        want = (math.exp(a) - math.exp(b)) / (math.exp(a) + math.exp(b) + V - 2)
        assert abs(O.top2_margin(l)[0] - want) < 1e-14
    l = np.array([[-30.0, 0.0]])                                               # two-id vocabulary
    assert abs(O.top2_margin(l)[0] - math.tanh(15.0)) < 1e-14


def test_top2_margin_batched_rows_and_shift():
    """[B, R, V] input gives the row-wise margins; a constant shift of a row changes nothing."""
    rng = np.random.default_rng(12)
    l = rng.normal(scale=3, size=(3, 5, 40))
    m = O.top2_margin(l)
    assert m.shape == (3, 5)
    for b in range(3):
        for r in range(5):
            p = np.sort(softmax(l[b, r]))
            assert abs(m[b, r] - (p[-1] - p[-2])) < 1e-14
    assert np.allclose(O.top2_margin(l + 57.0), m, rtol=0, atol=1e-13)
    assert np.all((m >= 0) & (m <= 1))
