"""GPU parity of the transfer rule + residual gate (Eq. 2-4) and of the fused
Eq. 1 reduction + gate on the gate-isolation workload: bf16 logits
[B, 32, 126464] of Gumbel noise plus a boosted target, a seeded 8-step argmax
history (persistence) and a half-masked state, B in {1, 8, 64}."""

import numpy as np
import pytest
import torch

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import build, configs, cora, synth

pytestmark = pytest.mark.gpu
GI = configs.GATE_ISOLATION


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available()
    build.build()
    cora.lib()


def gate_state(seed, B, R, V):
    hist = synth.gate_history(seed, B, R, V, GI["n_hist"], GI["keep"])
    persist, prev = O.persist_from_history(hist)
    unresolved = synth.gate_unresolved(seed, B, R, GI["masked_frac"])
    state = np.where(unresolved, 0, 1 + (np.arange(B * R).reshape(B, R) % 2)).astype(np.uint8)
    tokens = np.where(unresolved, V - 1, hist[-1]).astype(np.int64)
    return hist, persist, prev, state, tokens


def to_dev(a, dt):
    return torch.from_numpy(np.ascontiguousarray(a).astype(dt)).cuda()


def run_gpu_gate(conf, arg, tokens, state, persist, prev, k, tau, K, R=None):
    B, Rr = conf.shape
    d = dict(conf=to_dev(conf, np.float32), argmax=to_dev(arg, np.int32), prev=to_dev(prev, np.int32),
             persist=to_dev(persist, np.int32), state=to_dev(state, np.uint8), tokens=to_dev(tokens, np.int32),
             unmask=torch.zeros((B, Rr), dtype=torch.uint8, device="cuda"),
             accept=torch.zeros((B, Rr), dtype=torch.uint8, device="cuda"),
             done=torch.zeros(B, dtype=torch.uint8, device="cuda"))
    cora.cora_gate_transfer(d["conf"], d["argmax"], d["prev"], d["persist"], d["state"], d["tokens"], B, Rr, k, tau,
                            K, d["unmask"], d["accept"], d["done"])
    torch.cuda.synchronize()
    return {k2: v.cpu().numpy() for k2, v in d.items()}


def assert_same_gate(got, want):
    for key in ("tokens", "state", "persist", "prev", "unmask", "accept", "done"):
        assert np.array_equal(got[key].astype(np.int64), want[key].astype(np.int64)), key


@pytest.mark.parametrize("B", [1, 8, 64])
@pytest.mark.parametrize("tau,K,k", [(0.65, 1, 1), (0.9, 2, 3), (0.0, 0, 0), (2.0, 1, 1), (0.3, -1, 32)])
def test_gate_bit_exact_on_identical_inputs(B, tau, K, k):
    R, V = 32, 50000
    rng = np.random.default_rng(B * 100 + k)
    hist, persist, prev, state, tokens = gate_state(3, B, R, V)
    conf = rng.uniform(0, 1, (B, R)).astype(np.float32)
    conf[rng.random((B, R)) < 0.1] = np.float32(min(tau, 1.0))    # exact threshold hits
    conf[:, 5] = conf[:, 6]                                          # confidence ties
    arg = np.where(rng.random((B, R)) < 0.7, hist[-1], rng.integers(0, V, (B, R)))
    want = O.gate_batch(conf, arg, tokens, state, persist, prev, k, tau, K)
    got = run_gpu_gate(conf, arg, tokens, state, persist, prev, k, tau, K)
    assert_same_gate(got, want)


@pytest.mark.parametrize("R", [1, 5, 31])
def test_gate_ragged_blocks(R):
    B, V = 6, 100
    rng = np.random.default_rng(R)
    hist, persist, prev, state, tokens = gate_state(4, B, R, V)
    state[0] = 1                      # a block with nothing left to resolve
    conf = rng.uniform(0, 1, (B, R)).astype(np.float32)
    arg = rng.integers(0, V, (B, R))
    want = O.gate_batch(conf, arg, tokens, state, persist, prev, 2, 0.5, 1)
    got = run_gpu_gate(conf, arg, tokens, state, persist, prev, 2, 0.5, 1)
    assert_same_gate(got, want)
    assert got["done"][0] == 1


@pytest.mark.parametrize("B", [1, 8, 64])
def test_reduce_gate_isolation_workload(B):
    R, V = GI["rows"], GI["vocab"]
    tau, K, k = GI["tau"], GI["K"], GI["k_step"]
    seed = GI["seed"]
    hist, persist, prev, state, tokens = gate_state(seed, B, R, V)
    logits = synth.gate_logits_bf16(seed, B, R, V, hist[-1], GI["keep"])
    want = O.reduce_and_gate(synth.bf16_bits_to_f32(logits), tokens, state, persist, prev, k, tau, K)

    d = dict(prev=to_dev(prev, np.int32), persist=to_dev(persist, np.int32), state=to_dev(state, np.uint8),
             tokens=to_dev(tokens, np.int32))
    conf = torch.empty((B, R), dtype=torch.float32, device="cuda")
    arg = torch.empty((B, R), dtype=torch.int32, device="cuda")
    unmask = torch.zeros((B, R), dtype=torch.uint8, device="cuda")
    accept = torch.zeros((B, R), dtype=torch.uint8, device="cuda")
    done = torch.zeros(B, dtype=torch.uint8, device="cuda")
    lg = torch.from_numpy(logits.view(np.int16)).cuda()
    cora.cora_reduce_gate(lg, B, R, V, conf, arg, d["prev"], d["persist"], d["state"], d["tokens"], k, tau, K,
                          unmask, accept, done)
    torch.cuda.synchronize()
    c, a = conf.cpu().numpy(), arg.cpu().numpy()
    # Eq. 1: fp32 reduction of the same bf16 logits.
    assert np.all(np.abs(c - want["conf"]) <= 1e-4 * want["conf"] + 1e-7)
    assert np.array_equal(a, want["argmax"])
    # Gate decisions: equal wherever the fp32/fp64 confidence difference cannot flip them.
    eps = float(np.abs(c - want["conf"]).max()) * 2 + 1e-7
    cf = want["conf"]
    U = state == 0
    ok_rows = 0
    for b in range(B):
        cu = np.sort(cf[b][U[b]])[::-1]
        rank_gap_ok = len(cu) <= k or (cu[k - 1] - cu[k] > 2 * eps if k > 0 else True)
        thr_ok = np.all(np.abs(cf[b][U[b]] - tau) > eps)
        if rank_gap_ok and thr_ok:
            ok_rows += 1
            for key, arr in (("unmask", unmask), ("accept", accept)):
                assert np.array_equal(arr.cpu().numpy()[b], want[key][b]), (key, b)
            assert np.array_equal(d["tokens"].cpu().numpy()[b], want["tokens"][b])
            assert np.array_equal(d["state"].cpu().numpy()[b], want["state"][b])
            assert done.cpu().numpy()[b] == want["done"][b]
        assert np.array_equal(d["persist"].cpu().numpy()[b], want["persist"][b])    # argmax is exact
    assert ok_rows >= max(1, int(0.9 * B))
