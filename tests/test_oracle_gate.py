"""Pins for the transfer schedule, Eq. 2 (persistence), Eq. 3 (gate) and Eq. 4 (update).

An independent vectorised restatement (lexsort-based ranking, array masks)
is compared with the oracle's loop-based step over an exhaustive grid of
thresholds, and the invariants the paper fixes are checked directly.
"""

import itertools
import math

import numpy as np
import pytest

from oracle import cora_oracle as O


def test_schedule_sums_and_shape():
    assert O.transfer_schedule(32, 32) == [1] * 32
    assert O.transfer_schedule(10, 4) == [3, 3, 2, 2]
    assert O.transfer_schedule(3, 5) == [1, 1, 1, 0, 0]
    for n in range(0, 70):
        for T in range(1, 40):
            ks = O.transfer_schedule(n, T)
            assert sum(ks) == n and len(ks) == T
            assert max(ks) - min(ks) <= 1 and ks == sorted(ks, reverse=True)


def test_persistence_counter_hand_sequence():
    """Eq. 2: zero at the first executed step; +1 on an unchanged top-1; reset on a change."""
    st = O.BlockState.fresh([15])
    seq = [5, 5, 5, 7, 7, 7, 7, 2]
    want = [0, 1, 2, 0, 1, 2, 3, 0]
    got = []
    for x in seq:
        O.persistence_update(st, [x])
        got.append(int(st.persist[0]))
    assert got == want


def test_persistence_skips_resolved_positions():
    st = O.BlockState.fresh([15, 15])
    st.state[1] = O.TRANSFERRED
    O.persistence_update(st, [4, 4]); O.persistence_update(st, [4, 4])
    assert list(st.persist) == [1, 0] and list(st.prev) == [4, -1]


def test_gate_inclusive_boundaries():
    """Eq. 3 uses >= on both conditions."""
    assert O.gate_accepts(np.float32(0.65), 1, 0.65, 1)
    assert not O.gate_accepts(np.nextafter(np.float32(0.65), np.float32(0)), 1, 0.65, 1)
    assert not O.gate_accepts(np.float32(0.99), 0, 0.65, 1)
    assert O.gate_accepts(np.float32(0.0), 0, 0.0, 0)
    assert not O.gate_accepts(np.float32(1.0), 1000, 0.5, -1)       # K = inf never accepts


def _independent_step(conf, xhat, tokens, state, persist, prev, k, tau, K):
    """Vectorised restatement of one step for the cross-check."""
    conf = np.asarray(conf, np.float32)
    U = state == 0
    persist = np.where(U, np.where(prev == xhat, persist + 1, 0), persist)
    prev = np.where(U, xhat, prev)
    n = len(conf)
    order = np.lexsort((np.arange(n), -conf.astype(np.float64)))     # primary: -conf, then position
    order = [i for i in order if U[i]]
    T = np.zeros(n, bool); T[order[:min(k, len(order))]] = True
    A = U & ~T & (conf >= np.float32(tau)) & (persist >= K) & (K >= 0)
    tokens = np.where(T | A, xhat, tokens)
    state = np.where(T, 1, np.where(A, 2, state)).astype(np.uint8)
    return tokens, state, persist, prev, T, A


@pytest.mark.parametrize("tau,K", list(itertools.product([0.0, 0.5, 0.65, 0.9, 1.0, 1.01], [0, 1, 2, -1])))
def test_step_matches_independent_restatement(tau, K):
    rng = np.random.default_rng(int(tau * 100) * 10 + K + 5)
    for trial in range(60):
        n = int(rng.integers(1, 33))
        conf = rng.uniform(0, 1, n).astype(np.float32)
        conf[rng.random(n) < 0.2] = np.float32(tau) if tau <= 1 else 1.0   # exact-threshold hits
        conf[rng.random(n) < 0.15] = conf[0]                                # confidence ties
        xhat = rng.integers(0, 5, n)
        prev = np.where(rng.random(n) < 0.3, -1, rng.integers(0, 5, n))
        persist = np.where(prev < 0, 0, rng.integers(0, 4, n))
        state = np.where(rng.random(n) < 0.6, 0, rng.integers(1, 3, n)).astype(np.uint8)
        tokens = rng.integers(0, 5, n)
        k = int(rng.integers(0, 4))
        st = O.BlockState(tokens.copy(), state.copy(), persist.copy(), prev.copy())
        r = O.cora_step(st, conf, xhat, k, tau, K)
        tk, sa, pe, pv, T, A = _independent_step(conf, xhat, tokens, state, persist, prev, k, tau, K)
        assert np.array_equal(st.tokens, tk) and np.array_equal(st.state, sa)
        assert np.array_equal(st.persist, pe) and np.array_equal(st.prev, pv)
        assert sorted(r.transferred) == list(np.flatnonzero(T))
        assert sorted(r.accepted) == list(np.flatnonzero(A))


def test_step_invariants():
    rng = np.random.default_rng(11)
    for _ in range(300):
        n = int(rng.integers(1, 33))
        st = O.BlockState.fresh(np.full(n, 99))
        st.state[rng.random(n) < 0.4] = O.TRANSFERRED
        U0 = st.state == O.UNRESOLVED
        conf = rng.uniform(0, 1, n).astype(np.float32)
        xhat = rng.integers(0, 50, n)
        k = int(rng.integers(0, 5))
        frozen = st.tokens[~U0].copy()
        gate_off = O.transfer_set(conf, U0, k)
        r = O.cora_step(st, conf, xhat, k, 0.3, 0)
        T, A = set(r.transferred), set(r.accepted)
        assert not (T & A)                                    # gate acts only on U \ T
        assert T <= set(np.flatnonzero(U0)) and A <= set(np.flatnonzero(U0))
        assert len(T) == min(k, int(U0.sum()))
        assert sorted(T) == gate_off                          # transfer set = the gate-off rule's set
        assert np.array_equal(st.tokens[~U0], frozen)         # resolved tokens never change
        if T:                                                 # T holds the top-|T| confidences of U
            assert min(conf[list(T)]) >= max([conf[i] for i in np.flatnonzero(U0) if i not in T], default=-1)


def test_persist_from_history():
    h = np.array([[[1, 2]], [[1, 3]], [[1, 3]], [[4, 3]]])
    p, v = O.persist_from_history(h)
    assert p.tolist() == [[0, 2]] and v.tolist() == [[4, 3]]


@pytest.mark.parametrize("k", [0, 1, 3, 32])
@pytest.mark.parametrize("tau,K", [(0.65, 1), (0.0, 0), (0.9, 2), (0.5, -1)])
def test_gate_batch_matches_row_by_row_restatement(k, tau, K):
    """gate_batch (the expected values of the batched GPU gate) against the
    vectorised restatement applied to each row: every returned array,
    including the transfer/accept indicators and the done flags.  Rows differ
    from one another, so a swapped or shifted row index fails."""
    rng = np.random.default_rng(1000 + 7 * k + int(tau * 10) + K)
    for trial in range(25):
        B, R = int(rng.integers(1, 9)), int(rng.integers(1, 33))
        conf = rng.uniform(0, 1, (B, R)).astype(np.float32)
        conf[rng.random((B, R)) < 0.15] = np.float32(tau)                      # threshold hits
        conf[rng.random((B, R)) < 0.15] = conf[0, 0]                           # ties, also across rows
        arg = rng.integers(0, 6, (B, R))
        prev = np.where(rng.random((B, R)) < 0.3, -1, rng.integers(0, 6, (B, R)))
        persist = np.where(prev < 0, 0, rng.integers(0, 4, (B, R)))
        state = np.where(rng.random((B, R)) < 0.6, 0, rng.integers(1, 3, (B, R))).astype(np.uint8)
        if trial % 5 == 0:
            state[0] = 0                                                      # a fully unresolved row
        if trial % 7 == 0 and B > 1:
            state[-1] = 1                                                     # a row already done
        tokens = rng.integers(0, 6, (B, R)) + 100 * np.arange(B)[:, None]
        out = O.gate_batch(conf, arg, tokens, state, persist, prev, k, tau, K)
        for b in range(B):
            tk, sa, pe, pv, T, A = _independent_step(conf[b], arg[b], tokens[b], state[b], persist[b], prev[b],
                                                     k, tau, K)
            assert np.array_equal(out["tokens"][b], tk) and np.array_equal(out["state"][b], sa)
            assert np.array_equal(out["persist"][b], pe) and np.array_equal(out["prev"][b], pv)
            assert np.array_equal(out["unmask"][b], T.astype(np.uint8))
            assert np.array_equal(out["accept"][b], A.astype(np.uint8))
            assert out["done"][b] == int(not np.any(sa == 0))
        # inputs are not modified in place
        assert out["state"] is not state and out["tokens"] is not tokens


def test_reduce_and_gate_on_hand_built_logits():
    """Eq. 1 on logits with a known top-1 (closed-form confidence), ties to the
    lowest id, then the gate's decisions worked out by hand."""
    V = 20
    e = math.exp
    # row 0: id 7 boosted by 5 -> c = e^5 / (e^5 + 19); row 1: ids 12 and 4 tied at 3 -> argmax 4,
    # c = e^3 / (2 e^3 + 18); row 2: uniform -> argmax 0, c = 1/20; row 3: id 19 boosted by 9.
    lg = np.zeros((1, 4, V), np.float32)
    lg[0, 0, 7] = 5.0
    lg[0, 1, 12] = 3.0; lg[0, 1, 4] = 3.0
    lg[0, 3, 19] = 9.0
    want_c = np.array([e(5) / (e(5) + 19), e(3) / (2 * e(3) + 18), 1 / 20, e(9) / (e(9) + 19)])
    want_a = np.array([7, 4, 0, 19])
    tokens = np.full((1, 4), 99)
    state = np.zeros((1, 4), np.uint8)
    prev = np.array([[7, 4, 0, 19]])           # every row repeats its previous top-1 -> m = 1 after Eq. 2
    persist = np.zeros((1, 4), np.int64)
    out = O.reduce_and_gate(lg, tokens, state, persist, prev, 1, 0.65, 1)
    assert np.allclose(out["conf"][0], want_c, rtol=0, atol=1e-14)
    assert np.array_equal(out["argmax"][0], want_a)
    # transfer (k = 1): the highest confidence, row 3; accept: c >= 0.65 and m >= 1 among the rest -> row 0
    # (c = 0.886); rows 1 (0.47) and 2 (0.05) stay unresolved.
    assert out["unmask"][0].tolist() == [0, 0, 0, 1]
    assert out["accept"][0].tolist() == [1, 0, 0, 0]
    assert out["tokens"][0].tolist() == [7, 99, 99, 19]
    assert out["state"][0].tolist() == [O.ACCEPTED, O.UNRESOLVED, O.UNRESOLVED, O.TRANSFERRED]
    assert out["persist"][0].tolist() == [1, 1, 1, 1] and out["done"][0] == 0


def test_reduce_and_gate_decides_in_float32():
    """The gate sees float32 confidences: a float64 confidence just below
    delta_p that rounds to float32(delta_p) is accepted (Eq. 3 uses >=)."""
    tau = 0.65
    lo = np.float32(tau) - (np.float32(tau) - np.nextafter(np.float32(tau), np.float32(0))) / 2   # half an ulp below
    g0 = np.float32(math.log(tau / (1 - tau)))
    hit = None
    for i in range(-40, 41):                    # a float32 logit gap whose two-id softmax lands in [lo, tau)
        g = np.float32(g0 + np.float32(i) * np.float32(2 ** -26))
        c = 1.0 / (1.0 + math.exp(-float(g)))
        if float(lo) <= c < tau:
            hit = g
            break
    assert hit is not None
    lg = np.array([[[hit, 0.0], [hit, 0.0]]], np.float32)
    out = O.reduce_and_gate(lg, np.full((1, 2), 5), np.zeros((1, 2), np.uint8), np.zeros((1, 2), np.int64),
                            np.array([[0, 0]]), 0, tau, 1)
    assert out["conf"][0, 0] < tau and np.float32(out["conf"][0, 0]) == np.float32(tau)
    assert out["accept"][0].tolist() == [1, 1]
