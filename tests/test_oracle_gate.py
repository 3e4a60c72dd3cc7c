"""Pins for the transfer schedule, Eq. 2 (persistence), Eq. 3 (gate) and Eq. 4 (update).

An independent vectorised restatement (lexsort-based ranking, array masks)
is compared with the oracle's loop-based step over an exhaustive grid of
thresholds, and the invariants the paper fixes are checked directly.
"""

import itertools

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
