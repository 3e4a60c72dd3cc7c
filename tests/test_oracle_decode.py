"""Pins for the blockwise decode loop with residual acceptance and block termination.

Special cases that reduce to something coded separately or known in closed
form: the gate switched off reproduces the fixed-horizon dense decoder; a
gate that accepts everything ends each block after one or two passes; and
the count, disjointness and immutability invariants hold at every step.
"""

import numpy as np
import pytest

from oracle import cora_oracle as O
from paper_2608_11235_gb300 import synth

G, BL, T = 8, 4, 4


@pytest.fixture(scope="module")
def model(micro_cfg):
    return micro_cfg, synth.model_weights_f64(micro_cfg)


@pytest.fixture(scope="module")
def prompt(micro_cfg):
    return synth.prompts(3, 1, 6, micro_cfg["mask_id"])[0]


@pytest.mark.parametrize("tau,K", [(1.01, 1), (2.0, 0), (1.0, -1), (0.0, -1)])
def test_gate_off_is_dense_endpoint(model, prompt, tau, K):
    cfg, w = model
    dense_tokens, dense_passes = O.dense_decode(cfg, w, prompt, G, BL, T)
    tr = O.generate(cfg, w, prompt, G, BL, T, tau, K)
    assert np.array_equal(tr.tokens, dense_tokens)
    assert tr.passes_per_block == [T] * (G // BL) and dense_passes == G // BL * T


def test_accept_all_one_pass_per_block(model, prompt):
    cfg, w = model
    tr = O.generate(cfg, w, prompt, G, BL, T, 0.0, 0, record=True)
    assert tr.passes_per_block == [1] * (G // BL)
    for s in tr.steps:                                   # every position resolved on its first pass
        assert np.array_equal(s["after"].tokens, s["x_hat"])


def test_accept_all_with_one_persistence_check(model, prompt):
    """delta_p = 0, m = 1: nothing is accepted on a block's first pass; after
    that a block ends at the first pass on which every position still
    unresolved (and not transferred) repeats its previous prediction."""
    cfg, w = model
    tr = O.generate(cfg, w, prompt, G, BL, T, 0.0, 1, record=True)
    assert all(2 <= p <= T for p in tr.passes_per_block)
    for s in tr.steps:
        r = s["result"]
        U = s["before"].state == O.UNRESOLVED
        if s["step"] == 0:
            assert not r.accepted
            continue
        rest = [i for i in np.flatnonzero(U) if i not in r.transferred]
        stable = all(s["before"].prev[i] == s["x_hat"][i] for i in rest)
        assert r.done == stable


@pytest.mark.parametrize("tau,K", [(0.3, 1), (0.5, 0), (0.2, 2), (0.65, 1)])
def test_trace_invariants(model, prompt, tau, K):
    cfg, w = model
    tr = O.generate(cfg, w, prompt, G, BL, T, tau, K, record=True)
    per_block = {}
    for s in tr.steps:
        b, r = s["block"], s["result"]
        T_set, A_set = set(r.transferred), set(r.accepted)
        assert not (T_set & A_set)
        U0 = s["before"].state == O.UNRESOLVED
        assert sorted(T_set) == O.transfer_set(s["conf"], U0, O.transfer_schedule(BL, T)[s["step"]])
        resolved = ~U0
        assert np.array_equal(s["after"].tokens[resolved], s["before"].tokens[resolved])
        per_block[b] = per_block.get(b, 0) + len(T_set) + len(A_set)
        assert s["result"].done == (not np.any(s["after"].state == O.UNRESOLVED))
    assert all(v == BL for v in per_block.values())          # counts per block sum to the block length
    assert all(1 <= p <= T for p in tr.passes_per_block)
    assert not np.any(tr.tokens == -1)


def test_block_termination_counts_passes(model, prompt):
    cfg, w = model
    tr = O.generate(cfg, w, prompt, G, BL, T, 0.3, 1, record=True)
    steps_per_block = {}
    for s in tr.steps:
        steps_per_block.setdefault(s["block"], []).append(s)
    for b, ss in steps_per_block.items():
        assert len(ss) == tr.passes_per_block[b]
        assert ss[-1]["result"].done and not any(s["result"].done for s in ss[:-1])
