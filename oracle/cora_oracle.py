"""CPU oracle for one CORA-Diff denoising step and the blockwise decode loop.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may import this module.  The CUDA
path never calls it, and it shares no code with the CUDA path: inputs arrive
as plain numpy arrays (weights, prompts, logits), produced by the seeded
generator module, never by the GPU.

Plain, slow and written to be checked by eye against the paper:
  * floating point in float64; library matmul is the only primitive used;
  * the backbone is a pre-norm bidirectional Transformer (RMSNorm, RoPE,
    full non-causal softmax attention with grouped KV heads, SwiGLU FFN),
    the dense pass the paper keeps unchanged at every executed step (Sec. 3);
  * Eq. 1 (top-1 confidence and prediction), the original low-confidence
    transfer rule (Sec. 3.1), the persistence counter (Eq. 2), the residual
    acceptance gate (Eq. 3), the state update (Eq. 4) and block termination
    (Sec. 3 overview, "From acceptance to runtime" in Sec. 3.3).

Readings where the paper is silent (each is listed in the design notes):
  * transfer schedule: a block of n masked positions and horizon T fixes
    floor(n/T) positions per step, the first n mod T steps one more;
  * transfer candidates are the unresolved positions of the active block,
    ranked by confidence (higher first, then lower position);
  * argmax ties go to the lowest vocabulary id (the paper's "deterministically
    tie-broken" top-1, Sec. 3.2);
  * the transfer count of a step is the fixed schedule above; the
    "remaining-steps" variant recomputes ceil(|U| / (T - s)) each step;
  * the persistence counter and previous prediction reset at block start
    (a position's first executed step is the block's first pass);
  * the counter is updated for every position unresolved when the step
    starts, before the transfer rule and the gate act;
  * the gate compares in fp32, the precision of the kernel's confidences:
    float32(c) >= float32(delta_p) and integer m >= K; K < 0 means K = inf;
  * resolution is tracked by an explicit state, not by token == mask id.

Parity pins: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, invariants, special cases and brute force.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

# Position states of the generation canvas (match the CUDA library's codes).
# EOS_FILLED marks positions after a block that committed the EOS id (the
# EOS-aware stop variant): they take the EOS id without being decoded.
UNRESOLVED, TRANSFERRED, ACCEPTED, EOS_FILLED = 0, 1, 2, 3


# ---------------------------------------------------------------------------
# Backbone (Sec. 3: frozen, dense at every executed step).
# ---------------------------------------------------------------------------
def rms_norm(x: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * w."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * w


def rope_angles(positions: np.ndarray, head_dim: int, theta: float) -> np.ndarray:
    """[S, head_dim/2] angles pos * theta^(-2j/head_dim)."""
    j = np.arange(head_dim // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * j / head_dim)
    return np.asarray(positions, dtype=np.float64)[:, None] * inv_freq[None, :]


def rope(x: np.ndarray, positions: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing (j, j + hd/2), on [S, H, hd]."""
    hd = x.shape[-1]
    ang = rope_angles(positions, hd, theta)[:, None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., : hd // 2], x[..., hd // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Bidirectional (non-causal) softmax attention with grouped KV heads.

    q [S, Hq, hd], k/v [S, Hkv, hd]; query head h reads KV head h // (Hq/Hkv).
    Every query sees every key of its sequence (no mask).
    """
    S, Hq, hd = q.shape
    Hkv = k.shape[1]
    group = Hq // Hkv
    out = np.empty_like(q)
    for h in range(Hq):
        kh, vh = k[:, h // group, :], v[:, h // group, :]
        scores = q[:, h, :] @ kh.T / np.sqrt(hd)
        scores -= scores.max(axis=1, keepdims=True)
        p = np.exp(scores)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ vh
    return out


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def layer_forward(cfg: dict, lw: dict, h: np.ndarray, positions: np.ndarray) -> np.ndarray:
    """One pre-norm layer on the residual stream h [S, d]."""
    S = h.shape[0]
    hq, hkv, hd = cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    x = rms_norm(h, lw["attn_norm"], cfg["norm_eps"])
    q = (x @ lw["wq"].T).reshape(S, hq, hd)
    k = (x @ lw["wk"].T).reshape(S, hkv, hd)
    v = (x @ lw["wv"].T).reshape(S, hkv, hd)
    q = rope(q, positions, cfg["rope_theta"])
    k = rope(k, positions, cfg["rope_theta"])
    o = attention(q, k, v).reshape(S, hq * hd)
    h = h + o @ lw["wo"].T
    x = rms_norm(h, lw["ffn_norm"], cfg["norm_eps"])
    a = silu(x @ lw["w_gate"].T) * (x @ lw["w_up"].T)
    return h + a @ lw["w_down"].T


def forward_hidden(cfg: dict, w: dict, tokens: np.ndarray) -> np.ndarray:
    """Residual stream after the last layer, [S, d], for one sequence."""
    tokens = np.asarray(tokens)
    positions = np.arange(tokens.shape[0])
    h = w["embed"][tokens].astype(np.float64)
    for lw in w["layers"]:
        h = layer_forward(cfg, lw, h, positions)
    return h


# ---------------------------------------------------------------------------
# Prefix-cache step (a decoding variant): rows from `lo` on are recomputed,
# their queries attending to keys/values of the positions before `lo` kept
# from the block's first (dense) pass.
# ---------------------------------------------------------------------------
def layer_forward_prefix(cfg: dict, lw: dict, h: np.ndarray, positions: np.ndarray, k_pre: np.ndarray,
                         v_pre: np.ndarray):
    """One pre-norm layer on rows h [n, d] at `positions`, whose queries also
    see the given prefix keys/values [m, Hkv, hd] (after RoPE).  Returns
    (h_out, k, v) with this layer's keys/values of the n rows."""
    n = h.shape[0]
    hq, hkv, hd = cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    x = rms_norm(h, lw["attn_norm"], cfg["norm_eps"])
    q = rope((x @ lw["wq"].T).reshape(n, hq, hd), positions, cfg["rope_theta"])
    k = rope((x @ lw["wk"].T).reshape(n, hkv, hd), positions, cfg["rope_theta"])
    v = (x @ lw["wv"].T).reshape(n, hkv, hd)
    o = attention(q, np.concatenate([k_pre, k]), np.concatenate([v_pre, v])).reshape(n, hq * hd)
    h = h + o @ lw["wo"].T
    x = rms_norm(h, lw["ffn_norm"], cfg["norm_eps"])
    a = silu(x @ lw["w_gate"].T) * (x @ lw["w_up"].T)
    return h + a @ lw["w_down"].T, k, v


def forward_hidden_kv(cfg: dict, w: dict, tokens: np.ndarray):
    """The dense pass, also returning every layer's keys/values [S, Hkv, hd]."""
    tokens = np.asarray(tokens)
    hkv, hd = cfg["n_kv_heads"], cfg["head_dim"]
    empty = np.zeros((0, hkv, hd))
    h = w["embed"][tokens].astype(np.float64)
    cache = []
    for lw in w["layers"]:
        h, k, v = layer_forward_prefix(cfg, lw, h, np.arange(len(tokens)), empty, empty)
        cache.append((k, v))
    return h, cache


def forward_hidden_cached(cfg: dict, w: dict, tokens: np.ndarray, cache: list, lo: int) -> np.ndarray:
    """Residual stream of rows lo .. S-1 after the last layer, the positions
    before lo contributing only their cached keys/values."""
    tokens = np.asarray(tokens)
    h = w["embed"][tokens[lo:]].astype(np.float64)
    pos = np.arange(lo, len(tokens))
    for lw, (kc, vc) in zip(w["layers"], cache):
        h, _, _ = layer_forward_prefix(cfg, lw, h, pos, kc[:lo], vc[:lo])
    return h


def lm_logits(cfg: dict, w: dict, h_rows: np.ndarray) -> np.ndarray:
    """Logits of the given rows: final RMSNorm, then the (untied) LM head."""
    return rms_norm(h_rows, w["final_norm"], cfg["norm_eps"]) @ w["lm_head"].T


# ---------------------------------------------------------------------------
# Eq. 1: top-1 prediction and confidence over the full vocabulary.
# ---------------------------------------------------------------------------
def top1(logits: np.ndarray):
    """(c, x_hat): c = max_v softmax(l)_v, x_hat = argmax (lowest id on ties)."""
    l = np.asarray(logits, dtype=np.float64)
    p = np.exp(l - l.max(axis=-1, keepdims=True))
    p /= p.sum(axis=-1, keepdims=True)
    return p.max(axis=-1), np.argmax(l, axis=-1).astype(np.int64)


def top2_margin(logits: np.ndarray) -> np.ndarray:
    """p1 - p2, the gap between the two largest softmax probabilities."""
    l = np.asarray(logits, dtype=np.float64)
    p = np.exp(l - l.max(axis=-1, keepdims=True))
    p /= p.sum(axis=-1, keepdims=True)
    s = np.sort(p, axis=-1)
    return s[..., -1] - s[..., -2]


# ---------------------------------------------------------------------------
# Original transfer rule and its per-step schedule (Sec. 3.1).
# ---------------------------------------------------------------------------
def transfer_schedule(n: int, T: int) -> list[int]:
    """Per-step counts for n masked positions over T steps (sum = n)."""
    base, extra = divmod(n, T)
    return [base + (1 if s < extra else 0) for s in range(T)]


def remaining_step_count(n_unresolved: int, T: int, s: int) -> int:
    """The 'remaining-steps' schedule variant: at step s (0-based) of a block,
    fix ceil(|U| / (T - s)) positions, |U| the block's unresolved count when
    the step starts.  It fixes every position by step T - 1 and equals the
    fixed schedule when nothing is accepted and T divides the block length."""
    return -(-int(n_unresolved) // (T - s))


def transfer_set(conf, unresolved, k: int) -> list[int]:
    """The min(k, |U|) unresolved positions of highest confidence.

    Ranking: higher confidence first, then lower position.
    """
    cand = [i for i in range(len(unresolved)) if unresolved[i]]
    cand.sort(key=lambda i: (-float(conf[i]), i))
    return sorted(cand[: min(k, len(cand))])


# ---------------------------------------------------------------------------
# Eq. 2-4: persistence, residual gate, state update; one executed step.
# ---------------------------------------------------------------------------
@dataclass
class BlockState:
    """Per-block decoding state for one sequence (positions of the block)."""
    tokens: np.ndarray          # int64 [n]: current canvas ids of the block
    state: np.ndarray           # uint8 [n]: UNRESOLVED / TRANSFERRED / ACCEPTED
    persist: np.ndarray         # int64 [n]: m_i (Eq. 2)
    prev: np.ndarray            # int64 [n]: previous executed step's x_hat, -1 if none

    @staticmethod
    def fresh(tokens) -> "BlockState":
        n = len(tokens)
        return BlockState(np.array(tokens, dtype=np.int64), np.zeros(n, np.uint8),
                          np.zeros(n, np.int64), np.full(n, -1, np.int64))

    def copy(self) -> "BlockState":
        return BlockState(self.tokens.copy(), self.state.copy(), self.persist.copy(), self.prev.copy())


@dataclass
class StepResult:
    transferred: list = field(default_factory=list)   # T^(s)
    accepted: list = field(default_factory=list)      # A^(s)
    done: bool = False                                # U^(s+1) within the block is empty


def persistence_update(st: BlockState, x_hat) -> None:
    """Eq. 2 on every position unresolved at the start of the step."""
    for i in range(len(st.state)):
        if st.state[i] != UNRESOLVED:
            continue
        st.persist[i] = st.persist[i] + 1 if st.prev[i] == int(x_hat[i]) else 0
        st.prev[i] = int(x_hat[i])


def gate_accepts(c, m: int, tau: float, K: int) -> bool:
    """Eq. 3: a_i = 1[c_i >= delta_p and m_i >= m]; K < 0 encodes K = inf."""
    if K < 0:
        return False
    return bool(np.float32(c) >= np.float32(tau)) and int(m) >= K


def cora_step(st: BlockState, conf, x_hat, k: int, tau: float, K: int) -> StepResult:
    """One executed step on one block (mutates st): Eq. 2, transfer, Eq. 3, Eq. 4."""
    persistence_update(st, x_hat)
    unresolved = st.state == UNRESOLVED
    T_set = transfer_set(conf, unresolved, k)
    in_T = set(T_set)
    A_set = [i for i in range(len(unresolved))
             if unresolved[i] and i not in in_T and gate_accepts(conf[i], st.persist[i], tau, K)]
    for i in T_set:
        st.tokens[i] = int(x_hat[i])
        st.state[i] = TRANSFERRED
    for i in A_set:
        st.tokens[i] = int(x_hat[i])
        st.state[i] = ACCEPTED
    return StepResult(T_set, A_set, not bool(np.any(st.state == UNRESOLVED)))


# ---------------------------------------------------------------------------
# Blockwise decode with residual acceptance and block termination.
# ---------------------------------------------------------------------------
@dataclass
class DecodeTrace:
    tokens: np.ndarray                         # [G] generated ids
    passes_per_block: list                     # executed dense passes per block
    steps: list = field(default_factory=list)  # per executed step: dict of what happened


def generate(cfg: dict, w: dict, prompt, gen_len: int, block_len: int, T: int,
             tau: float, K: int, record: bool = False, forward=None, schedule: str = "fixed",
             eos_id: int = -1, persistence: str = "block", cache: str = "none") -> DecodeTrace:
    """Decode one sequence.  ``forward(tokens) -> hidden`` defaults to the oracle.

    schedule: "fixed" (the transfer schedule of the block length, the default)
    or "remaining" (remaining_step_count on the block's unresolved count).
    eos_id >= 0: EOS-aware stop -- once a block has terminated holding that id,
    every later generation position takes it (state EOS_FILLED) and the later
    blocks execute no pass (their entries in passes_per_block are 0).
    persistence: "block" (Eq. 2 counters start at each block's first pass, the
    default) or "carry" (every executed pass computes Eq. 1 for every
    generation position and updates the counter of every unresolved one, so
    a position's count starts at its first executed pass and carries into its
    block).
    cache: "none" (the dense pass at every step, the default) or "prefix"
    (a block's first pass is dense and keeps every layer's keys/values; its
    later passes recompute only the rows from the active block on, see
    forward_hidden_cached).  Not combined with carry-over persistence."""
    if forward is None:
        def forward(tok):
            return forward_hidden(cfg, w, tok)
    P = len(prompt)
    x = np.concatenate([np.asarray(prompt, np.int64), np.full(gen_len, cfg["mask_id"], np.int64)])
    gstate = np.zeros(gen_len, np.uint8)      # state of every generation position
    g_persist = np.zeros(gen_len, np.int64)   # carry mode: Eq. 2 state of every generation position
    g_prev = np.full(gen_len, -1, np.int64)
    passes = []
    steps = []
    for b in range(gen_len // block_len):
        lo = P + b * block_len
        st = BlockState.fresh(x[lo: lo + block_len])
        if persistence == "carry":
            st.persist[:] = g_persist[b * block_len:(b + 1) * block_len]
            st.prev[:] = g_prev[b * block_len:(b + 1) * block_len]
        sched = transfer_schedule(block_len, T)
        n_exec = 0
        kv = None
        for s in range(T):
            canvas, gs = (x.copy(), gstate.copy()) if record else (None, None)
            if cache == "prefix":
                if kv is None:
                    h, kv = forward_hidden_kv(cfg, w, x)
                else:
                    h = np.zeros((len(x), cfg["d_model"]))
                    h[lo:] = forward_hidden_cached(cfg, w, x, kv, lo)
            else:
                h = forward(x)
            logits = lm_logits(cfg, w, h[lo: lo + block_len])
            conf, x_hat = top1(logits)
            if persistence == "carry":
                # Eq. 2 for the unresolved positions outside the active block
                _, xh_all = top1(lm_logits(cfg, w, h[P:]))
                for j in range(gen_len):
                    if b * block_len <= j < (b + 1) * block_len or gstate[j] != UNRESOLVED:
                        continue
                    g_persist[j] = g_persist[j] + 1 if g_prev[j] == int(xh_all[j]) else 0
                    g_prev[j] = int(xh_all[j])
            before = st.copy() if record else None
            k = sched[s] if schedule == "fixed" else remaining_step_count(np.sum(st.state == UNRESOLVED), T, s)
            r = cora_step(st, conf, x_hat, k, tau, K)
            x[lo: lo + block_len] = st.tokens
            gstate[b * block_len: (b + 1) * block_len] = st.state
            if persistence == "carry":
                g_persist[b * block_len:(b + 1) * block_len] = st.persist
                g_prev[b * block_len:(b + 1) * block_len] = st.prev
            n_exec += 1
            if record:
                steps.append(dict(block=b, step=s, canvas=canvas, gen_state=gs, passes_before=n_exec - 1,
                                  conf=conf, x_hat=x_hat, logits=logits, before=before, after=st.copy(), result=r))
            if r.done:
                break
        passes.append(n_exec)
        if eos_id >= 0 and np.any(st.tokens == eos_id):
            x[lo + block_len:] = eos_id
            gstate[(b + 1) * block_len:] = EOS_FILLED
            passes.extend([0] * (gen_len // block_len - b - 1))
            break
    return DecodeTrace(x[P:].copy(), passes, steps)


def dense_decode(cfg: dict, w: dict, prompt, gen_len: int, block_len: int, T: int):
    """The unmodified fixed-horizon decoder (no residual gate), coded separately.

    Each step scores every still-masked position of the active block by its
    top-1 probability (-inf elsewhere) and commits the k_s best.  Returns
    (tokens [G], executed passes).
    """
    P = len(prompt)
    x = np.concatenate([np.asarray(prompt, np.int64), np.full(gen_len, cfg["mask_id"], np.int64)])
    masked = np.zeros(P + gen_len, bool)
    masked[P:] = True
    n_pass = 0
    for b in range(gen_len // block_len):
        lo, hi = P + b * block_len, P + (b + 1) * block_len
        counts = transfer_schedule(int(masked[lo:hi].sum()), T)
        for s in range(T):
            logits = lm_logits(cfg, w, forward_hidden(cfg, w, x)[lo:hi])
            conf, x_hat = top1(logits)
            n_pass += 1
            score = np.where(masked[lo:hi], conf, -np.inf)
            order = np.argsort(-score, kind="stable")[: counts[s]]
            for j in order:
                x[lo + j] = x_hat[j]
                masked[lo + j] = False
    return x[P:].copy(), n_pass


# ---------------------------------------------------------------------------
# Disagreement with the dense endpoint (Sec. 4): accepted-token and
# final-output disagreement of one prompt.
# ---------------------------------------------------------------------------
def disagreement(tokens, state, tokens_dense) -> tuple[float, float]:
    """(L_acc, L_out) of a CORA decode against the dense endpoint Y* on the
    same canvas: L_acc averages 1[token != Y*] over the positions the gate
    accepted (0 when none was), L_out over every generation position."""
    tokens, state, ref = np.asarray(tokens), np.asarray(state), np.asarray(tokens_dense)
    acc = [i for i in range(len(tokens)) if state[i] == ACCEPTED]
    l_acc = sum(int(tokens[i] != ref[i]) for i in acc) / max(1, len(acc))
    l_out = sum(int(tokens[i] != ref[i]) for i in range(len(tokens))) / len(tokens)
    return l_acc, l_out


# ---------------------------------------------------------------------------
# Gate-isolation path: logits -> (c, x_hat) -> one gate step, batched.
# ---------------------------------------------------------------------------
def persist_from_history(history: np.ndarray):
    """Run Eq. 2 over a [H, B, R] argmax history from a fresh block state.

    Returns (persist [B, R], prev [B, R]).
    """
    Hn, B, R = history.shape
    persist = np.zeros((B, R), np.int64)
    prev = np.full((B, R), -1, np.int64)
    for t in range(Hn):
        same = prev == history[t]
        persist = np.where(same, persist + 1, 0)
        prev = history[t].astype(np.int64)
    return persist, prev


def reduce_and_gate(logits_f32: np.ndarray, tokens, state, persist, prev, k: int, tau: float, K: int):
    """Batched gate-isolation step on [B, R, V] logits; returns a dict of outputs.

    Confidences are computed in float64 from the given logits and handed to
    the gate as float32, the precision the kernel decides in.
    """
    B, R, _ = logits_f32.shape
    conf = np.empty((B, R)); arg = np.empty((B, R), np.int64)
    for b in range(B):
        conf[b], arg[b] = top1(logits_f32[b].astype(np.float64))
    out = gate_batch(conf.astype(np.float32), arg, tokens, state, persist, prev, k, tau, K)
    out["conf"], out["argmax"] = conf, arg
    return out


def gate_batch(conf, arg, tokens, state, persist, prev, k: int, tau: float, K: int):
    """One cora_step per row b of [B, R] inputs; returns new state arrays and masks."""
    B, R = conf.shape
    res = dict(tokens=np.array(tokens, np.int64), state=np.array(state, np.uint8),
               persist=np.array(persist, np.int64), prev=np.array(prev, np.int64),
               unmask=np.zeros((B, R), np.uint8), accept=np.zeros((B, R), np.uint8),
               done=np.zeros(B, np.uint8))
    for b in range(B):
        st = BlockState(res["tokens"][b].copy(), res["state"][b].copy(),
                        res["persist"][b].copy(), res["prev"][b].copy())
        r = cora_step(st, conf[b], arg[b], k, tau, K)
        res["tokens"][b], res["state"][b], res["persist"][b], res["prev"][b] = st.tokens, st.state, st.persist, st.prev
        res["unmask"][b, r.transferred] = 1
        res["accept"][b, r.accepted] = 1
        res["done"][b] = int(r.done)
    return res
