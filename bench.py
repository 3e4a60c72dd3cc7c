#!/usr/bin/env python
"""Decode-throughput benchmark of the CORA-Diff hot path on GB300.

One bench step is one complete decode of the workload's batch: prompt
canvas -> every block -> every executed denoising step (dense bidirectional
forward, active-row LM head with Eq. 1 reduced on the fly, transfer rule and
residual gate with block termination) until every sequence has finished.
Metric: generated tokens/s = batch * gen_len * steps / device time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl cora|reference]
  python bench.py --gemm-shapes-only FILTER   # the GEMM beside cuBLAS at the projection shapes

Default workload: LLaDA-8B-shaped bidirectional Transformer (32 layers,
d 4096, 32 heads x 128, SwiGLU 12288, vocab 126464), random-init bf16
weights, batch 1, prompt 256 random ids, gen_len 256, block 32, 32 steps per
block, gate at the paper's frozen (delta_p, m) = (0.65, 1).

With N GPUs (torchrun, one process per GPU) every rank decodes its own
replica with its own prompts (replicas only: the method has no data-path
exchange); value = all ranks' tokens / the slowest rank's time.

--impl reference times the CPU oracle (float64 numpy) on the host cores on a
bounded sample of the same workload and reports the same metric.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# DRAM bytes (read + write) per launch from one ncu capture of each kernel on
# a workload's per-launch shapes, keyed by a hash of the kernel source at
# capture time and by the workload; null once the source changed, and for
# workloads without a capture.
NCU_TRAFFIC = {
    # gemm_tc2_kernel, mean of the QKV / O / gate-up / down launches (read + write), from
    # `ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum` over the GEMM-alone leg
    # (`bench.py --gemm-shapes-only WORKLOAD --gemm-reps 1`, the QKV launch with a plain bf16
    # store), one launch per projection (ncu flushes the caches before every profiled launch; the
    # four launches of a projection read within 0.5 % of each other; the 256 + 256 line was
    # re-captured after the 512-row gate/up launch moved to data-parallel waves, and the rules for
    # launches of at most 256 rows, none of these, left the other two valid; so did making the
    # work-split helpers callable from the host for cora_gemm_plan, which left the device code as it was):
    # (112.0 + 9.6 + 46.2 + 0.0 + 215.3 + 24.2 + 121.8 + 0.6) MB / 4 (the gate/up launch in data-parallel waves)
    ("gemm", "56665881d5de", "llada8b-shape-256+256"): 132_433_152,
    # (69.8 + 23.5 + 99.3 + 12.3 + 567.6 + 126.2 + 642.1 + 39.2) MB / 4
    ("gemm", "56665881d5de", "dream7b-shape-256+512-b4"): 394_803_648,
    # (719.5 + 300.0 + 453.3 + 168.0 + 1320.9 + 310.5 + 1620.7 + 191.3) MB / 4
    ("gemm", "56665881d5de", "llada8b-shape-512+1024-b8"): 1_270_657_856,
}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


def src_hash(name: str) -> str:
    with open(os.path.join(ROOT, "paper_2608_11235_gb300", "csrc", name), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:12]


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max([num(r[3]) for r in rows if num(r[3]) is not None], default=None)}


# ------------------------------------------------------------ distributed
def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    return ws, rank, local


def dist_max(x: float, ws: int) -> float:
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_barrier(ws: int):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------- oracle leg
def oracle_sample(cfg: dict, passes_per_seq: float, budget_s: float = 12.0):
    """Times the oracle on a bounded sample of one dense pass: layer 0 of the
    model on the full canvas (repeated until ``budget_s``) plus the LM head and
    Eq. 1 on the active rows over a vocabulary slice; extrapolates tokens/s."""
    from oracle import cora_oracle as O
    from paper_2608_11235_gb300 import synth

    S = cfg["prompt_len"] + cfg["gen_len"]
    B, G, BL = cfg["batch"], cfg["gen_len"], cfg["block_len"]
    lw = synth.layer_weights_f64(cfg, 0)
    V = cfg["vocab"]
    v_slice = min(V, 16384)
    head = {"final_norm": np.ones(cfg["d_model"]),
            "lm_head": synth.weight_f64(cfg, -1, synth.LM_HEAD, slice(0, v_slice))}
    prompt = synth.prompts(cfg["prompt_seed"], 1, cfg["prompt_len"], cfg["mask_id"])[0]
    x = np.concatenate([prompt, np.full(G, cfg["mask_id"])])
    h = np.stack([synth.weight_f64(cfg, -1, synth.EMBED, slice(int(t), int(t) + 1))[0] for t in x[:S]])
    t0 = time.perf_counter()
    n_layers_run = 0
    while True:
        O.layer_forward(cfg, lw, h, np.arange(S))
        n_layers_run += 1
        if time.perf_counter() - t0 > budget_s:
            break
    t_layer = (time.perf_counter() - t0) / n_layers_run
    t1 = time.perf_counter()
    lg = O.lm_logits(cfg, head, h[cfg["prompt_len"]: cfg["prompt_len"] + BL])
    O.top1(lg)
    t_head = (time.perf_counter() - t1) * V / v_slice
    t_pass = B * (cfg["n_layers"] * t_layer + t_head)      # the oracle decodes sequences one by one
    tok_s = B * G / (passes_per_seq * t_pass) if passes_per_seq > 0 else None
    try:
        from threadpoolctl import threadpool_info
        cores = max([p.get("num_threads", 1) for p in threadpool_info()] or [os.cpu_count()])
    except ImportError:
        cores = int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))
    sample = (f"{n_layers_run} x layer-0 forward (S={S}, fp64) + LM head/Eq.1 on {BL} rows over {v_slice} of {V} "
              f"vocab ids, extrapolated to {cfg['n_layers']} layers x {passes_per_seq:g} passes x B={B}")
    return tok_s, cores, sample, n_layers_run * t_layer + t_head * v_slice / V


# --------------------------------------------------------------- GPU leg
def kernel_costs(cfg: dict):
    """Algorithmic FLOPs / bytes per launch of each kernel class for one pass."""
    B, S = cfg["batch"], cfg["prompt_len"] + cfg["gen_len"]
    M, d, F, V = B * S, cfg["d_model"], cfg["ffn"], cfg["vocab"]
    hq, hkv, hd = cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    R = B * cfg["block_len"]
    return {
        "gemm_qkv_rope": 2.0 * M * d * (hq + 2 * hkv) * hd,
        "gemm_o_resid": 2.0 * M * hq * hd * d,
        "gemm_gate_up_swiglu": 2.0 * M * d * 2 * F,
        "gemm_down_resid": 2.0 * M * F * d,
        "attention": 4.0 * B * hq * S * S * hd,
        "lm_head_top1_bytes": 2.0 * V * d + 2.0 * R * d,
        "lm_head_top1_flops": 2.0 * R * d * V,
    }


def attn_kernel_name(cfg: dict) -> str:
    """The attention kernel a dense pass of this workload launches: one CTA per
    (sequence, head, 128-query tile) item for head_dim 64, and for head_dim 128
    while the items fit on the SMs; else the persistent two-query-tile kernel."""
    if cfg["head_dim"] != 128:
        return "attention_tc_kernel<64>"
    import torch
    items = -(-(cfg["prompt_len"] + cfg["gen_len"]) // 128) * cfg["n_heads"] * cfg["batch"]
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    return "attention_tc_kernel<128>" if items <= sms else "attention_tc2_kernel"


def tiny_leg(reps: int = 5):
    """The tiny two-layer model at its own operating point (tau 0.9, K 2): GPU
    decode rate through cora_generate (device loop), passes per block, and the
    oracle's whole decode of the same prompt timed on the host (numpy float64,
    the library's default thread count)."""
    import time as _t

    from oracle import cora_oracle as O
    from paper_2608_11235_gb300 import configs, cora, model, synth

    cfg = dict(configs.TINY)
    P, G, BL, T = cfg["prompt_len"], cfg["gen_len"], cfg["block_len"], cfg["steps_per_block"]
    prompt = synth.prompts(cfg["prompt_seed"], 1, P, cfg["mask_id"])
    m = model.create_model(cfg)
    try:
        cora.cora_generate(m, prompt, G, BL, T, cfg["tau"], cfg["K"])  # warm (graph capture)
        t0 = _t.perf_counter()
        for _ in range(reps):
            _, passes, _ = cora.cora_generate(m, prompt, G, BL, T, cfg["tau"], cfg["K"])
        gpu_s = (_t.perf_counter() - t0) / reps
    finally:
        cora.cora_model_destroy(m)
    w = synth.model_weights_f64(cfg)
    t0 = _t.perf_counter()
    tr = O.generate(cfg, w, prompt[0], G, BL, T, cfg["tau"], cfg["K"])
    ora_s = _t.perf_counter() - t0
    return {"workload": cfg["name"], "tokens_per_s": round(G / gpu_s, 2), "passes": int(passes[0]),
            "passes_per_block": round(float(passes[0]) / (G // BL), 2), "timing": "host wall clock, cora_generate",
            "cpu_baseline": {"kind": "oracle", "generate_s": round(ora_s, 3), "passes": int(sum(tr.passes_per_block)),
                             "tokens_per_s": round(G / ora_s, 2), "sample": "the whole decode of the same prompt"}}


def flush_l2(buf):
    """Evicts L2 by reading a 1 GiB buffer (a reduction: L2 ends up holding clean
    lines of it, so the timed kernel's reads evict without write-backs).  It
    runs ~0.15 ms on the GPU, long enough for the host to queue the timed
    launch before the start event is reached."""
    import torch
    buf.view(torch.int64).sum()


def gate_isolation(peaks, reps: int = 5, with_oracle: bool = False):
    """Eq. 1 from materialised bf16 logits [B, 32, 126464] + transfer rule +
    gate (cora_reduce_gate), B in {1, 8, 64}; HBM-bound.  Every timed launch
    starts from the workload's configured state: the persistence counters and
    previous predictions that the seeded 8-step argmax history leaves (run
    through the library's own gate with k = 0 and the gate off, so only Eq. 2
    acts), then half of the positions marked resolved.  The state is restored
    and L2 flushed (a 1 GiB read) before every timed launch; CUDA events
    bracket the launch only.  With ``with_oracle`` the oracle's reduction +
    gate on the same logits and state is timed on the host as the CPU baseline
    (float64 numpy, the library's default thread count; the bf16 -> float32
    widening of the logits is outside the timing)."""
    import torch

    from paper_2608_11235_gb300 import configs, cora, synth

    gi = configs.GATE_ISOLATION
    R, V = gi["rows"], gi["vocab"]
    flush = torch.zeros(1 << 30, dtype=torch.uint8, device="cuda")
    out = {}
    for B in gi["batches"]:
        hist = synth.gate_history(gi["seed"], B, R, V, gi["n_hist"], gi["keep"])
        lg_host = synth.gate_logits_bf16(gi["seed"], B, R, V, hist[-1], gi["keep"])
        lg = torch.from_numpy(lg_host.view(np.int16)).cuda()
        st = lambda dt: torch.zeros((B, R), dtype=dt, device="cuda")
        conf, arg, prev, persist = st(torch.float32), st(torch.int32), st(torch.int32), st(torch.int32)
        state, tokens, unmask, accept = st(torch.uint8), st(torch.int32), st(torch.uint8), st(torch.uint8)
        done = torch.zeros(B, dtype=torch.uint8, device="cuda")
        # Eq. 2 over the history on the GPU: every position unresolved, k = 0, gate off
        prev.fill_(-1)
        for t in range(hist.shape[0]):
            h = torch.from_numpy(np.ascontiguousarray(hist[t]).astype(np.int32)).cuda()
            cora.cora_gate_transfer(conf, h, prev, persist, state, tokens, B, R, 0, 2.0, -1, unmask, accept, done)
        unresolved = torch.from_numpy(synth.gate_unresolved(gi["seed"], B, R, gi["masked_frac"])).cuda()
        alt = (1 + torch.arange(B * R, device="cuda").reshape(B, R) % 2).to(torch.uint8)
        state0 = torch.where(unresolved, torch.zeros_like(state), alt)
        tokens0 = torch.where(unresolved, torch.full_like(tokens, V - 1),
                              torch.from_numpy(hist[-1].astype(np.int32)).cuda())
        prev0, persist0 = prev.clone(), persist.clone()
        ts = []
        for i in range(reps + 2):
            prev.copy_(prev0)
            persist.copy_(persist0)
            state.copy_(state0)
            tokens.copy_(tokens0)
            flush_l2(flush)  # ~0.15 ms on the GPU: the launch below is queued before e0 is reached
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            cora.cora_reduce_gate(lg, B, R, V, conf, arg, prev, persist, state, tokens, gi["k_step"], gi["tau"],
                                  gi["K"], unmask, accept, done)
            e1.record()
            e1.synchronize()
            if i >= 2:
                ts.append(e0.elapsed_time(e1))
        ms = statistics.median(ts)
        nbytes = B * R * V * 2
        gbs = nbytes / (ms * 1e-3) / 1e9
        out[f"B{B}"] = {"us": round(ms * 1e3, 2), "GB_s": round(gbs, 1),
                        "frac": round(gbs / peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]), 4), "bytes": nbytes,
                        "state": f"{gi['n_hist']}-step argmax history, {int(100 * gi['masked_frac'])} % masked",
                        "accepted": int(accept.sum().item()), "transferred": int(unmask.sum().item())}
        if with_oracle:
            from oracle import cora_oracle as O
            lf = synth.bf16_bits_to_f32(lg_host)
            s0 = state0.cpu().numpy()
            t0n = tokens0.cpu().numpy().astype(np.int64)
            p0 = persist0.cpu().numpy().astype(np.int64)
            v0 = prev0.cpu().numpy().astype(np.int64)
            t0 = time.perf_counter()
            O.reduce_and_gate(lf, t0n, s0, p0, v0, gi["k_step"], gi["tau"], gi["K"])
            dt = time.perf_counter() - t0
            out[f"B{B}"]["cpu_baseline"] = {"kind": "oracle", "us": round(dt * 1e6, 1),
                                            "GB_s": round(nbytes / dt / 1e9, 3)}
        del lg
    return out


def attention_shapes(peaks, reps: int = 5):
    """The attention kernel alone at the attention shape of each 8B-class
    workload (batch, canvas length, heads as configured; seeded N(0, 1) bf16
    Q/K/V from the device generator).  FLOPs per launch 4 B Hq S^2 hd against
    the burst bf16 peak (a kernel timed in isolation).  L2 is flushed (a 1 GiB
    read, long enough that the launch is queued before e0 is reached) before
    every timed launch; CUDA events bracket the launch only."""
    import torch

    from paper_2608_11235_gb300 import configs, cora, synth

    flush = torch.zeros(1 << 30, dtype=torch.uint8, device="cuda")
    peak = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    out = {}
    for name in ("llada8b-shape-256+256", "dream7b-shape-256+512-b4", "llada8b-shape-512+1024-b8"):
        c = configs.PRESETS[name]
        B, S = c["batch"], c["prompt_len"] + c["gen_len"]
        hq, hkv, hd = c["n_heads"], c["n_kv_heads"], c["head_dim"]
        n = B * S * (hq + 2 * hkv) * hd
        qkv = torch.empty(n, dtype=torch.int16, device="cuda")
        o = torch.empty(B * S * hq * hd, dtype=torch.int16, device="cuda")
        cora.cora_synth_normal_bf16(qkv, n, synth.stream_key(23, 1), 0, float(synth.normal_scale_f32(1.0)))
        ts = []
        for i in range(reps + 2):
            flush_l2(flush)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            cora.cora_op_attention(qkv, o, B, S, hq, hkv, hd)
            e1.record()
            e1.synchronize()
            if i >= 2:
                ts.append(e0.elapsed_time(e1))
        ms = statistics.median(ts)
        tf = 4.0 * B * hq * S * S * hd / (ms * 1e-3) / 1e12
        out[name] = {"B": B, "S": S, "Hq": hq, "Hkv": hkv, "hd": hd, "us": round(ms * 1e3, 2),
                     "achieved": round(tf, 1), "unit": "TFLOP/s", "peak": peak, "frac": round(tf / peak, 4)}
        del qkv, o
    out["peak_source"] = "bf16 burst (kernel timed alone)"
    return out


def gemm_shapes(peaks, only: str = "", reps: int = 20, warmup: int = 3):
    """The 2-SM GEMM alone at the four projection shapes of each 8B-class
    workload's dense pass (M = batch x canvas rows), beside cuBLAS (torch.matmul,
    bf16 out) on the same operands.  Epilogues as in the pass (residual fp32
    add, SwiGLU), except QKV, timed with the plain bf16 store (the RoPE
    epilogue needs a per-call table transpose).  CUDA events around `reps`
    back-to-back launches on the same seeded operands, both sides alike;
    `only` keeps the entries whose "workload/projection" name contains it."""
    import torch

    from paper_2608_11235_gb300 import configs, cora, synth

    peak = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    out = {}
    for name in ("llada8b-shape-256+256", "dream7b-shape-256+512-b4", "llada8b-shape-512+1024-b8"):
        c = configs.PRESETS[name]
        M = c["batch"] * (c["prompt_len"] + c["gen_len"])
        d, hd = c["d_model"], c["head_dim"]
        f = (c["ffn"] + 127) // 128 * 128
        projs = (("qkv", (c["n_heads"] + 2 * c["n_kv_heads"]) * hd, d, cora.EPI_STORE_BF16),
                 ("o", d, c["n_heads"] * hd, cora.EPI_RESID_F32),
                 ("gate_up", 2 * f, d, cora.EPI_SWIGLU),
                 ("down", d, f, cora.EPI_RESID_F32))
        for proj, N, K, epi in projs:
            key = f"{name}/{proj}"
            if only and only not in key:
                continue
            A = torch.empty(M * K, dtype=torch.int16, device="cuda")
            Bw = torch.empty(N * K, dtype=torch.int16, device="cuda")
            cora.cora_synth_normal_bf16(A, M * K, synth.stream_key(31, 1), 0, float(synth.normal_scale_f32(1.0)))
            cora.cora_synth_normal_bf16(Bw, N * K, synth.stream_key(31, 2), 0,
                                        float(synth.normal_scale_f32(K ** -0.5)))
            if epi == cora.EPI_RESID_F32:
                C, ldc = torch.zeros(M, N, dtype=torch.float32, device="cuda"), N
            elif epi == cora.EPI_SWIGLU:
                C, ldc = torch.zeros(M, N // 2, dtype=torch.int16, device="cuda"), N // 2
            else:
                C, ldc = torch.zeros(M, N, dtype=torch.int16, device="cuda"), N

            def ours():
                cora.cora_op_gemm(A, Bw, C, M, N, K, ldc, epi)

            At, Bt = A.view(torch.bfloat16).view(M, K), Bw.view(torch.bfloat16).view(N, K)
            D = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")

            def cublas():
                torch.matmul(At, Bt.t(), out=D)

            row = {"M": M, "N": N, "K": K, "epilogue": {0: "bf16 store", 1: "fp32 residual add", 2: "SwiGLU"}[epi]}
            for tag, fn in (("ours", ours), ("cublas", cublas)):
                for _ in range(warmup):
                    fn()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record()
                for _ in range(reps):
                    fn()
                e1.record()
                e1.synchronize()
                ms = e0.elapsed_time(e1) / reps
                row[f"{tag}_us"] = round(ms * 1e3, 1)
                row[f"{tag}_tflops"] = round(2.0 * M * N * K / (ms * 1e-3) / 1e12, 1)
            row["ours_frac"] = round(row["ours_tflops"] / peak, 4)
            row["vs_cublas"] = round(row["cublas_us"] / row["ours_us"], 3)
            out[key] = row
            del A, Bw, C, D
            torch.cuda.empty_cache()
    out["peak"] = peak
    out["peak_source"] = "bf16 burst (kernels timed alone)"
    return out


def profile_pass(cora, s, cfg, prompt_dev):
    """Per-launch device times of the first pass of a decode, two eager runs
    (CUDA events around every launch on the session's stream), the smaller
    time of each launch kept: {kind: [ms, ...]}."""
    cora.cora_session_reset(s, prompt_dev)
    prof = cora.cora_session_profile_step(s, cfg["n_layers"])
    cora.cora_session_reset(s, prompt_dev)
    prof2 = cora.cora_session_profile_step(s, cfg["n_layers"])
    by = {}
    for (k1, t1), (_, t2) in zip(prof, prof2):
        by.setdefault(k1, []).append(min(t1, t2))
    return by


def pass_rooflines(cora, s, cfg, prompt_dev, peaks, peak_src):
    """(roofline of the dominant GEMM kernel, per-kernel shares, LM head and
    attention rooflines) of one dense pass of workload ``cfg``."""
    by = profile_pass(cora, s, cfg, prompt_dev)
    costs = kernel_costs(cfg)
    gemm_kinds = ["gemm_qkv_rope", "gemm_o_resid", "gemm_gate_up_swiglu", "gemm_down_resid"]
    gemm_ms = sum(sum(by[k]) for k in gemm_kinds)
    gemm_flops = sum(costs[k] * len(by[k]) for k in gemm_kinds)
    n_gemm = sum(len(by[k]) for k in gemm_kinds)
    step_ms = sum(sum(v) for v in by.values())
    gemm_tflops = gemm_flops / (gemm_ms * 1e-3) / 1e12
    peak_tf = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    hbm = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
    head_ms = sum(by["lm_head_top1"]) / len(by["lm_head_top1"])
    head_gbs = costs["lm_head_top1_bytes"] / (head_ms * 1e-3) / 1e9
    attn_ms = sum(by["attention"]) / len(by["attention"])
    kernels = {k: {"launches_per_pass": len(v), "ms_per_launch": round(sum(v) / len(v), 5),
                   "share": round(sum(v) / step_ms, 4)} for k, v in sorted(by.items())}
    traffic = NCU_TRAFFIC.get(("gemm", src_hash("gemm.cu"), cfg["name"]))  # per workload: the shapes differ
    roofline = {"bound": "tensor", "kernel": "gemm_tc2_kernel (QKV+RoPE, O+res, gate/up+SwiGLU, down+res)",
                "achieved": round(gemm_tflops, 2), "peak": peak_tf, "unit": "TFLOP/s",
                "frac": round(gemm_tflops / peak_tf, 4), "traffic": traffic,
                "peak_source": f"{peak_src} bf16 sustained", "flops_per_launch": round(gemm_flops / n_gemm),
                "ms_per_launch": round(gemm_ms / n_gemm, 5)}
    others = {
        "lm_head_top1": {"bound": "hbm", "achieved": round(head_gbs, 1), "unit": "GB/s", "peak": hbm,
                         "frac": round(head_gbs / hbm, 4),
                         "bytes_per_launch": costs["lm_head_top1_bytes"], "ms_per_launch": round(head_ms, 5)},
        "attention": {"bound": "tensor", "kernel": attn_kernel_name(cfg),
                      "achieved": round(costs["attention"] / (attn_ms * 1e-3) / 1e12, 2), "unit": "TFLOP/s",
                      "peak": peak_tf, "frac": round(costs["attention"] / (attn_ms * 1e-3) / 1e12 / peak_tf, 4),
                      "ms_per_launch": round(attn_ms, 5)},
        "pass_model_tflops": round((gemm_flops + costs["attention"] * len(by["attention"]) +
                                    costs["lm_head_top1_flops"]) / (step_ms * 1e-3) / 1e12, 2),
        "eager_pass_ms": round(step_ms, 3),
    }
    return roofline, kernels, others


def timed_decode(cora, torch, m, cfg, prompt_dev, tau, K, opt=None, warm_steps=2):
    """One complete decode of ``cfg``'s batch through a fresh session, timed
    with CUDA events on the session's stream (device-resident prompt): the
    session is created (graphs captured), warmed by ``warm_steps`` executed
    steps, reset, then cora_session_run runs the whole decode.  Returns
    (session, ms, batched passes, per-sequence passes)."""
    B, P, G, BL, T = cfg["batch"], cfg["prompt_len"], cfg["gen_len"], cfg["block_len"], cfg["steps_per_block"]
    s = cora.cora_session_create(m, B, prompt_dev, P, G, BL, T, tau, K, options=opt)
    stream = torch.cuda.ExternalStream(cora.cora_session_stream(s))
    for _ in range(warm_steps):
        if cora.cora_denoise_step(s):
            break
    cora.cora_session_reset(s, prompt_dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    steps, _ = cora.cora_session_run(s)
    e1.record(stream)
    e1.synchronize()
    carry = opt is not None and opt.persistence == cora.PERSIST_CARRY  # Eq. 1 state on every generation row
    ctrl = cora.cora_session_read(s, B, P + G, G, BL, eq1_rows=G if carry else BL)["ctrl"]
    return s, e0.elapsed_time(e1), steps, ctrl[:, 2].astype(np.int64)


def workload_leg(name, peaks, peak_src, m_same=None):
    """A further 8B-class workload (the Dream-shaped batch of 4, or the
    fixed-horizon 512 + 1024 batch of 8): one complete decode with the
    configured N(0, 0.02) head and one with the gate-exercising head, each
    timed with CUDA events; executed passes per sequence against the horizon;
    GEMM and attention rooflines of its dense pass.  ``m_same``: a model
    handle with this workload's weights already resident (reused for the
    configured head)."""
    import torch

    from paper_2608_11235_gb300 import configs, cora, model, synth

    cfg = dict(configs.PRESETS[name])
    B, P, G, BL, T = cfg["batch"], cfg["prompt_len"], cfg["gen_len"], cfg["block_len"], cfg["steps_per_block"]
    horizon = (G // BL) * T
    out = {"workload": name, "batch": B, "prompt_len": P, "gen_len": G, "block_len": BL, "steps_per_block": T,
           "tau": cfg["tau"], "K": cfg["K"], "horizon": horizon,
           "timing": "CUDA events on the session stream around one complete decode (one graph launch), "
                     "device-resident prompt; weights larger than L2"}
    for variant in ("as_configured", "gate_exercising"):
        c = cfg if variant == "as_configured" else configs.gate_exercising(cfg)
        own = not (variant == "as_configured" and m_same is not None)
        m = model.create_model(c) if own else m_same
        try:
            prompt_dev = torch.from_numpy(synth.prompts(c["prompt_seed"], B, P, c["mask_id"])).cuda()
            s, ms, batched, passes = timed_decode(cora, torch, m, c, prompt_dev, c["tau"], c["K"])
            try:
                roof, kern, others = pass_rooflines(cora, s, c, prompt_dev, peaks, peak_src)
            finally:
                cora.cora_session_destroy(s)
        finally:
            if own:
                cora.cora_model_destroy(m)
        out[variant] = {"head_sigma": round(c["head_sigma"], 6), "tokens_per_s": round(B * G / (ms * 1e-3), 3),
                        "ms_per_decode": round(ms, 1), "batched_passes": int(batched),
                        "passes_per_seq": passes.tolist(), "passes_per_block": round(float(passes.mean()) / (G // BL), 3),
                        "rho": round(float(passes.mean()) / horizon, 4), "ms_per_batched_pass": round(ms / batched, 3),
                        "roofline": roof, "attention": others["attention"], "lm_head_top1": others["lm_head_top1"],
                        "pass_model_tflops": others["pass_model_tflops"],
                        "kernel_shares": {k: v["share"] for k, v in kern.items()}}
    return out


def run_cora(args, cfg, ws, rank, local):
    import torch

    from paper_2608_11235_gb300 import configs, cora, model, synth

    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    peaks, peak_src = load_peaks()

    B, P, G, BL, T = cfg["batch"], cfg["prompt_len"], cfg["gen_len"], cfg["block_len"], cfg["steps_per_block"]
    tau, K = cfg["tau"], cfg["K"]
    m = model.create_model(cfg, device=f"cuda:{local}")
    prompt = synth.prompts(cfg["prompt_seed"] + 7919 * rank, B, P, cfg["mask_id"])
    prompt_dev = torch.from_numpy(prompt).to(f"cuda:{local}")
    s = cora.cora_session_create(m, B, prompt_dev, P, G, BL, T, tau, K)
    stream = torch.cuda.ExternalStream(cora.cora_session_stream(s))

    device_loop = [False]

    def decode():
        # one complete decode: a single graph launch whose WHILE node runs
        # step after step until every sequence has finished
        cora.cora_session_reset(s, prompt_dev)
        steps, device_loop[0] = cora.cora_session_run(s)
        return steps

    for _ in range(args.warmup):
        passes = decode()
    # ----- timed region: K complete decodes, device-resident inputs
    dist_barrier(ws)
    torch.cuda.synchronize()
    clk = ClockSampler(local)
    clk.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    total_passes = 0
    for _ in range(args.steps):
        total_passes += decode()
    e1.record(stream)
    e1.synchronize()
    torch.cuda.synchronize()
    clocks = clk.stop()
    dist_barrier(ws)
    ms_local = e0.elapsed_time(e1)
    ms = dist_max(ms_local, ws)
    out = cora.cora_session_read(s, B, P + G, G, BL)
    per_seq_passes = out["ctrl"][:, 2].astype(float)

    # ----- the same decode with the prefix cache (decoding variant): a block's
    # first pass dense, its later passes over the rows from the active block on
    pc = None
    if not args.no_variant and BL == 32:
        sc = cora.cora_session_create(m, B, prompt_dev, P, G, BL, T, tau, K,
                                      options=cora.decode_options(cache=cora.CACHE_PREFIX))
        stc = torch.cuda.ExternalStream(cora.cora_session_stream(sc))
        cora.cora_session_reset(sc, prompt_dev)
        cora.cora_session_run(sc)
        reps = max(1, min(args.steps, 3))
        q0, q1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        q0.record(stc)
        steps_c = 0
        for _ in range(reps):
            cora.cora_session_reset(sc, prompt_dev)
            steps_c += cora.cora_session_run(sc)[0]
        q1.record(stc)
        q1.synchronize()
        ms_c = q0.elapsed_time(q1) / reps
        cora.cora_session_destroy(sc)
        pc = {"tokens_per_s": round(B * G / (ms_c * 1e-3), 3), "ms_per_decode": round(ms_c, 3),
              "passes": steps_c // reps, "dense_passes": G // BL, "cached_passes": steps_c // reps - G // BL,
              "timing": "CUDA events on the session stream, device-resident prompt"}

    # ----- per-kernel device times (one eager pass with events around each launch)
    roofline, kernels, others = pass_rooflines(cora, s, cfg, prompt_dev, peaks, peak_src)

    # ----- end to end through the public call, host buffers (pinned), copies inside
    prompt_pin = torch.from_numpy(prompt).pin_memory()
    for _ in range(1):
        cora.cora_generate(m, prompt_pin.numpy(), G, BL, T, tau, K)
    dist_barrier(ws)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        toks, passes_e2e, _ = cora.cora_generate(m, prompt_pin.numpy(), G, BL, T, tau, K)
    e2e_s = dist_max(time.perf_counter() - t0, ws)
    assert toks.shape == (B, G)

    # ----- gate-exercising variant (LM head scaled so confidences span (0, 1))
    gx = None
    if not args.no_variant:
        cfg_g = configs.gate_exercising(cfg)
        cora.cora_session_destroy(s)
        s = None
        mg = model.create_model(cfg_g, device=f"cuda:{local}")
        sg, msg, _, pg = timed_decode(cora, torch, mg, cfg_g, prompt_dev, tau, K)
        cora.cora_session_destroy(sg)
        gx = {"head_sigma": round(cfg_g["head_sigma"], 6), "tokens_per_s": round(B * G / (msg * 1e-3), 2),
              "passes_per_block": round(float(pg.mean()) / (G // BL), 3),
              "rho": round(float(pg.mean()) / ((G // BL) * T), 4),
              "timing": "CUDA events on the session stream around one complete decode (device-resident prompt)"}
        # (tau, K, schedule) sweep on the same model: the gate's operating
        # points and the remaining-steps schedule, each one decode timed with
        # CUDA events; the dense endpoint Y* of the same prompts (gate off)
        # gives the disagreement columns
        sd = cora.cora_session_create(mg, B, prompt_dev, P, G, BL, T, 2.0, K)
        cora.cora_session_run(sd)
        sweep = []
        for tau_s, K_s, sched, pers in ((tau, K, 0, 0), (tau, 0, 0, 0), (tau, 2, 0, 0), (0.9, K, 0, 0),
                                        (0.5, K, 0, 0), (tau, K, 1, 0), (tau, K, 0, 1), (2.0, K, 0, 0)):
            opt = cora.decode_options(schedule=sched, persistence=pers)
            sv, dt_ms, _, ps = timed_decode(cora, torch, mg, cfg_g, prompt_dev, tau_s, K_s, opt=opt)
            n_acc, n_ad, n_od = cora.cora_session_disagreement(sv, sd, B)
            cora.cora_session_destroy(sv)
            sweep.append({"tau": tau_s, "K": K_s, "schedule": "remaining" if sched else "fixed",
                          "persistence": "carry" if pers else "block",
                          "passes_per_block": round(float(ps.mean()) / (G // BL), 3),
                          "rho": round(float(ps.mean()) / ((G // BL) * T), 4),
                          "tokens_per_s": round(B * G / (dt_ms * 1e-3), 2),
                          "accepted_per_seq": float(n_acc.mean()),
                          "L_acc": round(float(np.mean(n_ad / np.maximum(1, n_acc))), 4),
                          "L_out": round(float(np.mean(n_od / G)), 4)})
        cora.cora_session_destroy(sd)
        gx["sweep"] = sweep
        cora.cora_model_destroy(mg)
    if s is not None:
        cora.cora_session_destroy(s)
    workloads = None
    if not args.no_variant and not args.no_workloads and ws == 1 and cfg["name"] == "llada8b-shape-256+256":
        workloads = {"llada8b-shape-512+1024-b8": workload_leg("llada8b-shape-512+1024-b8", peaks, peak_src, m_same=m)}
        cora.cora_model_destroy(m)
        m = None
        workloads["dream7b-shape-256+512-b4"] = workload_leg("dream7b-shape-256+512-b4", peaks, peak_src)
    if m is not None:
        cora.cora_model_destroy(m)
    gate_iso = None if args.no_variant else gate_isolation(
        peaks, with_oracle=(rank == 0 and ws == 1 and not args.no_cpu_baseline))
    tiny = None if args.no_variant else tiny_leg()
    attn_shapes = None if args.no_variant else attention_shapes(peaks)
    gemm_cmp = None if args.no_variant else gemm_shapes(peaks)

    value = ws * B * G * args.steps / (ms * 1e-3)
    # the launches of one pass as the eager profile recorded them (embed, final norm, LM head,
    # gate; per layer 4 GEMMs and attention, plus the RMSNorms not carried by a residual GEMM);
    # the device loop adds the kernel that counts the pass and sets the WHILE condition
    launches_per_pass = sum(k["launches_per_pass"] for k in kernels.values()) + (1 if device_loop[0] else 0)
    result = {
        "metric": "generated tokens/s (LLaDA-8B shape, gen 256)",
        "value": round(value, 3), "unit": "tokens/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms / args.steps, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded random-init weights and prompt ids)",
        "config": {"workload": cfg["name"], "batch": B, "prompt_len": P, "gen_len": G, "block_len": BL,
                   "steps_per_block": T, "tau": tau, "K": K, "n_layers": cfg["n_layers"], "d_model": cfg["d_model"],
                   "vocab": cfg["vocab"], "weights": f"bf16 N(0,{cfg['init_sigma']}) (approx.), head N(0,{cfg['head_sigma']})",
                   "l2": "inputs larger than L2 (16 GB of weights streamed every pass)",
                   "passes_per_seq": float(per_seq_passes.mean()),
                   "passes_per_block": round(float(per_seq_passes.mean()) / (G // BL), 3),
                   "rho": round(float(per_seq_passes.mean()) / ((G // BL) * T), 4),
                   "parallelism": f"replicas x{ws}",
                   "decode_loop": "device (one graph launch per decode, conditional WHILE node)" if device_loop[0]
                   else "host (one graph launch per step)"},
        "e2e": {"value": round(ws * B * G * args.steps / e2e_s, 3), "unit": "tokens/s",
                "h2d_bytes_per_step": int(B * P * 4), "d2h_bytes_per_step": int(B * G * 4 + B * 8),
                "timing": "host wall clock around cora_generate (pinned host prompt in, host tokens out)"},
        "roofline": roofline,
        "kernels": kernels,
        "other_rooflines": others,
        "gpu_launches": int(total_passes * launches_per_pass + args.steps),
        "clocks": clocks,
        "gate_exercising": gx,
        "prefix_cache": pc,
        "gate_isolation": gate_iso,
        "tiny": tiny,
        "attention_shapes": attn_shapes,
        "gemm_shapes": gemm_cmp,
        "workloads": workloads,
    }
    return result, float(per_seq_passes.mean())


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["cora", "reference"], default="cora")
    ap.add_argument("--workload", default="llada8b-shape-256+256")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-variant", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the Dream-shaped and 512+1024 x 8 decodes (about four minutes)")
    ap.add_argument("--layers", type=int, default=0, help="override n_layers (same per-launch shapes)")
    ap.add_argument("--gemm-shapes-only", default=None, metavar="FILTER",
                    help="time only the GEMM-vs-cuBLAS shapes whose workload/projection name contains FILTER "
                         "('' = all), print them as JSON and exit")
    ap.add_argument("--gemm-reps", type=int, default=20)
    args = ap.parse_args()
    if args.gemm_shapes_only is not None:
        peaks, _ = load_peaks()
        print(json.dumps(gemm_shapes(peaks, args.gemm_shapes_only, reps=args.gemm_reps,
                                     warmup=min(args.warmup, 3))))
        return
    from paper_2608_11235_gb300 import configs
    cfg = dict(configs.PRESETS[args.workload])
    if args.layers:
        cfg = configs.with_layers(cfg, args.layers)
    ws, rank, local = dist_setup()

    if args.impl == "reference":
        if rank != 0:
            return
        horizon = (cfg["gen_len"] // cfg["block_len"]) * cfg["steps_per_block"]
        vals, times = [], []
        for i in range(args.warmup + args.steps):
            tok_s, cores, sample, t = oracle_sample(cfg, horizon, budget_s=8.0)
            if i >= args.warmup:
                vals.append(tok_s)
                times.append(t)
        v = statistics.mean(vals)
        print(json.dumps({
            "impl": "reference", "metric": "generated tokens/s (LLaDA-8B shape, gen 256)", "value": v,
            "unit": "tokens/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * statistics.mean(times), 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg["name"], "batch": cfg["batch"], "prompt_len": cfg["prompt_len"],
                       "gen_len": cfg["gen_len"], "passes_per_seq": horizon, "parallelism": "none (host cores)"},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }))
        return

    result, passes = run_cora(args, cfg, ws, rank, local)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        tok_s, cores, sample, _ = oracle_sample(cfg, passes)
        result["cpu_baseline"] = {"value": tok_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                                  "sample": sample}
    elif rank == 0:
        result["cpu_baseline"] = None
    if rank == 0:
        print(json.dumps(result))


if __name__ == "__main__":
    main()
