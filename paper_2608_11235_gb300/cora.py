"""Thin ctypes binding of libcora.so (argument marshalling only).

Every function here forwards to the C entry point of the same name declared
in include/cora.h; all arithmetic of the decoding path runs in the library's
CUDA kernels.  Tensors may be passed as torch tensors (their data pointer is
used), numpy arrays (host memory) or raw integer addresses.  If the library
has not been built the first call raises: there is no CPU fallback.
"""

from __future__ import annotations

import ctypes as C
import os

import numpy as np

from . import build as _build

CORA_OK, CORA_EINVAL, CORA_ECUDA, CORA_ENOMEM, CORA_ETIMEOUT, CORA_ESTATE = 0, -1, -2, -3, -4, -5
UNRESOLVED, TRANSFERRED, ACCEPTED = 0, 1, 2
EPI_STORE_BF16, EPI_RESID_F32, EPI_SWIGLU, EPI_ROPE_BF16 = 0, 1, 2, 3

EXPORTED = [
    "cora_last_error", "cora_version", "cora_model_create", "cora_model_destroy", "cora_session_create",
    "cora_session_destroy", "cora_session_reset", "cora_denoise_step", "cora_session_run", "cora_session_read", "cora_session_write",
    "cora_session_batched_passes", "cora_generate", "cora_gate_transfer", "cora_reduce_top1", "cora_reduce_gate",
    "cora_op_gemm", "cora_op_attention", "cora_op_rmsnorm", "cora_op_lm_head_top1", "cora_synth_normal_bf16",
    "cora_device_error", "cora_session_profile_step", "cora_session_stream", "cora_reduce_top1_noalloc",
    "cora_session_create_ex", "cora_generate_ex", "cora_session_disagreement", "cora_check_wait_timeout",
    "cora_session_finished", "cora_op_attention_rows", "cora_gemm_plan",
]
DTYPE_BF16, DTYPE_F32 = 0, 1
SCHEDULE_FIXED, SCHEDULE_REMAINING = 0, 1
PERSIST_BLOCK, PERSIST_CARRY = 0, 1
CACHE_NONE, CACHE_PREFIX = 0, 1
KIND_NAMES = ["embed", "rmsnorm", "gemm_qkv_rope", "attention", "gemm_o_resid", "gemm_gate_up_swiglu",
              "gemm_down_resid", "final_norm", "lm_head_top1", "gate"]


class CoraError(RuntimeError):
    def __init__(self, fn: str, code: int, msg: str):
        super().__init__(f"{fn} failed with status {code}: {msg}")
        self.code = code


class DecodeOptions(C.Structure):
    _fields_ = [("schedule", C.c_int32), ("persistence", C.c_int32), ("eos_id", C.c_int32), ("cache", C.c_int32)]


def decode_options(schedule=SCHEDULE_FIXED, persistence=PERSIST_BLOCK, eos_id=-1, cache=0) -> DecodeOptions:
    return DecodeOptions(schedule, persistence, eos_id, cache)


class ModelConfig(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("ffn", C.c_int32), ("vocab", C.c_int32),
                ("mask_id", C.c_int32), ("rope_theta", C.c_float), ("norm_eps", C.c_float)]


PP = C.POINTER(C.c_void_p)


class Weights(C.Structure):
    _fields_ = [("embed", C.c_void_p), ("lm_head", C.c_void_p), ("final_norm", C.c_void_p),
                ("attn_norm", PP), ("wq", PP), ("wk", PP), ("wv", PP), ("wo", PP), ("ffn_norm", PP),
                ("w_gate", PP), ("w_up", PP), ("w_down", PP), ("dtype", C.c_int32)]


_lib = None


def library_path() -> str:
    return _build.LIB


def lib():
    """Loads libcora.so (raises if it is missing)."""
    global _lib
    if _lib is None:
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with `python -m paper_2608_11235_gb300.build`")
        L = C.CDLL(path)
        vp, i32, i64, f32, u64 = C.c_void_p, C.c_int32, C.c_int64, C.c_float, C.c_uint64
        sig = {
            "cora_last_error": ([], C.c_char_p),
            "cora_version": ([], C.c_int),
            "cora_model_create": ([C.POINTER(ModelConfig), C.POINTER(Weights), C.POINTER(vp)], C.c_int),
            "cora_model_destroy": ([vp], C.c_int),
            "cora_session_create": ([vp, i32, vp, i32, i32, i32, i32, f32, i32, C.POINTER(vp)], C.c_int),
            "cora_session_destroy": ([vp], C.c_int),
            "cora_session_reset": ([vp, vp], C.c_int),
            "cora_denoise_step": ([vp, i32, i32, vp, vp, vp], C.c_int),
            "cora_session_finished": ([vp, vp], C.c_int),
            "cora_session_run": ([vp, vp, vp], C.c_int),
            "cora_session_read": ([vp] + [vp] * 9, C.c_int),
            "cora_session_write": ([vp] + [vp] * 5, C.c_int),
            "cora_session_batched_passes": ([vp, vp], C.c_int),
            "cora_session_profile_step": ([vp, i32, vp, vp, vp], C.c_int),
            "cora_session_stream": ([vp, C.POINTER(vp)], C.c_int),
            "cora_generate": ([vp, vp, i32, i32, i32, i32, i32, f32, i32, vp, vp, vp], C.c_int),
            "cora_session_create_ex": ([vp, i32, vp, i32, i32, i32, i32, f32, i32, vp, C.POINTER(vp)], C.c_int),
            "cora_generate_ex": ([vp, vp, i32, i32, i32, i32, i32, f32, i32, vp, vp, vp, vp], C.c_int),
            "cora_session_disagreement": ([vp, vp, vp, vp, vp], C.c_int),
            "cora_gate_transfer": ([vp] * 6 + [i32, i32, i32, f32, i32] + [vp] * 3 + [vp], C.c_int),
            "cora_reduce_top1": ([vp, i32, i32, vp, vp, vp], C.c_int),
            "cora_reduce_top1_noalloc": ([vp, i32, i32, vp, vp, vp], C.c_int),
            "cora_reduce_gate": ([vp, i32, i32, i32] + [vp] * 6 + [i32, f32, i32] + [vp] * 3 + [vp], C.c_int),
            "cora_op_gemm": ([vp, vp, vp, i32, i32, i32, i32, i32, vp, i32, i32, i32, vp], C.c_int),
            "cora_gemm_plan": ([i32, i32, i32, i32, i32, vp, vp, i32, vp], C.c_int),
            "cora_op_attention": ([vp, vp, i32, i32, i32, i32, i32, vp], C.c_int),
            "cora_op_attention_rows": ([vp, vp, i32, i32, i32, i32, i32, i32, i32, vp], C.c_int),
            "cora_op_rmsnorm": ([vp, vp, vp, i32, i32, f32, vp], C.c_int),
            "cora_op_lm_head_top1": ([vp, vp, i32, i32, i32, vp, vp, vp], C.c_int),
            "cora_synth_normal_bf16": ([vp, i64, u64, i64, f32, vp], C.c_int),
            "cora_device_error": ([vp, i32], C.c_int),
            "cora_check_wait_timeout": ([i32, vp], C.c_int),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes, f.restype = args, res
        _lib = L
    return _lib


def ptr(x) -> int | None:
    """Address of a torch tensor, numpy array, ctypes object or integer (None stays NULL)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    return C.addressof(x)


def _check(fn: str, rc: int) -> None:
    if rc != CORA_OK:
        raise CoraError(fn, rc, lib().cora_last_error().decode())


def _stream(stream) -> int | None:
    if stream is None:
        return None
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


# --------------------------------------------------------------------- API
def cora_version() -> int:
    return lib().cora_version()


def _weight_dtype(t, default: int) -> int:
    if not hasattr(t, "dtype"):          # raw addresses: the caller states the type
        return default
    name = str(t.dtype)
    if "float32" in name:
        return DTYPE_F32
    if "int16" in name:
        return DTYPE_BF16
    raise TypeError(f"weights must be float32 or bf16 bit patterns (int16/uint16), got {name}")


def cora_model_create(cfg: dict, tensors: dict) -> int:
    """``tensors`` holds tensors in nn.Linear layout, all float32 or all bf16
    bit patterns (uint16/int16): embed, lm_head, optional final_norm, and
    per-layer lists wq, wk, wv, wo, w_gate, w_up, w_down, optional attn_norm /
    ffn_norm.  The element type is passed to the library as cora_weights.dtype
    (for raw integer addresses, from the optional ``dtype`` entry)."""
    c = ModelConfig(cfg["n_layers"], cfg["d_model"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"],
                    cfg["ffn"], cfg["vocab"], cfg["mask_id"], cfg["rope_theta"], cfg["norm_eps"])
    L = cfg["n_layers"]
    keep = []

    def arr(key):
        if key not in tensors or tensors[key] is None:
            return None
        a = (C.c_void_p * L)(*[ptr(t) for t in tensors[key]])
        keep.append(a)
        return C.cast(a, PP)

    w = Weights(ptr(tensors["embed"]), ptr(tensors["lm_head"]), ptr(tensors.get("final_norm")),
                arr("attn_norm"), arr("wq"), arr("wk"), arr("wv"), arr("wo"), arr("ffn_norm"),
                arr("w_gate"), arr("w_up"), arr("w_down"), _weight_dtype(tensors["embed"], tensors.get("dtype", DTYPE_BF16)))
    out = C.c_void_p()
    _check("cora_model_create", lib().cora_model_create(C.byref(c), C.byref(w), C.byref(out)))
    return out.value


def cora_model_destroy(model: int) -> None:
    _check("cora_model_destroy", lib().cora_model_destroy(model))


def cora_session_create(model, batch, prompt, prompt_len, gen_len, block_len, steps_per_block, tau, K,
                        options: DecodeOptions | None = None) -> int:
    out = C.c_void_p()
    if options is None:
        _check("cora_session_create", lib().cora_session_create(model, batch, ptr(prompt), prompt_len, gen_len,
                                                                block_len, steps_per_block, tau, K, C.byref(out)))
    else:
        _check("cora_session_create_ex", lib().cora_session_create_ex(
            model, batch, ptr(prompt), prompt_len, gen_len, block_len, steps_per_block, tau, K,
            C.cast(C.byref(options), C.c_void_p), C.byref(out)))
    return out.value


def cora_session_destroy(session) -> None:
    _check("cora_session_destroy", lib().cora_session_destroy(session))


def cora_session_reset(session, prompt) -> None:
    _check("cora_session_reset", lib().cora_session_reset(session, ptr(prompt)))


def cora_denoise_step(session, block: int = -1, step: int = -1, conf_out=None, argmax_out=None,
                      done_out=None) -> bool:
    """One executed step (cora_denoise_step), then cora_session_finished:
    returns True once every sequence has finished.  block/step = -1 skip the
    check of the session's position; the outputs are optional [B, block_len]
    float32 / int32 and [B] uint8 buffers (numpy or torch)."""
    _check("cora_denoise_step", lib().cora_denoise_step(session, int(block), int(step), ptr(conf_out),
                                                        ptr(argmax_out), ptr(done_out)))
    return cora_session_finished(session)


def cora_session_finished(session) -> bool:
    out = np.zeros(1, np.uint8)
    _check("cora_session_finished", lib().cora_session_finished(session, ptr(out)))
    return bool(out[0])


def cora_session_run(session) -> tuple:
    """Whole decode (one graph launch where available): (steps, on_device)."""
    steps = np.zeros(1, np.int32)
    dev = np.zeros(1, np.uint8)
    _check("cora_session_run", lib().cora_session_run(session, ptr(steps), ptr(dev)))
    return int(steps[0]), bool(dev[0])


def cora_session_disagreement(session, dense, B):
    """Per-sequence (n_acc, n_acc_diff, n_out_diff) against the dense session's canvas."""
    n = [np.zeros(B, np.int64) for _ in range(3)]
    _check("cora_session_disagreement", lib().cora_session_disagreement(session, dense, *[ptr(a) for a in n]))
    return tuple(n)


def cora_session_read(session, B, S, G, BL, eq1_rows=None) -> dict:
    """eq1_rows: rows of persist/prev/conf/argmax per sequence: BL, or G for a
    carry-over persistence session (the library writes B * G entries there,
    so a smaller buffer would be overrun)."""
    E = BL if eq1_rows is None else eq1_rows
    out = dict(tokens=np.zeros((B, S), np.int32), state=np.zeros((B, G), np.uint8),
               persist=np.zeros((B, E), np.int32), prev=np.zeros((B, E), np.int32),
               ctrl=np.zeros((B, 4), np.int32), conf=np.zeros((B, E), np.float32),
               argmax=np.zeros((B, E), np.int32), unmask=np.zeros((B, BL), np.uint8),
               accept=np.zeros((B, BL), np.uint8))
    _check("cora_session_read", lib().cora_session_read(session, *[ptr(out[k]) for k in (
        "tokens", "state", "persist", "prev", "ctrl", "conf", "argmax", "unmask", "accept")]))
    return out


def cora_session_write(session, tokens=None, state=None, persist=None, prev=None, ctrl=None) -> None:
    def c(a, dt):
        return None if a is None else np.ascontiguousarray(a, dtype=dt)
    arrs = [c(tokens, np.int32), c(state, np.uint8), c(persist, np.int32), c(prev, np.int32), c(ctrl, np.int32)]
    _check("cora_session_write", lib().cora_session_write(session, *[ptr(a) for a in arrs]))


def cora_session_profile_step(session, n_layers: int):
    """Runs one step eagerly with events around each launch: [(kind name, ms), ...]."""
    cap = 4 + 7 * n_layers
    kinds = np.zeros(cap, np.int32)
    ms = np.zeros(cap, np.float32)
    n = np.zeros(1, np.int32)
    _check("cora_session_profile_step", lib().cora_session_profile_step(session, cap, ptr(kinds), ptr(ms), ptr(n)))
    return [(KIND_NAMES[int(kinds[i])], float(ms[i])) for i in range(int(n[0]))]


def cora_session_stream(session) -> int:
    out = C.c_void_p()
    _check("cora_session_stream", lib().cora_session_stream(session, C.byref(out)))
    return out.value or 0


def cora_session_batched_passes(session) -> int:
    out = np.zeros(1, np.int64)
    _check("cora_session_batched_passes", lib().cora_session_batched_passes(session, ptr(out)))
    return int(out[0])


def cora_generate(model, prompt, gen_len, block_len, steps_per_block, tau, K,
                  options: DecodeOptions | None = None):
    """prompt: [B, P] int32 (host numpy or device tensor).  Returns (tokens [B, G], passes [B], batched)."""
    B, P = prompt.shape
    tokens = np.zeros((B, gen_len), np.int32)
    passes = np.zeros(B, np.int64)
    batched = np.zeros(1, np.int64)
    if isinstance(prompt, np.ndarray):
        prompt = np.ascontiguousarray(prompt, dtype=np.int32)
    if options is None:
        _check("cora_generate", lib().cora_generate(model, ptr(prompt), B, P, gen_len, block_len, steps_per_block,
                                                    tau, K, ptr(tokens), ptr(passes), ptr(batched)))
    else:
        _check("cora_generate_ex", lib().cora_generate_ex(
            model, ptr(prompt), B, P, gen_len, block_len, steps_per_block, tau, K,
            C.cast(C.byref(options), C.c_void_p), ptr(tokens), ptr(passes), ptr(batched)))
    return tokens, passes, int(batched[0])


def cora_gate_transfer(conf, argmax, prev, persist, state, tokens, B, R, k, tau, K, unmask, accept, done,
                       stream=None) -> None:
    _check("cora_gate_transfer", lib().cora_gate_transfer(
        ptr(conf), ptr(argmax), ptr(prev), ptr(persist), ptr(state), ptr(tokens), B, R, k, tau, K,
        ptr(unmask), ptr(accept), ptr(done), _stream(stream)))


def cora_reduce_top1(logits, rows, V, conf, argmax, stream=None) -> None:
    _check("cora_reduce_top1", lib().cora_reduce_top1(ptr(logits), rows, V, ptr(conf), ptr(argmax),
                                                      _stream(stream)))


def cora_reduce_top1_noalloc(logits, rows, V, conf, argmax, stream=None) -> None:
    _check("cora_reduce_top1_noalloc", lib().cora_reduce_top1_noalloc(ptr(logits), rows, V, ptr(conf), ptr(argmax),
                                                                      _stream(stream)))


def cora_reduce_gate(logits, B, R, V, conf, argmax, prev, persist, state, tokens, k, tau, K, unmask, accept, done,
                     stream=None) -> None:
    _check("cora_reduce_gate", lib().cora_reduce_gate(
        ptr(logits), B, R, V, ptr(conf), ptr(argmax), ptr(prev), ptr(persist), ptr(state), ptr(tokens), k, tau, K,
        ptr(unmask), ptr(accept), ptr(done), _stream(stream)))


def cora_gemm_plan(M: int, N: int, K: int, epilogue: int, num_sms: int):
    """Host-side work split of a GEMM (cora_gemm_plan): (info dict, segments [n, 6] int32 array of
    unit, tile, kb0, kb1, row block, column block in each unit's visiting order)."""
    info = np.zeros(7, np.int32)
    n = np.zeros(1, np.int32)
    _check("cora_gemm_plan", lib().cora_gemm_plan(M, N, K, epilogue, num_sms, ptr(info), None, 0, ptr(n)))
    seg = np.zeros((max(int(n[0]), 1), 6), np.int32)
    _check("cora_gemm_plan", lib().cora_gemm_plan(M, N, K, epilogue, num_sms, ptr(info), ptr(seg), int(n[0]),
                                                  ptr(n)))
    keys = ("kernel", "units", "tiles", "kb", "splits", "split_pair", "dp_waves")
    return dict(zip(keys, (int(x) for x in info))), seg[: int(n[0])]


def cora_op_gemm(A, B, Cm, M, N, K, ldc, epilogue, rope=None, seq=0, head_dim=0, rope_cols=0, stream=None) -> None:
    _check("cora_op_gemm", lib().cora_op_gemm(ptr(A), ptr(B), ptr(Cm), M, N, K, ldc, epilogue, ptr(rope), seq,
                                              head_dim, rope_cols, _stream(stream)))


def cora_op_attention(qkv, out, B, S, Hq, Hkv, hd, stream=None) -> None:
    _check("cora_op_attention", lib().cora_op_attention(ptr(qkv), ptr(out), B, S, Hq, Hkv, hd, _stream(stream)))


def cora_op_attention_rows(qkv, out, B, S, Hq, Hkv, hd, q_start, q_len, stream=None) -> None:
    _check("cora_op_attention_rows", lib().cora_op_attention_rows(ptr(qkv), ptr(out), B, S, Hq, Hkv, hd, q_start,
                                                                  q_len, _stream(stream)))


def cora_op_rmsnorm(x, w, out, M, d, eps, stream=None) -> None:
    _check("cora_op_rmsnorm", lib().cora_op_rmsnorm(ptr(x), ptr(w), ptr(out), M, d, eps, _stream(stream)))


def cora_op_lm_head_top1(x, W, R, V, d, conf, argmax, stream=None) -> None:
    _check("cora_op_lm_head_top1", lib().cora_op_lm_head_top1(ptr(x), ptr(W), R, V, d, ptr(conf), ptr(argmax),
                                                              _stream(stream)))


def cora_synth_normal_bf16(out, count, key, start, scale, stream=None) -> None:
    _check("cora_synth_normal_bf16", lib().cora_synth_normal_bf16(ptr(out), count, key, start, float(scale),
                                                                  _stream(stream)))


def cora_check_wait_timeout(which: int) -> int:
    """Runs the bounded-wait self-check (0: an mbarrier nothing arrives at, 1: a
    flag nothing sets); returns the error code the kernel recorded."""
    code = np.zeros(1, np.int32)
    _check("cora_check_wait_timeout", lib().cora_check_wait_timeout(int(which), ptr(code)))
    return int(code[0])


def cora_device_error(clear: bool = False) -> int:
    code = np.zeros(1, np.int32)
    _check("cora_device_error", lib().cora_device_error(ptr(code), int(clear)))
    return int(code[0])
