"""CPU checks of the C ABI: the library builds, loads, exports every declared
entry point, and rejects bad arguments with CORA_EINVAL before touching a GPU."""

import os
import re

import numpy as np
import pytest

from paper_2608_11235_gb300 import build, cora

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    return cora.lib()


def declared_entry_points():
    text = open(os.path.join(ROOT, "include", "cora.h")).read()
    return sorted(set(re.findall(r"CORA_API\s+(?:const\s+char\s*\*|int)\s+(cora_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported(L):
    names = declared_entry_points()
    assert len(names) >= 20
    for n in names:
        assert hasattr(L, n), n
    assert sorted(cora.EXPORTED) == names


def test_version(L):
    assert cora.cora_version() == 200


def test_invalid_arguments_rejected_before_launch(L):
    z = np.zeros(64, np.int32)
    p = z.ctypes.data
    # R > 32: one warp per block
    rc = L.cora_gate_transfer(p, p, p, p, p, p, 1, 33, 1, 0.5, 1, p, p, p, None)
    assert rc == cora.CORA_EINVAL and b"R <= 32" in L.cora_last_error()
    rc = L.cora_gate_transfer(None, p, p, p, p, p, 1, 8, 1, 0.5, 1, p, p, p, None)
    assert rc == cora.CORA_EINVAL
    rc = L.cora_op_gemm(p, p, p, 128, 256, 63, 256, 0, None, 0, 0, 0, None)       # K % 64 != 0
    assert rc == cora.CORA_EINVAL
    rc = L.cora_op_gemm(p, p, p, 128, 384, 64, 384, 2, None, 0, 0, 0, None)       # SWIGLU needs N % 256
    assert rc == cora.CORA_EINVAL
    rc = L.cora_op_attention(p, p, 1, 16, 6, 4, 128, None)                         # Hq % Hkv != 0
    assert rc == cora.CORA_EINVAL
    rc = L.cora_op_lm_head_top1(p, p, 257, 100, 64, p, p, None)                    # R > 256
    assert rc == cora.CORA_EINVAL
    rc = L.cora_reduce_top1(p, 0, 10, p, p, None)
    assert rc == cora.CORA_EINVAL


def test_model_config_validation(L):
    cfg = dict(n_layers=1, d_model=96, n_heads=2, n_kv_heads=2, head_dim=64, ffn=64, vocab=10, mask_id=9,
               rope_theta=1e4, norm_eps=1e-5)
    with pytest.raises(cora.CoraError) as e:
        cora.cora_model_create(cfg, {"embed": 16, "lm_head": 16})
    assert e.value.code == cora.CORA_EINVAL
    cfg.update(d_model=128, head_dim=96)
    with pytest.raises(cora.CoraError) as e:
        cora.cora_model_create(cfg, {"embed": 16, "lm_head": 16})
    assert e.value.code == cora.CORA_EINVAL


def test_session_argument_validation(L):
    from ctypes import byref, c_void_p
    out = c_void_p()
    z = np.zeros(8, np.int32)
    assert L.cora_session_create(16, 1, z.ctypes.data, 8, 64, 33, 32, 0.5, 1, byref(out)) == cora.CORA_EINVAL
    assert L.cora_session_create(16, 1, z.ctypes.data, 8, 60, 32, 32, 0.5, 1, byref(out)) == cora.CORA_EINVAL
    assert L.cora_session_create(16, 9, z.ctypes.data, 8, 64, 32, 32, 0.5, 1, byref(out)) == cora.CORA_EINVAL
    assert L.cora_session_create(16, 1, z.ctypes.data, 8, 64, 32, 0, 0.5, 1, byref(out)) == cora.CORA_EINVAL


def test_decode_options_validation(L):
    """Unknown or not-yet-supported decoding options are rejected before the
    model is touched (the model handle here is a dummy)."""
    from ctypes import byref, c_void_p
    out = c_void_p()
    z = np.zeros(8, np.int32)
    for opt in (cora.decode_options(schedule=2), cora.decode_options(persistence=5),
                cora.decode_options(eos_id=-7)):
        rc = L.cora_session_create_ex(16, 1, z.ctypes.data, 8, 64, 32, 32, 0.5, 1, byref(opt), byref(out))
        assert rc == cora.CORA_EINVAL, (opt.schedule, opt.persistence, opt.eos_id)


def test_unknown_weight_dtype_rejected(L):
    cfg = dict(n_layers=1, d_model=128, n_heads=2, n_kv_heads=2, head_dim=64, ffn=64, vocab=10, mask_id=9,
               rope_theta=1e4, norm_eps=1e-5)
    with pytest.raises(cora.CoraError) as e:
        cora.cora_model_create(cfg, {"embed": 16, "lm_head": 16, "dtype": 7})
    assert e.value.code == cora.CORA_EINVAL and "dtype" in str(e.value)


def test_denoise_step_argument_validation(L):
    """NULL session and block/step below -1 are rejected before the session is read."""
    assert L.cora_denoise_step(None, -1, -1, None, None, None) == cora.CORA_EINVAL
    assert L.cora_denoise_step(16, -2, 0, None, None, None) == cora.CORA_EINVAL
    assert L.cora_denoise_step(16, 0, -5, None, None, None) == cora.CORA_EINVAL
    assert L.cora_session_finished(None, None) == cora.CORA_EINVAL
