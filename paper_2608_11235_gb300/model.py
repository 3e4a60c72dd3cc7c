"""Building a device-resident model from seeded synthetic weights.

bf16 weights are written straight into device memory by the library's own
implementation of the seeded generator (``cora_synth_normal_bf16``), or
uploaded from host arrays made by ``synth`` (same bits); fp32 weights come
from ``synth`` as float32 arrays.  Either is handed to ``cora_model_create``,
which copies (or rounds) them into its kernel layout.
"""

from __future__ import annotations

import numpy as np
import torch

from . import cora, synth

KINDS = {"wq": synth.WQ, "wk": synth.WK, "wv": synth.WV, "wo": synth.WO,
         "w_gate": synth.WGATE, "w_up": synth.WUP, "w_down": synth.WDOWN}


def _device_tensor(cfg: dict, layer: int, kind: int, device) -> torch.Tensor:
    shp = synth.weight_shapes(cfg)[kind]
    t = torch.empty(shp, dtype=torch.int16, device=device)
    key = synth.stream_key(cfg["seed"], synth.tensor_stream(layer, kind))
    scale = float(synth.normal_scale_f32(synth.weight_sigma(cfg, kind)))
    cora.cora_synth_normal_bf16(t, t.numel(), key, 0, scale)
    return t


def _host_tensor(cfg: dict, layer: int, kind: int, device) -> torch.Tensor:
    bits = synth.weight_bf16_bits(cfg, layer, kind)
    return torch.from_numpy(bits.view(np.int16)).to(device)


def _f32_device_tensor(cfg: dict, layer: int, kind: int, device) -> torch.Tensor:
    return torch.from_numpy(synth.weight_f32(cfg, layer, kind)).to(device)


def _f32_host_array(cfg: dict, layer: int, kind: int, device) -> np.ndarray:
    return np.ascontiguousarray(synth.weight_f32(cfg, layer, kind))


def create_model(cfg: dict, device="cuda", on_device_fill: bool = True) -> int:
    """Returns a cora_model handle with the seeded weights of ``cfg``.

    fp32-weight workloads hand the library float32 tensors (device tensors, or
    with ``on_device_fill=False`` pageable host arrays), which it rounds to
    bf16 on the device; bf16 workloads hand it bf16 bit patterns."""
    if synth.is_f32_weights(cfg):
        make = _f32_device_tensor if on_device_fill else _f32_host_array
    else:
        make = _device_tensor if on_device_fill else _host_tensor
    L = cfg["n_layers"]
    t = {"embed": make(cfg, -1, synth.EMBED, device), "lm_head": make(cfg, -1, synth.LM_HEAD, device)}
    for name, kind in KINDS.items():
        t[name] = [make(cfg, l, kind, device) for l in range(L)]
    torch.cuda.synchronize()
    handle = cora.cora_model_create(cfg, t)
    del t
    torch.cuda.empty_cache()
    return handle
