"""The bench's algorithmic work per launch, against hand-derived totals.

The roofline fractions in the bench line divide these FLOP and byte counts by
measured kernel times, so a wrong factor here would misstate every fraction.
The expected totals are worked out by hand from the workload shapes (a dense
pass = four projections per layer, 2 M N K FLOPs each, plus QK^T and PV of the
bidirectional attention, 2 * 2 B Hq S^2 hd; the LM head streams V d bf16
weights once per pass).
"""

import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
from paper_2608_11235_gb300 import configs  # noqa: E402

GEMM_KINDS = ["gemm_qkv_rope", "gemm_o_resid", "gemm_gate_up_swiglu", "gemm_down_resid"]


@pytest.mark.parametrize("name,gemm_tf,attn_tf", [
    # M = 512: 2 * 512 * 4096 * (12288 + 4096 + 24576 + 12288) * 32 layers
    ("llada8b-shape-256+256", 7.146, 0.1374),
    # M = 8 * 1536: 24x the tokens of the above; attention 8 * (1536 / 512)^2 = 72x
    ("llada8b-shape-512+1024-b8", 171.5, 9.895),
    # M = 4 * 768: 2 * 3072 * 3584 * (4608 + 3584 + 37888 + 18944) * 28 layers
    ("dream7b-shape-256+512-b4", 40.09, 0.947),
])
def test_pass_flops_match_hand_totals(name, gemm_tf, attn_tf):
    cfg = configs.PRESETS[name]
    c = bench.kernel_costs(cfg)
    L = cfg["n_layers"]
    assert sum(c[k] for k in GEMM_KINDS) * L / 1e12 == pytest.approx(gemm_tf, rel=2e-3)
    assert c["attention"] * L / 1e12 == pytest.approx(attn_tf, rel=2e-3)


def test_lm_head_bytes_and_flops():
    cfg = configs.PRESETS["llada8b-shape-256+256"]
    c = bench.kernel_costs(cfg)
    # 126464 x 4096 bf16 weights + 32 active rows x 4096 bf16
    assert c["lm_head_top1_bytes"] == 126464 * 4096 * 2 + 32 * 4096 * 2
    assert c["lm_head_top1_flops"] == 2 * 32 * 4096 * 126464
    dream = bench.kernel_costs(configs.PRESETS["dream7b-shape-256+512-b4"])
    assert dream["lm_head_top1_bytes"] == 152064 * 3584 * 2 + 4 * 32 * 3584 * 2
