"""CPU checks of the GEMM work split (cora_gemm_plan: the host computes the
kernels' own rules and segment walk, no GPU needed): every (tile, k-block)
iteration of a projection is assigned to exactly one unit, tiles map one to
one onto the output's row and column blocks, and the schedule chosen for the
projections of the 8B-class passes and of prefix-cache passes is the intended
one (two k-pieces sharing the fix-up, skewed pieces, stream-K, whole tiles,
data-parallel waves)."""

import itertools

import numpy as np
import pytest

from paper_2608_11235_gb300 import build, cora

SMS = 152
STORE, RESID, SWIGLU, ROPE = cora.EPI_STORE_BF16, cora.EPI_RESID_F32, cora.EPI_SWIGLU, cora.EPI_ROPE_BF16


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    cora.lib()


def projections(M, d, n_q, n_kv, ffn):
    """QKV, O, gate/up, down of one layer: (M, N, K, epilogue)."""
    f_pad = (ffn + 127) // 128 * 128
    return [(M, n_q + 2 * n_kv, d, ROPE), (M, d, n_q, RESID), (M, 2 * f_pad, d, SWIGLU), (M, d, f_pad, RESID)]


LLADA = dict(d=4096, n_q=4096, n_kv=4096, ffn=12288)
DREAM = dict(d=3584, n_q=3584, n_kv=512, ffn=18944)
TINY = dict(d=256, n_q=256, n_kv=256, ffn=688)

SHAPES = (projections(512, **LLADA) + projections(12288, **LLADA) + projections(3072, **DREAM) +
          [s for M in (32, 64, 96, 128, 160, 192, 224, 256) for s in projections(M, **LLADA)] +
          projections(96, **TINY) + projections(288, **TINY) +
          [(300, 512, 320, STORE), (130, 256, 1024, RESID), (1800, 10240, 192, STORE), (100, 16384, 512, RESID),
           (2048, 12288, 256, STORE), (1536, 8192, 512, RESID), (96, 768, 2048, STORE), (256, 256, 4096, STORE)])


def blocks(info, M, N, epi):
    if info["kernel"] == 2:
        return (M + 255) // 256, N // 256
    bn = 256 if (N % 256 == 0 or epi == SWIGLU) else 128
    return (M + 127) // 128, N // bn


@pytest.mark.parametrize("M,N,K,epi", SHAPES)
def test_every_iteration_assigned_once(M, N, K, epi):
    info, seg = cora.cora_gemm_plan(M, N, K, epi, SMS)
    if info["kernel"] == 0:  # the few-row kernel (at most 64 rows) has its own split
        assert M <= 64 and len(seg) == 0
        return
    KB = K // 64
    num_m, num_n = blocks(info, M, N, epi)
    assert info["tiles"] == num_m * num_n and info["kb"] == KB
    assert 1 <= info["units"] <= (SMS // 2 if info["kernel"] == 2 else SMS)
    count = np.zeros((info["tiles"], KB), np.int64)
    coords = {}
    for u, t, kb0, kb1, mb, nb in seg:
        assert 0 <= u < info["units"] and 0 <= t < info["tiles"] and 0 <= kb0 < kb1 <= KB
        assert 0 <= mb < num_m and 0 <= nb < num_n
        assert coords.setdefault(t, (mb, nb)) == (mb, nb)
        count[t, kb0:kb1] += 1
    assert np.all(count == 1)
    assert len(set(coords.values())) == info["tiles"]  # one tile per output block
    # a unit's only mid-tile start is its first segment (it contributes a partial)
    for u in range(info["units"]):
        rows = seg[seg[:, 0] == u]
        assert np.all(rows[1:, 2] == 0)


def test_llada_dense_pass_schedules():
    qkv, o, gu, down = [cora.cora_gemm_plan(*s, SMS)[0] for s in projections(512, **LLADA)]
    assert qkv["kernel"] == 2 and qkv["units"] == 76 and qkv["splits"] == 0 and qkv["dp_waves"] == 0  # stream-K
    for p in (o, down):  # 32 pair-tiles, two pieces each sharing the fix-up
        assert p["units"] == 64 and p["splits"] == 2 and p["split_pair"] == 1
    assert gu["dp_waves"] == 2 and gu["units"] == 76  # 192 tiles: two waves of 76 + a stream-K remainder


def test_pair_pieces_split_k_in_halves():
    for M, N, K, epi in [(512, 4096, 4096, RESID), (256, 4096, 12288, RESID), (96, 4096, 4096, RESID)]:
        info, seg = cora.cora_gemm_plan(M, N, K, epi, SMS)
        assert info["split_pair"] == 1 and info["units"] == 2 * info["tiles"]
        KB = K // 64
        for t in range(info["tiles"]):
            mine = seg[seg[:, 1] == t]
            assert sorted(mine[:, 0].tolist()) == [2 * t, 2 * t + 1]
            assert sorted((int(a), int(b)) for a, b in mine[:, 2:4]) == [(0, KB // 2), (KB // 2, KB)]


def test_one_row_block_whole_tiles():
    # prefix-cache QKV at 129-256 rows: 48 pair-tiles, no more than the 76 pairs
    for M in (160, 192, 256):
        info, seg = cora.cora_gemm_plan(M, 12288, 4096, ROPE, SMS)
        assert info["kernel"] == 2 and info["units"] == 48 and info["splits"] == 0
        assert len(seg) == 48 and np.all(seg[:, 2] == 0) and np.all(seg[:, 3] == 64)
        assert sorted(seg[:, 0].tolist()) == list(range(48))


def test_long_k_keeps_skewed_pieces_on_the_one_cta_kernel():
    info, seg = cora.cora_gemm_plan(96, 4096, 12288, RESID, SMS)
    assert info["kernel"] == 1 and info["splits"] == 4 and info["split_pair"] == 0
    for t in range(info["tiles"]):
        mine = seg[seg[:, 1] == t]
        assert len(mine) == 4
        finisher = [int(b - a) for a, b in mine[:, 2:4] if a == 0][0]
        assert finisher == max(int(b - a) for a, b in mine[:, 2:4])  # the piece holding k-block 0 is longest


def test_many_row_blocks_run_waves():
    info, seg = cora.cora_gemm_plan(12288, 24576, 4096, SWIGLU, SMS)
    assert info["dp_waves"] == info["tiles"] // info["units"]
    whole = seg[(seg[:, 2] == 0) & (seg[:, 3] == 64)]
    assert len(whole) >= info["dp_waves"] * info["units"]


def test_plan_rejects_bad_arguments():
    info = np.zeros(7, np.int32)
    n = np.zeros(1, np.int32)
    L = cora.lib()
    assert L.cora_gemm_plan(512, 4096, 100, STORE, SMS, cora.ptr(info), None, 0, cora.ptr(n)) != 0   # K % 64
    assert L.cora_gemm_plan(512, 4000, 4096, STORE, SMS, cora.ptr(info), None, 0, cora.ptr(n)) != 0  # N % 128
    assert L.cora_gemm_plan(0, 4096, 4096, STORE, SMS, cora.ptr(info), None, 0, cora.ptr(n)) != 0
    assert L.cora_gemm_plan(512, 4096, 4096, 7, SMS, cora.ptr(info), None, 0, cora.ptr(n)) != 0
    assert L.cora_gemm_plan(512, 4096, 4096, STORE, SMS, None, None, 0, cora.ptr(n)) != 0
