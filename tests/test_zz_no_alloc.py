"""The allocation-free Eq. 1 reduction matches the regular one.

cora_reduce_top1_noalloc exists for callers that cannot allocate device
memory when they call it (their memory pool already owns the device, or
their loop must not enter the allocator): its scratch is a fixed array
inside the library.  This test calls it through the C ABI twice in a row
(the second call reuses the array the first one left behind) and compares
each result with cora_reduce_top1 on the same logits, within the tolerance
the other Eq. 1 tests use, and checks that the device's free memory does not
change across the second call.  It lives in its own file, collected last.
"""

import numpy as np
import pytest
import torch

from paper_2608_11235_gb300 import build, cora, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available()
    build.build()
    cora.lib()


@pytest.mark.parametrize("rows,V", [(64, 126464), (3, 1001), (256, 32768)])
def test_noalloc_matches_regular_reduction_twice(rows, V):
    hist = synth.gate_history(9, 1, rows, V)
    lg = torch.from_numpy(synth.gate_logits_bf16(9, 1, rows, V, hist[-1]).reshape(rows, V).view(np.int16)).cuda()
    ref_c = torch.empty(rows, dtype=torch.float32, device="cuda")
    ref_a = torch.empty(rows, dtype=torch.int32, device="cuda")
    cora.cora_reduce_top1(lg, rows, V, ref_c, ref_a)
    rc, ra = ref_c.cpu().numpy(), ref_a.cpu().numpy()
    outs = [(torch.empty(rows, dtype=torch.float32, device="cuda"), torch.empty(rows, dtype=torch.int32, device="cuda"))
            for _ in range(2)]
    free = []
    for c, a in outs:
        c.fill_(-1.0)
        a.fill_(-1)
        torch.cuda.synchronize()
        free.append(torch.cuda.mem_get_info()[0])        # cudaMemGetInfo before the call
        cora.cora_reduce_top1_noalloc(lg, rows, V, c, a)
        torch.cuda.synchronize()
        free.append(torch.cuda.mem_get_info()[0])        # ... and after it
        assert np.array_equal(a.cpu().numpy(), ra)
        assert np.all(np.abs(c.cpu().numpy() - rc) <= 1e-4 * rc + 1e-7)
    # The first call on a device may load the library part holding the fixed
    # array (lazy module loading); the second call reserves no device memory.
    assert free[2] == free[3], (free[2], free[3])


def test_noalloc_rejects_rows_beyond_the_fixed_scratch():
    lg = torch.zeros((8, 16), dtype=torch.int16, device="cuda")
    c = torch.empty(8, dtype=torch.float32, device="cuda")
    a = torch.empty(8, dtype=torch.int32, device="cuda")
    with pytest.raises(cora.CoraError) as e:
        cora.cora_reduce_top1_noalloc(lg, 16385, 16, c, a)
    assert e.value.code == cora.CORA_EINVAL
