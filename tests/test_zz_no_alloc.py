"""grkv_select_noalloc: selection for callers that cannot give the library a
workspace (an engine plugin whose host owns all device memory, a serving loop
that must not call cudaMalloc on the request path).  Its scratch is a fixed
array in the library's device image, so its results must match grkv_select
with a caller workspace exactly, call after call, even though every call
reuses the same array.  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from paper_2605_31105_gb300 import binding as b

pytestmark = pytest.mark.gpu


def _scores(seed, units, prefix):
    rng = np.random.default_rng(seed)
    s = rng.random((units, prefix), dtype=np.float32) ** 4
    s[:, ::97] = s[:, 1::97]          # plant ties across pooling windows
    return torch.from_numpy(s).cuda()


@pytest.mark.parametrize("pool_type", ["max", "avg"])
def test_noalloc_select_matches_workspace_select_twice(grkv_lib, pool_type):
    # n - w > 32768 takes the selection that pools into the shared array; the
    # shorter shapes stay in shared memory.  Long shapes back to back with
    # other sizes show that a call never reads what an earlier one left there.
    shapes = [(2, 65600, 32, 512), (3, 40000, 16, 300), (8, 8192, 32, 512),
              (2, 65600, 32, 2048)]
    for call, (units, n, w, budget) in enumerate(shapes):
        p = b.params(units, 4, n, w, budget, pool_type=pool_type)
        scores = _scores(100 + call, units, n - w)
        ws = torch.empty(b.grkv_workspace_size(p), dtype=torch.uint8, device="cuda")
        ref = torch.empty((units, budget), dtype=torch.int32, device="cuda")
        b.grkv_select(p, scores, ref, ws)
        got = torch.full((units, budget), -1, dtype=torch.int32, device="cuda")
        assert b.grkv_select_noalloc(p, scores, got) == b.GRKV_OK
        torch.cuda.synchronize()
        assert torch.equal(got, ref), f"call {call}: indices differ"


def test_noalloc_select_rejects_sizes_beyond_its_array(grkv_lib):
    p = b.params(128, 4, 40032, 32, 2048)        # 128 * 40000 floats > 4 Mi
    z = torch.empty(16, dtype=torch.float32, device="cuda")
    zi = torch.empty(16, dtype=torch.int32, device="cuda")
    assert b.grkv_select_noalloc(p, z, zi, check=False) == b.GRKV_ERR_WORKSPACE_TOO_SMALL


def test_noalloc_select_takes_any_unit_count_for_short_prefixes(grkv_lib):
    """256 units of n - w = 32736 (the 32-layer workload's selection) need no
    scratch at all, so the array's size does not limit them."""
    units, n, w, budget = 256, 32768, 32, 2048
    p = b.params(units, 4, n, w, budget)
    scores = _scores(7, units, n - w)
    ws = torch.empty(b.grkv_workspace_size(p), dtype=torch.uint8, device="cuda")
    ref = torch.empty((units, budget), dtype=torch.int32, device="cuda")
    b.grkv_select(p, scores, ref, ws)
    got = torch.full((units, budget), -1, dtype=torch.int32, device="cuda")
    assert b.grkv_select_noalloc(p, scores, got) == b.GRKV_OK
    torch.cuda.synchronize()
    assert torch.equal(got, ref)
