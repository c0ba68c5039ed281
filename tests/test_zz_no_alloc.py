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
    shapes = [(8, 8192, 32, 512), (3, 2000, 16, 200)]    # second call: other sizes
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
    p = b.params(256, 4, 32768, 32, 2048)        # 256 * 32736 floats > 4 Mi
    z = torch.empty(16, dtype=torch.float32, device="cuda")
    zi = torch.empty(16, dtype=torch.int32, device="cuda")
    assert b.grkv_select_noalloc(p, z, zi, check=False) == b.GRKV_ERR_WORKSPACE_TOO_SMALL
