"""namoh_route_noalloc: routing for callers that cannot allocate device memory.

Some callers cannot hand the library a workspace: code inside a stream capture (where
cudaMalloc would break the capture), serving loops that must never synchronise, and
runtimes that own all device memory through their own pools.  This entry point takes
its scratch from an array built into the library instead.  It must give exactly what
the workspace entry point gives, call after call (the array keeps the previous call's
contents).  This file is collected last so that a failure here cannot hide others.
"""
import ctypes

import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import GATE_RTOL

pytestmark = pytest.mark.gpu


def _noalloc(lib, scores, K):
    B, T, H = scores.shape
    i32 = dict(dtype=torch.int32, device=scores.device)
    out = dict(topk_head=torch.empty((B, T, K), **i32), gate=torch.empty((B, T, K), dtype=torch.float32,
                                                                           device=scores.device),
               rank=torch.empty((B, T, K), **i32), row=torch.empty((B, T, K), **i32),
               seg_offsets=torch.empty(B * H + 1, **i32), row_src=torch.empty(B * T * K, **i32),
               status=torch.zeros(1, **i32))
    rc = lib.namoh_route_noalloc(scores.data_ptr(), B, T, H, K, out["topk_head"].data_ptr(), out["gate"].data_ptr(),
                                 out["rank"].data_ptr(), out["row"].data_ptr(), out["seg_offsets"].data_ptr(),
                                 out["row_src"].data_ptr(), out["status"].data_ptr(),
                                 torch.cuda.current_stream().cuda_stream)
    return rc, out


def test_noalloc_route_matches_workspace_route_in_a_row():
    import paper_2609_38832_gb300 as namoh
    from paper_2609_38832_gb300 import _abi
    lib = _abi.load()
    # different routings in a row, each on the scratch the one before left behind: the balanced
    # workload; a long sequence whose count table (512 chunks x 32 heads per sequence) is large
    # enough for the scan kernel, which uses the second half of the scratch; then a small one
    shapes = ((0, (4, 4096, 16, 4)), (2, (1, 131072, 32, 4)), (1, (3, 1000, 32, 3)))
    assert lib.namoh_route_workspace_size(1, 131072, 32, 4) <= (4 << 20)
    for seed, (B, T, H, K) in shapes:
        scores = torch.from_numpy(ni.router_scores(seed, B, T, H)).cuda()
        rc, got = _noalloc(lib, scores, K)
        assert rc == 0, lib.namoh_status_string(rc)
        ref = namoh.namoh_route(scores, K)
        torch.cuda.synchronize()
        for name in ("topk_head", "rank", "row", "seg_offsets", "row_src"):
            np.testing.assert_array_equal(got[name].cpu().numpy(), getattr(ref, name).cpu().numpy(), err_msg=name)
        np.testing.assert_allclose(got["gate"].cpu().numpy(), ref.gate.cpu().numpy(), rtol=GATE_RTOL, atol=0)
        assert int(got["status"].item()) == 0


def test_noalloc_route_rejects_shapes_beyond_its_scratch():
    from paper_2609_38832_gb300 import _abi
    lib = _abi.load()
    B, T, H, K = 64, 131072, 32, 4  # needs far more than the built-in 4 MiB
    assert lib.namoh_route_workspace_size(B, T, H, K) > (4 << 20)
    fake = ctypes.c_void_p(256)
    rc = lib.namoh_route_noalloc(fake, B, T, H, K, fake, fake, fake, fake, fake, fake, fake, None)
    assert rc == _abi.NAMOH_ERR_WORKSPACE
