"""The kernels' bounded waits, exercised without a fault: a wait that runs out reports
NAMOH_DEV_TIMEOUT with the barrier and the warp that gave up, every role of the attention kernel
drains its copies and MMAs and exits, and the context and the plan stay usable.

The attention kernel is run with every CTA's first query tile withheld (a barrier nothing
completes) and a 1 ms limit on the MMA issuer's waits (namoh_attention_timeout_probe).
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import dev_bf16

pytestmark = pytest.mark.gpu


def test_attention_wait_runs_out_and_reports():
    import paper_2609_38832_gb300 as namoh
    wl = ni.PrefillWorkload("timeout_probe", B=2, T=700, H=4, K=2, d=128, seed=70)
    q, k, v = (dev_bf16(a) for a in wl.qkv())
    ro = namoh.namoh_route(torch.from_numpy(wl.scores()).cuda(), wl.Kr)
    kw = dict(B=wl.B, T=wl.T, H=wl.H, K=wl.K)
    y_ref, _, _ = namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, rope_base=wl.base,
                                      status=ro.status, **kw)
    plan = namoh.namoh_attention_plan(ro.seg_offsets, **kw)
    q_rot, kc, vc = namoh.namoh_rope_pack(q, k, v, ro.seg_offsets, rope_base=wl.base, status=ro.status, plan=plan,
                                          **kw)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    namoh.namoh_attention_timeout_probe(q_rot, kc, vc, ro.seg_offsets, ro.row_src, ro.gate, plan,
                                        wait_limit_ns=1_000_000, status=st, **kw)
    torch.cuda.synchronize()  # the call returned: every CTA exited
    word = int(st.item()) & 0xFFFFFFFF
    assert word & namoh.NAMOH_DEV_TIMEOUT, hex(word)
    assert (word >> 24) & 0xFF == 5, hex(word)      # the MMA issuer's warp gave up
    assert (word >> 16) & 0x7F == 4, hex(word)      # on the query tile's barrier
    assert word & (namoh.NAMOH_DEV_CAPACITY | namoh.NAMOH_DEV_NONFINITE_SCORE) == 0
    # the context and the same plan still work: the next call gives namoh_prefill's bytes
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = namoh.namoh_attention(q_rot, kc, vc, ro.seg_offsets, ro.row_src, ro.gate, plan, status=st2, **kw)
    torch.cuda.synchronize()
    assert int(st2.item()) == 0
    assert torch.equal(y.view(torch.int16), y_ref.view(torch.int16))


def test_timeout_probe_rejects_limits_out_of_range():
    import paper_2609_38832_gb300 as namoh
    t = torch.zeros(16, dtype=torch.int32, device="cuda")
    for bad in (0, 999, 3_000_000_000):
        with pytest.raises(namoh.NamohError):
            namoh.namoh_attention_timeout_probe(t, t, t, t, t, t, t, B=1, T=1, H=1, K=1, wait_limit_ns=bad)
