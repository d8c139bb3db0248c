"""Failure handling on the GPU without faulting it.

A device wait that runs out of time must end in an error status the host can read,
with the context still usable afterwards.  rf_selftest_bounded_wait runs the attention
kernel's bounded mbarrier wait on a barrier nothing arrives at (inside a CTA holding
tensor memory); the test checks the status, the time it took, and that attention runs
correctly right after."""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from attn_check import compare

pytestmark = pytest.mark.gpu


def test_bounded_wait_expires_with_status_and_context_survives(cuda_lib):
    rf = cuda_lib
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    rf.rf_selftest_bounded_wait(status, 50_000)  # 50 ms
    b.record()
    torch.cuda.synchronize()
    assert status.item() & 0xFF == 5            # RF_ERR_DEVICE_TIMEOUT
    ms = a.elapsed_time(b)
    assert 45.0 <= ms < 2000.0, ms

    # the context and tensor memory are usable: a full attention call right after
    w = wl.get("tiny")
    Q, K, V = (x.cuda() for x in wl.qkv(w))
    O = torch.zeros_like(Q)
    act = torch.zeros(w.F, dtype=torch.int32, device="cuda")
    skp = torch.zeros_like(act)
    cnt = torch.zeros(2, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    rf.rf_schedule_compact(torch.ones(w.F, dtype=torch.uint8, device="cuda"), w.F, w.N, act, skp,
                           None, cnt)
    rf.rf_attn(O, None, Q, K, V, Q.stride(0), O.stride(0), w.F, w.N, w.H, w.d, act, cnt,
               w.softmax_scale, None, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    Oref, _ = oracle.attention(Q.cpu(), K.cpu(), V.cpu(), range(w.S_tok), w.softmax_scale)
    compare(O.cpu().float().numpy(), Oref, label="after self-test")


def test_selftest_rejects_bad_limits(cuda_lib):
    rf = cuda_lib
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for bad in (0, 99, 2_000_001):
        with pytest.raises(rf.RFError):
            rf.rf_selftest_bounded_wait(status, bad)
