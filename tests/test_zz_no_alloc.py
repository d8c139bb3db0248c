"""rf_attn_noalloc: attention for callers that cannot allocate device memory.

Some callers of this library cannot call cudaMalloc: code running inside another
engine's execution callback that forbids allocation, serving loops that must not
take cudaMalloc's device-wide synchronisation, or C hosts without a device
allocator.  rf_attn_noalloc gives them the same split-KV attention using scratch
that the library holds itself.  This test calls it through the C ABI twice in a
row and checks each result against the regular entry point given a workspace,
with the tolerances the other attention tests use.
"""
import math

import numpy as np
import pytest
import torch

from attn_check import compare

pytestmark = pytest.mark.gpu

DEV = "cuda"
SENTINEL = 7.0


@pytest.mark.parametrize("F,N,H,d,mask", [
    (3, 1560, 2, 128, [1, 1, 1]),      # 38 work items on 152 CTAs: split into 4 KV ranges
    (4, 64, 2, 64, [1, 0, 0, 1]),      # head dim 64, a skipped frame
    (13, 1560, 12, 128, [1] * 13),     # 960 items: the last round is split 3 ways
])
def test_noalloc_matches_workspace_entry_point(cuda_lib, F, N, H, d, mask):
    rf = cuda_lib
    g = torch.Generator(device=DEV).manual_seed(F * 131 + N + d)
    Q, K, V = (torch.randn(F * N, H, d, generator=g, device=DEV).to(torch.bfloat16)
               for _ in range(3))
    scale = 1.0 / math.sqrt(d)
    act = torch.zeros(F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(torch.tensor(mask, dtype=torch.uint8, device=DEV), F, N, act, skp,
                           None, cnt)

    # the existing entry point, with a caller-allocated (zero-filled) workspace
    ws = torch.zeros((rf.rf_attn_workspace_bytes(d) + 3) // 4, dtype=torch.int32, device=DEV)
    O_ref = torch.empty(F * N, H, d, dtype=torch.bfloat16, device=DEV)
    L_ref = torch.empty(H, F * N, dtype=torch.float32, device=DEV)
    rf.rf_attn(O_ref, L_ref, Q, K, V, Q.stride(0), O_ref.stride(0), F, N, H, d, act, cnt, scale,
               ws, status)
    torch.cuda.synchronize()
    assert status.item() == 0

    rows = [f * N + p for f in range(F) if mask[f] for p in range(N)]
    skipped = sorted(set(range(F * N)) - set(rows))
    for call in range(2):  # two calls in a row share the library's scratch
        O = torch.full((F * N, H, d), SENTINEL, dtype=torch.bfloat16, device=DEV)
        L = torch.full((H, F * N), SENTINEL, dtype=torch.float32, device=DEV)
        rf.rf_attn_noalloc(O, L, Q, K, V, Q.stride(0), O.stride(0), F, N, H, d, act, cnt, scale,
                           status)
        torch.cuda.synchronize()
        assert status.item() == 0
        compare(O.float()[rows].cpu().numpy(), O_ref.float()[rows].cpu().numpy(),
                L[:, rows].cpu().numpy(), L_ref[:, rows].cpu().numpy(), f"noalloc call {call}")
        if skipped:
            assert (O[skipped].float() == SENTINEL).all()
