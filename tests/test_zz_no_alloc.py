"""fd_op_attention_static: attention whose key-range-split workspace lives in the library's
static device memory, for callers that cannot allocate device memory (a plug-in held to a
device-memory budget owned by its host framework, or a real-time loop that cannot take an
allocation's device synchronisation). Its results must match fd_op_attention run with a
caller-allocated workspace, call after call, since every call reuses the same static array.

This file is collected last on purpose: it must pass in a fresh process and after every other
test has run in the same process."""
import numpy as np
import pytest
import torch

from helpers import assert_close_scaled, bf16_values, dev, randn

pytestmark = pytest.mark.gpu

fdp = pytest.importorskip("paper_2607_14898_gb300.flashdec")

STATIC_BYTES = 32 << 20  # FD_STATIC_ATTN_SCRATCH_BYTES


def case(Lq, heads, groups, n_keys, seed):
    pitch = -(-n_keys // 128) * 128
    q = bf16_values(randn((Lq, heads * 64), seed, 1.5))
    k = bf16_values(randn((groups, pitch, 64), seed + 1))
    v = randn((groups, pitch, 64), seed + 2)
    vt = np.ascontiguousarray(np.transpose(v, (0, 2, 1)))
    return (dev(q, torch.bfloat16), dev(k, torch.bfloat16), dev(vt, torch.float16), pitch)


def run_both(Lq, heads, groups, n_keys, parts, seed):
    q, k, vt, pitch = case(Lq, heads, groups, n_keys, seed)
    err = torch.zeros(2, dtype=torch.int32, device="cuda")
    ref = torch.zeros(Lq, heads * 64, dtype=torch.bfloat16, device="cuda")
    ws_bytes = fdp.attention_workspace_bytes(Lq, heads, groups, n_keys, parts)
    ws = torch.empty(max(1, ws_bytes // 4), dtype=torch.float32, device="cuda")
    fdp.op_attention(q, k, vt, heads, groups, pitch, n_keys, ref, parts=parts, workspace=ws,
                     err=err[0:1])
    got = torch.zeros_like(ref)
    fdp.op_attention_static(q, k, vt, heads, groups, pitch, n_keys, got, parts=parts,
                            err=err[1:2])
    torch.cuda.synchronize()
    assert err.cpu().tolist() == [0, 0]
    return got.float().cpu(), ref.float().cpu(), ws_bytes


def test_static_workspace_attention_matches_allocated_workspace():
    torch.cuda.set_device(0)
    # two calls in a row through the shared static array, different shapes and inputs; both
    # cut tile pairs across CTAs, so the static workspace really carries partial results
    for Lq, heads, groups, n_keys, parts, seed in [(520, 4, 2, 1300, 3, 31),
                                                   (1560, 16, 4, 6240, 0, 37)]:
        got, ref, ws_bytes = run_both(Lq, heads, groups, n_keys, parts, seed)
        assert 0 < ws_bytes <= STATIC_BYTES
        assert_close_scaled(got, ref, 1.5e-2, f"static vs allocated workspace, Lq={Lq}")


def test_static_workspace_rejects_oversize_requests():
    L = fdp.lib()
    Lq, heads, groups, n_keys = 6240, 16, 4, 24960
    assert fdp.attention_workspace_bytes(Lq, heads, groups, n_keys, 300) > STATIC_BYTES
    # rejected before any launch: pointers are never touched
    assert L.fd_op_attention_static(Lq, heads, groups, 0, 0, 0, 24960, n_keys, 0, 300, 0, 0) == 1
