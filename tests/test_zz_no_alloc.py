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
    # calls in a row through the shared static array, different shapes and inputs; both cut
    # tile pairs across CTAs, so the static workspace really carries partial results. The
    # combine order is fixed, so the two workspaces must give the same bits; the small case
    # runs again after the large one, so counters or partials a larger call left behind would
    # show.
    cases = [(520, 4, 2, 1300, 3, 31), (1560, 16, 4, 6240, 0, 37), (520, 4, 2, 1300, 3, 31)]
    for Lq, heads, groups, n_keys, parts, seed in cases:
        got, ref, ws_bytes = run_both(Lq, heads, groups, n_keys, parts, seed)
        assert 0 < ws_bytes <= STATIC_BYTES
        assert torch.equal(got, ref), f"static vs allocated workspace differ, Lq={Lq}"
        assert_close_scaled(got, ref, 0.0, f"static vs allocated workspace, Lq={Lq}")


def test_static_workspace_call_allocates_no_device_memory():
    """After a first call (which may be where the library's module is loaded), further calls
    change the device's free memory by nothing."""
    torch.cuda.set_device(0)
    Lq, heads, groups, n_keys, parts = 1560, 16, 4, 6240, 0
    q, k, vt, pitch = case(Lq, heads, groups, n_keys, 41)
    out = torch.zeros(Lq, heads * 64, dtype=torch.bfloat16, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    fdp.op_attention_static(q, k, vt, heads, groups, pitch, n_keys, out, parts=parts, err=err)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        fdp.op_attention_static(q, k, vt, heads, groups, pitch, n_keys, out, parts=parts,
                                err=err)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert int(err.item()) == 0


def test_static_workspace_rejects_oversize_requests():
    """A request needing more than the static array is refused by the size check alone (real
    buffers and a real error word are passed, so no other check can be what refuses it), and
    the same shape with parts = 1 (no workspace) is accepted."""
    L = fdp.lib()
    Lq, heads, groups, n_keys = 6240, 16, 4, 24960
    assert fdp.attention_workspace_bytes(Lq, heads, groups, n_keys, 300) > STATIC_BYTES
    q, k, vt, pitch = case(Lq, heads, groups, n_keys, 43)
    out = torch.zeros(Lq, heads * 64, dtype=torch.bfloat16, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    args = (Lq, heads, groups, q.data_ptr(), k.data_ptr(), vt.data_ptr(), pitch, n_keys,
            out.data_ptr())
    assert L.fd_op_attention_static(*args, 300, err.data_ptr(), None) == 1
    torch.cuda.synchronize()
    assert not bool(out.float().abs().sum())   # refused before any launch
    assert L.fd_op_attention_static(*args, 1, err.data_ptr(), None) == 0
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and bool(out.float().abs().sum())
