"""asd_verify_noalloc against asd_verify, through the C ABI.

asd_verify_noalloc serves callers that may not allocate device memory while
they verify (a serving loop with a fixed device-memory budget, a plug-in whose
host framework owns every device allocation, a latency-bound path where
cudaMalloc or cudaFree could synchronise the device): it keeps its scratch in a
fixed array inside the library instead of a caller workspace. Its results must
equal asd_verify's bit for bit, call after call (the ledger carries over and
the shared scratch is reused). This file sorts last so that a failure here
leaves the other tests' results in place; it also passes on its own in a fresh
process (the first call sets the scratch up).
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu
SCRATCH_LIMIT = 10  # ASD_ERR_SCRATCH_LIMIT


def _noalloc_fn(lib):
    fn = lib.asd_verify_noalloc
    vp, i32, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    fn.argtypes = [vp, i32, i32, i32, i32, vp, vp, f32, i32, vp, vp, vp, vp, vp, vp, vp]
    fn.restype = i32
    return fn


def _call_noalloc(asd, logits, draft, ledger, gate, cap, out):
    fn = _noalloc_fn(asd.load())
    B, K1, V = logits.shape
    code = asd.BF16 if logits.dtype == torch.bfloat16 else asd.F32
    return fn(logits.data_ptr(), code, B, K1 - 1, V, draft.data_ptr(), ledger.data_ptr(), gate, cap,
              out["accepted_len"].data_ptr(), out["committed"].data_ptr(), out["recovery"].data_ptr(),
              out["row_argmax"].data_ptr(), out["row_regret"].data_ptr(), out["status"].data_ptr(),
              torch.cuda.current_stream().cuda_stream)


@pytest.mark.parametrize("shape", [(32, 8, 151936, torch.bfloat16), (4, 8, 1024, torch.float32),
                                   (256, 4, 129280, torch.float32)])
def test_noalloc_equals_verify_on_two_calls_in_a_row(asd, shape):
    B, K, V, dtype = shape
    led_noalloc = asd.make_ledger(B, 4.0)
    led_verify = asd.make_ledger(B, 4.0)
    ws = asd.Workspace(B, K, V, asd.BF16 if dtype == torch.bfloat16 else asd.F32)
    for call in range(2):
        blk = inputs.gen_block(B, K, V, dtype, 90_000 + call + V, "cuda")
        out_n = asd.alloc_outputs(B, K)
        rc = _call_noalloc(asd, blk.logits, blk.draft, led_noalloc, 1.0, 2, out_n)
        assert rc == 0, asd.status_string(rc)
        out_v = asd.verify(blk.logits, blk.draft, led_verify, 1.0, 2, workspace=ws)
        torch.cuda.synchronize()
        for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
            assert torch.equal(out_n[key], out_v[key]), f"call {call}: {key}"
        assert np.array_equal(out_n["row_regret"].cpu().numpy().view(np.uint32),
                              out_v["row_regret"].cpu().numpy().view(np.uint32)), f"call {call}: row_regret"
        assert np.array_equal(led_noalloc.cpu().numpy().view(np.uint32),
                              led_verify.cpu().numpy().view(np.uint32)), f"call {call}: ledger"


def test_noalloc_rejects_problems_beyond_its_scratch(asd):
    limit = 1 << 20
    B, K, V = 60000, 31, 1
    assert asd.workspace_size(B, K, V, asd.F32) > limit
    logits = torch.zeros(1, dtype=torch.float32, device="cuda")
    draft = torch.zeros(1, dtype=torch.int32, device="cuda")
    led = torch.zeros(2, dtype=torch.float32, device="cuda")
    out = {k: torch.full((1,), -7, dtype=torch.int32, device="cuda")
           for k in ("accepted_len", "committed", "recovery", "row_argmax", "status")}
    out["row_regret"] = torch.zeros(1, device="cuda")
    fn = _noalloc_fn(asd.load())
    rc = fn(logits.data_ptr(), asd.F32, B, K, V, draft.data_ptr(), led.data_ptr(), 1.0, 2,
            out["accepted_len"].data_ptr(), out["committed"].data_ptr(), out["recovery"].data_ptr(),
            out["row_argmax"].data_ptr(), out["row_regret"].data_ptr(), out["status"].data_ptr(),
            torch.cuda.current_stream().cuda_stream)
    assert rc == SCRATCH_LIMIT
    torch.cuda.synchronize()
    assert int(out["accepted_len"][0]) == -7  # nothing was launched


def _same(out_n, out_v, led_n, led_v, what):
    for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
        assert torch.equal(out_n[key], out_v[key]), f"{what}: {key}"
    assert np.array_equal(out_n["row_regret"].cpu().numpy().view(np.uint32),
                          out_v["row_regret"].cpu().numpy().view(np.uint32)), f"{what}: row_regret"
    assert np.array_equal(led_n.cpu().numpy().view(np.uint32), led_v.cpu().numpy().view(np.uint32)), f"{what}: ledger"


def test_noalloc_binding_with_resident_inputs(asd):
    """The Python binding (asd.verify_noalloc) with ASD_RESIDENT_INPUTS, against asd.verify with the same
    flag, on two calls in a row of the Qwen3-14B-shaped step."""
    B, K, V = 32, 8, 151936
    led_n, led_v = asd.make_ledger(B, 4.0), asd.make_ledger(B, 4.0)
    ws = asd.Workspace(B, K, V, asd.BF16)
    for call in range(2):
        blk = inputs.gen_block(B, K, V, torch.bfloat16, 91_000 + call, "cuda")
        out_n = asd.verify_noalloc(blk.logits, blk.draft, led_n, 1.0, 2, resident=True)
        out_v = asd.verify(blk.logits, blk.draft, led_v, 1.0, 2, workspace=ws, resident=True)
        torch.cuda.synchronize()
        _same(out_n, out_v, led_n, led_v, f"call {call}")


def test_noalloc_at_its_scratch_limit(asd):
    """The largest batch whose workspace fits ASD_NOALLOC_SCRATCH_BYTES (K=7) runs and matches asd_verify
    on two calls in a row; the first batch beyond it is rejected before anything is launched."""
    limit = 1 << 20
    K, V = 7, 64
    B = 1
    while asd.workspace_size(B + 1, K, V, asd.F32) <= limit:  # the largest batch that fits
        B += 1
    B_over = B + 1
    assert asd.workspace_size(B, K, V, asd.F32) <= limit < asd.workspace_size(B_over, K, V, asd.F32)
    led_n, led_v = asd.make_ledger(B, 4.0), asd.make_ledger(B, 4.0)
    ws = asd.Workspace(B, K, V, asd.F32)
    for call in range(2):
        blk = inputs.gen_block(B, K, V, torch.float32, 92_000 + call, "cuda")
        out_n = asd.verify_noalloc(blk.logits, blk.draft, led_n, 1.0, 2)
        out_v = asd.verify(blk.logits, blk.draft, led_v, 1.0, 2, workspace=ws)
        torch.cuda.synchronize()
        _same(out_n, out_v, led_n, led_v, f"call {call}")
    blk = inputs.gen_block(B_over, K, V, torch.float32, 92_100, "cuda")
    with pytest.raises(asd.AsdError) as err:
        asd.verify_noalloc(blk.logits, blk.draft, asd.make_ledger(B_over, 4.0), 1.0, 2)
    assert err.value.code == SCRATCH_LIMIT
