"""Python access to the C oracle of the ASD verifier (arXiv 2608.03447, Sec. 3.2-3.3).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's
CPU-baseline leg load this module. It shares no code with the CUDA library and
never imports it.

The arithmetic lives in ``asd_oracle.c`` (Eq. 1-14, Alg. 1); this file only
compiles it with ``gcc`` (no fused multiply-adds, no fast-math), loads it with
ctypes and converts numpy arrays. ctypes releases the GIL during each call, so
threads can run independent requests side by side.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(HERE, "asd_oracle.c")
LIBRARY = os.path.join(HERE, "liboracle.so")

DTYPE_F32 = 0
DTYPE_BF16 = 1

STATUS_DRAFT_RANGE = 1
STATUS_NAN_LOGIT = 2
STATUS_BAD_LEDGER = 4

CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-std=c11"]

_lock = threading.Lock()
_handle = None


def compile_library(source: str = SOURCE, output: str = LIBRARY) -> str:
    """Compile the oracle C source into a shared library and return its path."""
    tmp = f"{output}.{os.getpid()}.tmp"
    subprocess.run(["gcc", *CFLAGS, source, "-o", tmp, "-lm"], check=True)
    os.replace(tmp, output)
    return output


def _bind(lib: ctypes.CDLL) -> ctypes.CDLL:
    vp, i32, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.oracle_verify.restype = i32
    lib.oracle_verify.argtypes = [vp, i32, i32, i32, i32, vp, vp, f32, i32, i32,
                                  vp, vp, vp, vp, vp, vp]
    lib.oracle_select.restype = i32
    lib.oracle_select.argtypes = [i32, i32, vp, vp, vp, vp, vp, f32, i32, i32, vp, vp, vp, vp]
    lib.oracle_opportunity.restype = None
    lib.oracle_opportunity.argtypes = [vp, vp, vp, vp, i32, i32, vp, i32, vp, i32, vp, vp]
    lib.oracle_commit.restype = None
    lib.oracle_commit.argtypes = [i32, i32, vp, vp, i32, vp, vp, vp, i32, vp]
    lib.oracle_lmhead_logits.restype = None
    lib.oracle_lmhead_logits.argtypes = [vp, vp, i32, i32, vp, i32, vp, vp]
    return lib


def load_library(path: str | None = None) -> ctypes.CDLL:
    """Load (compiling first when stale or missing) the oracle library.

    With ``path`` given, load that file as is: the tests use this to load
    deliberately broken copies of the oracle and check that the pins catch them.
    """
    global _handle
    if path is not None:
        return _bind(ctypes.CDLL(path))
    with _lock:
        if _handle is None:
            stale = (not os.path.exists(LIBRARY)
                     or os.path.getmtime(LIBRARY) < os.path.getmtime(SOURCE))
            if stale:
                compile_library()
            _handle = _bind(ctypes.CDLL(LIBRARY))
    return _handle


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def bf16_bits(x) -> np.ndarray:
    """Accept a torch bf16 tensor or a uint16/int16 array; return uint16 bit patterns."""
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    except ImportError:  # pragma: no cover
        pass
    a = np.ascontiguousarray(x)
    if a.dtype == np.int16:
        a = a.view(np.uint16)
    assert a.dtype == np.uint16
    return a


def verify(logits, draft, ledger=None, gate: float = 1.0, cap: int = 2, strict: bool = False,
           dtype: int | None = None, lib: ctypes.CDLL | None = None) -> dict:
    """Run the oracle on one batch of draft blocks.

    logits: [B, K+1, V] float32 array, or bf16 (torch bf16 tensor / uint16 bits)
    draft:  [B, K] int32;  ledger: [B, 2] float32 (budget, spent) or None (strict)
    Returns numpy arrays: accepted_len, committed, recovery, row_argmax,
    row_regret, status, ledger (the updated copy).
    """
    lib = lib or load_library()
    if dtype is None:
        try:
            import torch
            is_bf16 = isinstance(logits, torch.Tensor) and logits.dtype == torch.bfloat16
            if isinstance(logits, torch.Tensor) and logits.dtype == torch.float32:
                logits = logits.detach().cpu().numpy()
        except ImportError:  # pragma: no cover
            is_bf16 = False
        if is_bf16 or (isinstance(logits, np.ndarray) and logits.dtype in (np.uint16, np.int16)):
            dtype = DTYPE_BF16
        else:
            dtype = DTYPE_F32
    if dtype == DTYPE_BF16:
        z = bf16_bits(logits)
    else:
        z = np.ascontiguousarray(logits, dtype=np.float32)
    B, K1, V = z.shape
    K = K1 - 1
    x = np.ascontiguousarray(np.asarray(draft), dtype=np.int32).reshape(B, K)
    if ledger is None:
        led = np.zeros((B, 2), np.float32)
    else:
        led = np.array(np.asarray(ledger, dtype=np.float32).reshape(B, 2), copy=True)
    out = {
        "accepted_len": np.zeros(B, np.int32),
        "committed": np.zeros((B, K1), np.int32),
        "recovery": np.zeros(B, np.int32),
        "row_argmax": np.zeros((B, K1), np.int32),
        "row_regret": np.zeros((B, K), np.float32),
        "status": np.zeros(B, np.int32),
    }
    rc = lib.oracle_verify(_ptr(z), dtype, B, K, V, _ptr(x), _ptr(led), float(gate), int(cap),
                           1 if strict else 0, _ptr(out["accepted_len"]), _ptr(out["committed"]),
                           _ptr(out["recovery"]), _ptr(out["row_argmax"]),
                           _ptr(out["row_regret"]), _ptr(out["status"]))
    if rc != 0:
        raise ValueError(f"oracle_verify rejected its arguments (B={B}, K={K}, V={V})")
    out["ledger"] = led
    return out


def select(draft, row_argmax, row_regret, row_status, ledger, gate: float, cap: int,
           strict: bool = False, lib: ctypes.CDLL | None = None) -> dict:
    """Alg. 1 alone, replayed on the row-stage results of an earlier (strict) oracle run."""
    lib = lib or load_library()
    y = np.ascontiguousarray(row_argmax, dtype=np.int32)
    B, K1 = y.shape
    K = K1 - 1
    x = np.ascontiguousarray(draft, dtype=np.int32).reshape(B, K)
    r = np.ascontiguousarray(row_regret, dtype=np.float32).reshape(B, K)
    st_in = np.ascontiguousarray(row_status, dtype=np.int32).reshape(B)
    led = np.array(np.asarray(ledger, dtype=np.float32).reshape(B, 2), copy=True)
    out = {
        "accepted_len": np.zeros(B, np.int32),
        "committed": np.zeros((B, K1), np.int32),
        "recovery": np.zeros(B, np.int32),
        "status": np.zeros(B, np.int32),
    }
    rc = lib.oracle_select(B, K, _ptr(x), _ptr(y), _ptr(r), _ptr(st_in), _ptr(led), float(gate), int(cap),
                           1 if strict else 0, _ptr(out["accepted_len"]), _ptr(out["committed"]),
                           _ptr(out["recovery"]), _ptr(out["status"]))
    if rc != 0:
        raise ValueError("oracle_select rejected its arguments")
    out["ledger"] = led
    return out


def verify_blocks(blocks, ledger, gate: float, cap: int, strict: bool = False,
                  lib: ctypes.CDLL | None = None) -> list[dict]:
    """Run sequential blocks of the same requests, carrying the ledger (Sec. 3.2, (B, s))."""
    results = []
    led = np.array(ledger, dtype=np.float32, copy=True)
    for logits, draft in blocks:
        res = verify(logits, draft, led, gate, cap, strict, lib=lib)
        led = res["ledger"]
        results.append(res)
    return results


def lmhead_logits(h, W, tokens=None, lib: ctypes.CDLL | None = None) -> tuple[np.ndarray, np.ndarray]:
    """fp64 logits z = h[tokens] W^T from bf16 inputs; returns (fp64 [T, V], fp32 [T, V])."""
    lib = lib or load_library()
    hb = bf16_bits(h)
    wb = bf16_bits(W)
    H = hb.shape[1]
    V = wb.shape[0]
    assert wb.shape[1] == H
    if tokens is None:
        tokens = np.arange(hb.shape[0], dtype=np.int32)
    tok = np.ascontiguousarray(tokens, dtype=np.int32)
    T = tok.shape[0]
    out64 = np.zeros((T, V), np.float64)
    out32 = np.zeros((T, V), np.float32)
    lib.oracle_lmhead_logits(_ptr(hb), _ptr(wb), H, V, _ptr(tok), T, _ptr(out64), _ptr(out32))
    return out64, out32


def lmhead_logits_matmul(h, W, v_block: int = 8192) -> np.ndarray:
    """fp64 logits z = h W^T of every row of h, from bf16 inputs, with numpy's float64 matmul.

    The same definition as ``lmhead_logits`` (bf16 widened exactly, products and sums in fp64), with a
    library matmul as the summation step instead of the C loop, for full-size shapes (576 x 5120 x
    151936) that the loop takes minutes over; fp64 summation order differs only far below the logits'
    fp32 rounding. W is widened one block of rows at a time. Returns [T, V] float64.
    """
    import torch
    hb = torch.from_numpy(bf16_bits(h).view(np.int16)).view(torch.bfloat16)
    wb = torch.from_numpy(bf16_bits(W).view(np.int16)).view(torch.bfloat16)
    h64 = hb.double().numpy()
    V = wb.shape[0]
    out = np.empty((h64.shape[0], V), np.float64)
    for v0 in range(0, V, v_block):
        w64 = wb[v0:v0 + v_block].double().numpy()
        np.matmul(h64, w64.T, out=out[:, v0:v0 + w64.shape[0]])
    return out


def opportunity(row_argmax, draft, row_regret, taus, ps, status=None, lib: ctypes.CDLL | None = None):
    """Eq. 4 counts: (num [len(taus), len(ps)] int64, den int) over the given blocks."""
    lib = lib or load_library()
    y = np.ascontiguousarray(row_argmax, dtype=np.int32)
    n, K1 = y.shape
    K = K1 - 1
    x = np.ascontiguousarray(draft, dtype=np.int32).reshape(n, K)
    r = np.ascontiguousarray(row_regret, dtype=np.float32).reshape(n, K)
    st = None if status is None else np.ascontiguousarray(status, dtype=np.int32).reshape(n)
    tau = np.ascontiguousarray(taus, dtype=np.float32)
    p = np.ascontiguousarray(ps, dtype=np.int32)
    num = np.zeros(len(tau) * len(p), np.int64)
    den = np.zeros(1, np.int64)
    lib.oracle_opportunity(_ptr(y), _ptr(x), _ptr(r), None if st is None else _ptr(st), n, K, _ptr(tau),
                           len(tau), _ptr(p), len(p), _ptr(num), _ptr(den))
    return num.reshape(len(tau), len(p)), int(den[0])


def commit(accepted_len, committed, pending, kv_len, tokens, token_len, lib: ctypes.CDLL | None = None) -> dict:
    """Sec. 3.3 advance along the emitted sequence; returns updated copies (kv_len, tokens, token_len, status)."""
    lib = lib or load_library()
    a = np.ascontiguousarray(accepted_len, dtype=np.int32)
    c = np.ascontiguousarray(committed, dtype=np.int32)
    B, K1 = c.shape
    kv = np.array(kv_len, dtype=np.int32, copy=True)
    tok = np.array(tokens, dtype=np.int32, copy=True)
    tl = np.array(token_len, dtype=np.int32, copy=True)
    st = np.zeros(B, np.int32)
    lib.oracle_commit(B, K1 - 1, _ptr(a), _ptr(c), int(pending), _ptr(kv), _ptr(tok), _ptr(tl), tok.shape[1], _ptr(st))
    return {"kv_len": kv, "tokens": tok, "token_len": tl, "status": st}
