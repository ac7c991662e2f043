"""ctypes binding of libasd (include/asd.h): argument marshalling only.

Every step of the verifier runs in the library's CUDA kernels; this module
turns torch tensors into device pointers, passes torch's current CUDA stream,
and raises on a non-zero return code. There is no fallback: if libasd.so is
missing the first call raises.

Entry points mirror the C names: ``verify`` (asd_verify), ``verify_strict``
(asd_verify_strict), ``workspace_size``, ``workspace_init``, ``status_string``.
Ledgers are float32 tensors of shape [B, 2] holding (budget, spent), the
memory layout of ``asd_ledger``.
"""
from __future__ import annotations

import ctypes
import os
import re
import threading

import torch

PKG = os.path.dirname(os.path.abspath(__file__))
LIBRARY = os.path.join(PKG, "libasd.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "asd.h")

F32 = 0
BF16 = 1

OK = 0
STATUS_DRAFT_RANGE = 1
STATUS_NAN_LOGIT = 2
STATUS_BAD_LEDGER = 4
STATUS_OVERFLOW = 8
STATUS_INCOMPLETE = 16
MAX_K = 31
RESIDENT_INPUTS = 0x100  # ASD_RESIDENT_INPUTS, ORed into the dtype code
INT32_MAX = 2**31 - 1

_lock = threading.Lock()
_lib = None


class AsdError(RuntimeError):
    def __init__(self, fn: str, code: int):
        self.code = code
        super().__init__(f"{fn} returned {code}: {status_string(code) if _lib else code}")


def _declare(lib: ctypes.CDLL) -> ctypes.CDLL:
    vp, i32, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    lib.asd_workspace_size.argtypes = [i32, i32, i32, i32, ctypes.POINTER(sz)]
    lib.asd_workspace_size.restype = i32
    lib.asd_workspace_init.argtypes = [vp, sz, vp]
    lib.asd_workspace_init.restype = i32
    lib.asd_workspace_error.argtypes = [vp, ctypes.POINTER(i32), vp]
    lib.asd_workspace_error.restype = i32
    lib.asd_selftest_wait_timeout.argtypes = [vp, sz, vp]
    lib.asd_selftest_wait_timeout.restype = i32
    lib.asd_verify.argtypes = [vp, i32, i32, i32, i32, vp, vp, f32, i32, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.asd_verify.restype = i32
    lib.asd_verify_strict.argtypes = [vp, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.asd_verify_strict.restype = i32
    lib.asd_status_string.argtypes = [i32]
    lib.asd_status_string.restype = ctypes.c_char_p
    lib.asd_host_alias.argtypes = [vp, ctypes.POINTER(vp)]
    lib.asd_host_alias.restype = i32
    lib.asd_verify_launches.argtypes = [i32, i32, i32, i32, ctypes.POINTER(i32)]
    lib.asd_verify_launches.restype = i32
    lib.asd_blocks_workspace_size.argtypes = [i32, i32, i32, i32, i32, ctypes.POINTER(sz)]
    lib.asd_blocks_workspace_size.restype = i32
    lib.asd_verify_blocks.argtypes = [vp, i32, i32, i32, i32, i32, vp, vp, f32, i32, vp, vp, vp, vp, vp, vp, vp, sz,
                                      vp]
    lib.asd_verify_blocks.restype = i32
    lib.asd_shard_partials.argtypes = [vp, i32, i32, i32, i32, i32, i32, vp, vp, vp, sz, vp]
    lib.asd_shard_partials.restype = i32
    lib.asd_shard_combine.argtypes = [vp, i32, i32, i32, i32, vp, vp, f32, i32, vp, vp, vp, vp, vp, vp, vp]
    lib.asd_shard_combine.restype = i32
    lib.asd_commit.argtypes = [i32, i32, vp, vp, i32, vp, vp, vp, i32, vp, vp]
    lib.asd_commit.restype = i32
    lib.asd_opportunity.argtypes = [vp, vp, vp, vp, i32, i32, vp, i32, vp, i32, vp, vp]
    lib.asd_opportunity.restype = i32
    if hasattr(lib, "asd_verify_noalloc"):
        lib.asd_verify_noalloc.argtypes = [vp, i32, i32, i32, i32, vp, vp, f32, i32, vp, vp, vp, vp, vp, vp, vp]
        lib.asd_verify_noalloc.restype = i32
    lib.asd_lmhead_workspace_size.argtypes = [i32, i32, i32, i32, ctypes.POINTER(sz)]
    lib.asd_lmhead_workspace_size.restype = i32
    lib.asd_lmhead_verify.argtypes = [vp, vp, i32, i32, i32, i32, vp, vp, f32, i32,
                                      vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.asd_lmhead_verify.restype = i32
    lib.asd_lmhead_logits.argtypes = [vp, vp, i32, i32, i32, vp, vp]
    lib.asd_lmhead_logits.restype = i32
    lib.asd_lmhead_partials.argtypes = [vp, vp, i32, i32, i32, i32, i32, i32, vp, vp, vp, sz, vp]
    lib.asd_lmhead_partials.restype = i32
    lib.asd_set_launch_options.argtypes = [vp]
    lib.asd_set_launch_options.restype = i32
    lib.asd_get_launch_options.argtypes = [vp]
    lib.asd_get_launch_options.restype = i32
    return lib


class _LaunchOptions(ctypes.Structure):
    _fields_ = [("path", ctypes.c_int), ("fused_select", ctypes.c_int), ("no_pdl", ctypes.c_int)]


PATHS = {"auto": 0, "small": 1, "stream": 2, "tma": 3}


def set_launch_options(path: str = "auto", fused_select: bool = False, pdl: bool = True) -> None:
    """asd_set_launch_options: which row-stage kernel the verify calls use (process-wide)."""
    opt = _LaunchOptions(PATHS[path], int(fused_select), int(not pdl))
    _check("asd_set_launch_options", load().asd_set_launch_options(ctypes.byref(opt)))


def get_launch_options() -> dict:
    opt = _LaunchOptions()
    _check("asd_get_launch_options", load().asd_get_launch_options(ctypes.byref(opt)))
    names = {v: k for k, v in PATHS.items()}
    return {"path": names[opt.path], "fused_select": bool(opt.fused_select), "pdl": not opt.no_pdl}


def reset_launch_options() -> None:
    _check("asd_set_launch_options", load().asd_set_launch_options(None))


def load(path: str = LIBRARY) -> ctypes.CDLL:
    """Open libasd.so (once). Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build() "
                                   "(python -m paper_2608_03447_gb300.build)")
            _lib = _declare(ctypes.CDLL(path))
    return _lib


def declared_functions(header: str = HEADER) -> list[str]:
    """Names of the functions that include/asd.h declares."""
    with open(header) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(asd_[a-z0-9_]+)\s*\(", text)))


def status_string(code: int) -> str:
    return load().asd_status_string(int(code)).decode()


def _check(fn: str, rc: int) -> None:
    if rc != OK:
        raise AsdError(fn, rc)


def _ptr(t: torch.Tensor | None) -> int | None:
    if t is None:
        return None
    return t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _flag(resident: bool) -> int:
    return RESIDENT_INPUTS if resident else 0


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"logits must be float32 or bfloat16, got {t.dtype}")


def host_alias(t: torch.Tensor) -> int:
    """asd_host_alias: device address of a pinned host tensor's data (for reading it from kernels)."""
    if t.is_cuda or not t.is_pinned():
        raise ValueError("host_alias needs a pinned host tensor")
    out = ctypes.c_void_p(0)
    _check("asd_host_alias", load().asd_host_alias(t.data_ptr(), ctypes.byref(out)))
    return out.value


def verify_launches(B: int, K: int, V: int, dtype: int) -> int:
    """asd_verify_launches: kernels one asd_verify call launches for this shape."""
    n = ctypes.c_int(0)
    _check("asd_verify_launches", load().asd_verify_launches(B, K, V, dtype, ctypes.byref(n)))
    return n.value


def workspace_size(B: int, K: int, V: int, dtype: int) -> int:
    n = ctypes.c_size_t(0)
    _check("asd_workspace_size", load().asd_workspace_size(B, K, V, dtype, ctypes.byref(n)))
    return n.value


class Workspace:
    """Device scratch for one stream of verify calls; zeroed once at creation."""

    def __init__(self, B: int, K: int, V: int, dtype: int, device=None, stream=None):
        self.nbytes = workspace_size(B, K, V, dtype)
        self.buffer = torch.empty(self.nbytes, dtype=torch.uint8, device=device or "cuda")
        _check("asd_workspace_init", load().asd_workspace_init(self.buffer.data_ptr(), self.nbytes, _stream(stream)))

    @property
    def ptr(self) -> int:
        return self.buffer.data_ptr()

    def error(self, stream=None) -> int:
        """The sticky error word (asd_workspace_error); synchronises the stream."""
        word = ctypes.c_int(0)
        _check("asd_workspace_error", load().asd_workspace_error(self.ptr, ctypes.byref(word), _stream(stream)))
        return word.value

    def reset(self, stream=None) -> None:
        """Zero the workspace again (asd_workspace_init), e.g. after a non-zero error word."""
        _check("asd_workspace_init", load().asd_workspace_init(self.ptr, self.nbytes, _stream(stream)))


def selftest_wait_timeout(workspace: "Workspace", stream=None) -> None:
    """asd_selftest_wait_timeout: a bounded wait on a barrier nothing signals (about one second); the
    workspace's error word then reads ASD_ERR_TIMEOUT."""
    _check("asd_selftest_wait_timeout", load().asd_selftest_wait_timeout(workspace.ptr, workspace.nbytes,
                                                                         _stream(stream)))


def make_ledger(B: int, budget: float, spent: float = 0.0, device="cuda") -> torch.Tensor:
    led = torch.empty(B, 2, dtype=torch.float32, device=device)
    led[:, 0] = budget
    led[:, 1] = spent
    return led


def alloc_outputs(B: int, K: int, device="cuda", with_rows: bool = True) -> dict:
    out = {
        "accepted_len": torch.empty(B, dtype=torch.int32, device=device),
        "committed": torch.empty(B, K + 1, dtype=torch.int32, device=device),
        "recovery": torch.empty(B, dtype=torch.int32, device=device),
        "status": torch.empty(B, dtype=torch.int32, device=device),
    }
    if with_rows:
        out["row_argmax"] = torch.empty(B, K + 1, dtype=torch.int32, device=device)
        out["row_regret"] = torch.empty(B, K, dtype=torch.float32, device=device)
    return out


def _shape(logits: torch.Tensor, draft: torch.Tensor):
    if logits.dim() != 3 or not logits.is_cuda or not logits.is_contiguous():
        raise ValueError("logits must be a contiguous CUDA tensor [B, K+1, V]")
    B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (B, K) or draft.dtype != torch.int32 or not draft.is_contiguous():
        raise ValueError("draft must be a contiguous int32 tensor [B, K]")
    return B, K, V


def verify(logits: torch.Tensor, draft: torch.Tensor, ledger: torch.Tensor, gate: float, cap: int,
           workspace: Workspace | None = None, out: dict | None = None, stream=None, resident: bool = False) -> dict:
    """asd_verify: ASD verification of a batch of draft blocks; updates ``ledger`` in place.

    ``resident=True`` passes ASD_RESIDENT_INPUTS: no kernel still running or queued ahead on the stream
    writes ``logits`` or ``draft``, so the row stage may stream them while the previous kernel finishes.
    """
    B, K, V = _shape(logits, draft)
    if ledger.shape != (B, 2) or ledger.dtype != torch.float32 or not ledger.is_contiguous():
        raise ValueError("ledger must be a contiguous float32 tensor [B, 2] of (budget, spent)")
    code = _dtype_code(logits)
    ws = workspace or Workspace(B, K, V, code, logits.device, stream)
    o = out or alloc_outputs(B, K, logits.device)
    rc = load().asd_verify(_ptr(logits), code | _flag(resident), B, K, V, _ptr(draft), _ptr(ledger), float(gate),
                           int(cap),
                           _ptr(o["accepted_len"]), _ptr(o["committed"]), _ptr(o["recovery"]),
                           _ptr(o.get("row_argmax")), _ptr(o.get("row_regret")), _ptr(o.get("status")),
                           ws.ptr, ws.nbytes, _stream(stream))
    _check("asd_verify", rc)
    return o


def verify_noalloc(logits: torch.Tensor, draft: torch.Tensor, ledger: torch.Tensor, gate: float, cap: int,
                   out: dict | None = None, stream=None, resident: bool = False) -> dict:
    """asd_verify_noalloc: asd_verify with the library's fixed scratch instead of a workspace.

    For callers that may not allocate device memory while verifying. Calls that
    may overlap on the GPU share that scratch and must be ordered on one stream.
    """
    B, K, V = _shape(logits, draft)
    if ledger.shape != (B, 2) or ledger.dtype != torch.float32 or not ledger.is_contiguous():
        raise ValueError("ledger must be a contiguous float32 tensor [B, 2] of (budget, spent)")
    o = out or alloc_outputs(B, K, logits.device)
    rc = load().asd_verify_noalloc(_ptr(logits), _dtype_code(logits) | _flag(resident), B, K, V, _ptr(draft),
                                   _ptr(ledger),
                                   float(gate), int(cap), _ptr(o["accepted_len"]), _ptr(o["committed"]),
                                   _ptr(o["recovery"]), _ptr(o.get("row_argmax")), _ptr(o.get("row_regret")),
                                   _ptr(o.get("status")), _stream(stream))
    _check("asd_verify_noalloc", rc)
    return o


def verify_strict(logits: torch.Tensor, draft: torch.Tensor, workspace: Workspace | None = None,
                  out: dict | None = None, stream=None, resident: bool = False) -> dict:
    """asd_verify_strict: strict greedy verification (Eq. 2)."""
    B, K, V = _shape(logits, draft)
    code = _dtype_code(logits)
    ws = workspace or Workspace(B, K, V, code, logits.device, stream)
    o = out or alloc_outputs(B, K, logits.device)
    rc = load().asd_verify_strict(_ptr(logits), code | _flag(resident), B, K, V, _ptr(draft),
                                  _ptr(o["accepted_len"]), _ptr(o["committed"]), _ptr(o["recovery"]),
                                  _ptr(o.get("row_argmax")), _ptr(o.get("row_regret")), _ptr(o.get("status")),
                                  ws.ptr, ws.nbytes, _stream(stream))
    _check("asd_verify_strict", rc)
    return o


_aliases: dict = {}
_ALIAS_CACHE = 64  # the most recently used pinned buffers keep their looked-up device address


def _alias(t: torch.Tensor) -> int:
    key = (t.data_ptr(), t.numel() * t.element_size())
    addr = _aliases.pop(key, None)
    if addr is None:
        addr = host_alias(t)
    _aliases[key] = addr  # re-inserted: dicts keep insertion order, so the oldest entry is first
    while len(_aliases) > _ALIAS_CACHE:
        _aliases.pop(next(iter(_aliases)))
    return addr


def verify_from_host(logits_host: torch.Tensor, draft_host: torch.Tensor, ledger: torch.Tensor, gate: float,
                     cap: int, workspace: Workspace, out: dict, host_out: dict, stream=None,
                     resident: bool = False) -> dict:
    """End-to-end step from pinned host buffers: verify reading them in place, copy the results out.

    The kernels read the pinned logits and drafts through their device aliases
    (asd_host_alias), so the host-to-device transfer is the verify's own
    stream of reads over the host link, with no separate copy; the ledger stays
    on the device (the request state carried between rounds); the per-request
    results are copied back to pinned host tensors, asynchronously on ``stream``.
    """
    if logits_host.dim() != 3 or not logits_host.is_pinned() or not draft_host.is_pinned():
        raise ValueError("verify_from_host needs pinned host logits [B, K+1, V] and drafts [B, K]")
    B, K1, V = logits_host.shape
    K = K1 - 1
    code = _dtype_code(logits_host)
    rc = load().asd_verify(_alias(logits_host), code | _flag(resident), B, K, V, _alias(draft_host), _ptr(ledger),
                           float(gate),
                           int(cap), _ptr(out["accepted_len"]), _ptr(out["committed"]), _ptr(out["recovery"]),
                           _ptr(out.get("row_argmax")), _ptr(out.get("row_regret")), _ptr(out.get("status")),
                           workspace.ptr, workspace.nbytes, _stream(stream))
    _check("asd_verify", rc)
    for k in ("accepted_len", "committed", "recovery"):
        host_out[k].copy_(out[k], non_blocking=True)
    return host_out


def lmhead_workspace(B: int, K: int, V: int, H: int, device=None, stream=None) -> Workspace:
    n = ctypes.c_size_t(0)
    _check("asd_lmhead_workspace_size", load().asd_lmhead_workspace_size(B, K, V, H, ctypes.byref(n)))
    ws = Workspace.__new__(Workspace)
    ws.nbytes = n.value
    ws.buffer = torch.empty(ws.nbytes, dtype=torch.uint8, device=device or "cuda")
    _check("asd_workspace_init", load().asd_workspace_init(ws.buffer.data_ptr(), ws.nbytes, _stream(stream)))
    return ws


def _lm_shapes(hidden: torch.Tensor, weight: torch.Tensor):
    for name, t in (("hidden", hidden), ("weight", weight)):
        if t.dtype != torch.bfloat16 or t.dim() != 2 or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous 2-D bf16 CUDA tensor")
    if hidden.shape[1] != weight.shape[1]:
        raise ValueError("hidden and weight must share the hidden size H")
    return hidden.shape[0], weight.shape[0], hidden.shape[1]


def lmhead_verify(hidden: torch.Tensor, weight: torch.Tensor, draft: torch.Tensor, ledger: torch.Tensor,
                  gate: float, cap: int, workspace: Workspace | None = None, out: dict | None = None,
                  stream=None) -> dict:
    """asd_lmhead_verify: logits = hidden @ weight.T on the tensor cores, reduced on chip, then Alg. 1."""
    T, V, H = _lm_shapes(hidden, weight)
    B, K = draft.shape
    if T != B * (K + 1):
        raise ValueError("hidden must hold B*(K+1) rows")
    ws = workspace or lmhead_workspace(B, K, V, H, hidden.device, stream)
    o = out or alloc_outputs(B, K, hidden.device)
    if "row_top" not in o:
        o["row_top"] = torch.empty(B, K + 1, dtype=torch.float32, device=hidden.device)
    rc = load().asd_lmhead_verify(_ptr(hidden), _ptr(weight), H, B, K, V, _ptr(draft), _ptr(ledger), float(gate),
                                  int(cap), _ptr(o["accepted_len"]), _ptr(o["committed"]), _ptr(o["recovery"]),
                                  _ptr(o.get("row_argmax")), _ptr(o.get("row_regret")), _ptr(o.get("row_top")),
                                  _ptr(o.get("status")), ws.ptr, ws.nbytes, _stream(stream))
    _check("asd_lmhead_verify", rc)
    return o


def lmhead_partials(hidden: torch.Tensor, weight_shard: torch.Tensor, draft: torch.Tensor, v_offset: int, V: int,
                    workspace: Workspace | None = None, out: torch.Tensor | None = None,
                    stream=None) -> torch.Tensor:
    """asd_lmhead_partials: one vocabulary shard of the fused LM-head verify, as int32 [B*(K+1), 6] partials.

    weight_shard [Vs, H] holds rows v_offset .. v_offset+Vs-1 of the LM-head weight; draft holds global ids.
    """
    T, Vs, H = _lm_shapes(hidden, weight_shard)
    B, K = draft.shape
    if T != B * (K + 1):
        raise ValueError("hidden must hold B*(K+1) rows")
    ws = workspace or lmhead_workspace(B, K, Vs, H, hidden.device, stream)
    o = out if out is not None else torch.empty(T, PARTIAL_WORDS, dtype=torch.int32, device=hidden.device)
    _check("asd_lmhead_partials", load().asd_lmhead_partials(_ptr(hidden), _ptr(weight_shard), H, B, K, Vs,
                                                             int(v_offset), int(V), _ptr(draft), _ptr(o), ws.ptr,
                                                             ws.nbytes, _stream(stream)))
    return o


def lmhead_logits(hidden: torch.Tensor, weight: torch.Tensor, out: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    """asd_lmhead_logits: the same tensor-core GEMM, writing the fp32 logits [T, V]."""
    T, V, H = _lm_shapes(hidden, weight)
    o = out if out is not None else torch.empty(T, V, dtype=torch.float32, device=hidden.device)
    _check("asd_lmhead_logits", load().asd_lmhead_logits(_ptr(hidden), _ptr(weight), H, T, V, _ptr(o),
                                                         _stream(stream)))
    return o


def blocks_workspace(nblk: int, B: int, K: int, V: int, dtype: int, device=None, stream=None) -> Workspace:
    n = ctypes.c_size_t(0)
    _check("asd_blocks_workspace_size", load().asd_blocks_workspace_size(nblk, B, K, V, dtype, ctypes.byref(n)))
    ws = Workspace.__new__(Workspace)
    ws.nbytes = n.value
    ws.buffer = torch.empty(max(ws.nbytes, 1), dtype=torch.uint8, device=device or "cuda")
    _check("asd_workspace_init", load().asd_workspace_init(ws.buffer.data_ptr(), ws.nbytes, _stream(stream)))
    return ws


def verify_blocks(logits: torch.Tensor, draft: torch.Tensor, ledger: torch.Tensor, gate: float, cap: int,
                  workspace: Workspace | None = None, out: dict | None = None, stream=None,
                  resident: bool = False) -> dict:
    """asd_verify_blocks: nblk sequential blocks of the same requests in one call.

    logits [nblk, B, K+1, V], draft [nblk, B, K], ledger [B, 2]; outputs carry a
    leading nblk dimension.
    """
    if logits.dim() != 4 or not logits.is_cuda or not logits.is_contiguous():
        raise ValueError("logits must be a contiguous CUDA tensor [nblk, B, K+1, V]")
    nblk, B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (nblk, B, K) or draft.dtype != torch.int32 or not draft.is_contiguous():
        raise ValueError("draft must be a contiguous int32 tensor [nblk, B, K]")
    if ledger.shape != (B, 2) or ledger.dtype != torch.float32 or not ledger.is_contiguous():
        raise ValueError("ledger must be a contiguous float32 tensor [B, 2] of (budget, spent)")
    code = _dtype_code(logits)
    ws = workspace or blocks_workspace(nblk, B, K, V, code, logits.device, stream)
    if out is None:
        flat = alloc_outputs(nblk * B, K, logits.device)
        out = {k: v.view(nblk, B, *v.shape[1:]) for k, v in flat.items()}
    rc = load().asd_verify_blocks(_ptr(logits), code | _flag(resident), nblk, B, K, V, _ptr(draft), _ptr(ledger),
                                  float(gate),
                                  int(cap), _ptr(out["accepted_len"]), _ptr(out["committed"]), _ptr(out["recovery"]),
                                  _ptr(out.get("row_argmax")), _ptr(out.get("row_regret")), _ptr(out.get("status")),
                                  ws.ptr, ws.nbytes, _stream(stream))
    _check("asd_verify_blocks", rc)
    return out


def opportunity(row_argmax: torch.Tensor, draft: torch.Tensor, row_regret: torch.Tensor, taus, ps,
                status: torch.Tensor | None = None, counts: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """asd_opportunity: Eq. 4 counts over the block-requests' row outputs (accumulated into ``counts``).

    Returns the int64 counts tensor [len(taus) * len(ps) + 1] (the last entry is |M|).
    """
    import numpy as _np
    n, K1 = row_argmax.shape[0], row_argmax.shape[-1]
    tau = _np.ascontiguousarray(taus, dtype=_np.float32)
    pv = _np.ascontiguousarray(ps, dtype=_np.int32)
    if counts is None:
        counts = torch.zeros(len(tau) * len(pv) + 1, dtype=torch.int64, device=row_argmax.device)
    rc = load().asd_opportunity(_ptr(row_argmax), _ptr(draft), _ptr(row_regret), _ptr(status), n, K1 - 1,
                                tau.ctypes.data, len(tau), pv.ctypes.data, len(pv), _ptr(counts), _stream(stream))
    _check("asd_opportunity", rc)
    return counts


PARTIAL_WORDS = 6  # asd_partial: uint64 key, float top, float draft_logit, uint32 flags, uint32 reserved


def shard_partials(logits: torch.Tensor, draft: torch.Tensor, v_offset: int, V: int,
                   workspace: Workspace | None = None, out: torch.Tensor | None = None, stream=None,
                   resident: bool = False) -> torch.Tensor:
    """asd_shard_partials: one vocabulary shard's per-row partials, as int32 [B*(K+1), 6] (asd_partial).

    logits [B, K+1, Vs] hold vocabulary entries v_offset .. v_offset+Vs-1 of V; draft holds global ids.
    """
    B, K, Vs = _shape(logits, draft)
    code = _dtype_code(logits)
    ws = workspace or Workspace(B, K, Vs, code, logits.device, stream)
    o = out if out is not None else torch.empty(B * (K + 1), PARTIAL_WORDS, dtype=torch.int32, device=logits.device)
    rc = load().asd_shard_partials(_ptr(logits), code | _flag(resident), B, K, Vs, int(v_offset), int(V), _ptr(draft),
                                   _ptr(o),
                                   ws.ptr, ws.nbytes, _stream(stream))
    _check("asd_shard_partials", rc)
    return o


def shard_combine(partials: torch.Tensor, draft: torch.Tensor, ledger: torch.Tensor, gate: float, cap: int, V: int,
                  out: dict | None = None, stream=None) -> dict:
    """asd_shard_combine: partials [S, B*(K+1), 6] of all shards -> the outputs of asd_verify."""
    S, R, words = partials.shape
    B, K = draft.shape
    if words != PARTIAL_WORDS or R != B * (K + 1) or partials.dtype != torch.int32 or not partials.is_contiguous():
        raise ValueError("partials must be a contiguous int32 tensor [S, B*(K+1), 6]")
    o = out or alloc_outputs(B, K, partials.device)
    rc = load().asd_shard_combine(_ptr(partials), S, B, K, int(V), _ptr(draft), _ptr(ledger), float(gate), int(cap),
                                  _ptr(o["accepted_len"]), _ptr(o["committed"]), _ptr(o["recovery"]),
                                  _ptr(o.get("row_argmax")), _ptr(o.get("row_regret")), _ptr(o.get("status")),
                                  _stream(stream))
    _check("asd_shard_combine", rc)
    return o


def allgather_partials(part: torch.Tensor, group=None) -> torch.Tensor:
    """The exchange step of tensor-parallel verification: every rank's [B*(K+1), 6] partials -> [S, ...]."""
    import torch.distributed as dist
    world = dist.get_world_size(group)
    parts = [torch.empty_like(part) for _ in range(world)]
    dist.all_gather(parts, part.contiguous(), group=group)
    return torch.stack(parts).contiguous()


def commit(accepted_len: torch.Tensor, committed: torch.Tensor, pending: int = 1, kv_len: torch.Tensor | None = None,
           tokens: torch.Tensor | None = None, token_len: torch.Tensor | None = None,
           status: torch.Tensor | None = None, stream=None) -> None:
    """asd_commit: append the emitted tokens to the history and advance the KV length (in place)."""
    B, K1 = committed.shape
    max_tokens = tokens.shape[1] if tokens is not None else 0
    rc = load().asd_commit(B, K1 - 1, _ptr(accepted_len), _ptr(committed), int(pending), _ptr(kv_len), _ptr(tokens),
                           _ptr(token_len), max_tokens, _ptr(status), _stream(stream))
    _check("asd_commit", rc)
