"""Python binding of libhdl, the GB300 kernels for HDL (arXiv 2609.36864).

Each function has the name of the C entry point it calls (include/hdl.h) and
only marshals arguments: it checks devices, dtypes and contiguity, fills in
the current CUDA stream, optionally allocates output tensors with torch, and
passes raw pointers.  Every step of the computation runs in the library's
CUDA kernels; there is no CPU fallback.  Importing this package does not load
the library; the first call does, and fails loudly if libhdl.so is missing.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

__all__ = [
    "HdlError", "lib", "library_path", "HDL_OK", "HDL_BF16", "HDL_F32",
    "hdl_abi_version", "hdl_status_string", "hdl_rescore_workspace_bytes",
    "hdl_rescore", "hdl_device_status", "hdl_select_branches",
    "hdl_assign_continuations", "hdl_suffix_mask", "hdl_rescore_noalloc",
    "HDL_STATIC_SCRATCH_BYTES", "hdl_rescore_ex", "hdl_rescore_ex_workspace_bytes",
    "hdl_rescore_shard", "hdl_rescore_shard_workspace_bytes", "hdl_merge_vocab_shards",
    "hdl_grpo_loss", "hdl_grpo_loss_workspace_bytes",
]

HDL_OK, HDL_ERR_INVALID_ARG, HDL_ERR_UNSUPPORTED, HDL_ERR_WORKSPACE = 0, 1, 2, 3
HDL_ERR_CUDA, HDL_ERR_TIMEOUT, HDL_ERR_BAD_TARGET = 4, 5, 6
HDL_BF16, HDL_F32 = 0, 1
HDL_STATIC_SCRATCH_BYTES = 64 << 20

_PKG = os.path.dirname(os.path.abspath(__file__))
_lib = None
_lock = threading.Lock()


def library_path() -> str:
    return os.path.join(_PKG, "libhdl.so")


class HdlError(RuntimeError):
    def __init__(self, fn: str, code: int):
        self.code = code
        super().__init__(f"{fn} failed: {_status_name(code)} ({code})")


class _RescoreOpts(ctypes.Structure):
    _fields_ = [("entropy_orig", ctypes.c_void_p), ("entropy_hind", ctypes.c_void_p),
                ("wait_timeout_ns", ctypes.c_uint64), ("fault_inject", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32)]


class _SelectOpts(ctypes.Structure):
    _fields_ = [("min_gap", ctypes.c_int32), ("gap_mode", ctypes.c_int32),
                ("lo", ctypes.c_int32), ("hi", ctypes.c_int32)]


def _declare(L):
    vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    L.hdl_abi_version.restype = i32
    L.hdl_abi_version.argtypes = []
    L.hdl_status_string.restype = ctypes.c_char_p
    L.hdl_status_string.argtypes = [ctypes.c_int]
    L.hdl_rescore_workspace_bytes.restype = sz
    L.hdl_rescore_workspace_bytes.argtypes = [i64, i32, i32, ctypes.c_int]
    L.hdl_rescore.restype = ctypes.c_int
    L.hdl_rescore.argtypes = [vp, vp, vp, ctypes.c_int, vp, i64, i32, i32, vp, vp, vp,
                              vp, sz, vp]
    L.hdl_rescore_ex_workspace_bytes.restype = sz
    L.hdl_rescore_ex_workspace_bytes.argtypes = [i64, i32, i32, ctypes.c_int,
                                                 ctypes.POINTER(_RescoreOpts)]
    L.hdl_rescore_ex.restype = ctypes.c_int
    L.hdl_rescore_ex.argtypes = [vp, vp, vp, ctypes.c_int, vp, i64, i32, i32, vp, vp, vp,
                                 ctypes.POINTER(_RescoreOpts), vp, sz, vp]
    L.hdl_rescore_shard_workspace_bytes.restype = sz
    L.hdl_rescore_shard_workspace_bytes.argtypes = [i64, i32, i32, ctypes.c_int]
    L.hdl_rescore_shard.restype = ctypes.c_int
    L.hdl_rescore_shard.argtypes = [vp, vp, vp, ctypes.c_int, vp, i64, i32, i32, i32, vp, vp,
                                    sz, vp]
    L.hdl_merge_vocab_shards.restype = ctypes.c_int
    L.hdl_merge_vocab_shards.argtypes = [vp, i32, i64, vp, vp, vp, vp, vp, vp]
    L.hdl_grpo_loss_workspace_bytes.restype = sz
    L.hdl_grpo_loss_workspace_bytes.argtypes = []
    L.hdl_grpo_loss.restype = ctypes.c_int
    L.hdl_grpo_loss.argtypes = [vp, vp, vp, i64, vp, i32, vp, vp, i32, ctypes.c_float,
                                ctypes.c_float, vp, vp, vp, vp, sz, vp]
    L.hdl_device_status.restype = ctypes.c_int
    L.hdl_device_status.argtypes = [vp, sz, vp, ctypes.POINTER(ctypes.c_uint32)]
    L.hdl_select_branches.restype = ctypes.c_int
    L.hdl_select_branches.argtypes = [vp, vp, i64, vp, i32, i32,
                                      ctypes.POINTER(_SelectOpts), vp, vp, vp, vp]
    L.hdl_assign_continuations.restype = ctypes.c_int
    L.hdl_assign_continuations.argtypes = [vp, vp, i32, i32, vp, i32, vp, i64, vp]
    L.hdl_suffix_mask.restype = ctypes.c_int
    L.hdl_suffix_mask.argtypes = [vp, vp, i32, vp, vp, i64, vp]
    L.hdl_rescore_noalloc.restype = ctypes.c_int
    L.hdl_rescore_noalloc.argtypes = [vp, vp, vp, ctypes.c_int, vp, i64, i32, i32, vp, vp, vp,
                                      ctypes.POINTER(ctypes.c_void_p), vp]
    return L


def lib():
    """Load libhdl.so (built by ``__graft_entry__.build()``); raise if absent."""
    global _lib
    if _lib is None:
        with _lock:
            if _lib is None:
                path = library_path()
                if not os.path.exists(path):
                    raise RuntimeError(
                        f"libhdl.so not found at {path}: build it first with "
                        "`python -c 'import __graft_entry__ as g; g.build()'`")
                _lib = _declare(ctypes.CDLL(path))
    return _lib


def _status_name(code: int) -> str:
    try:
        return lib().hdl_status_string(code).decode()
    except Exception:  # the name is only cosmetic
        return str(code)


def _check(fn: str, code: int):
    if code != HDL_OK:
        raise HdlError(fn, code)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream, device=None) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream(device)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _dev(t: torch.Tensor, name: str, dtype=None, numel: Optional[int] = None,
         device: Optional[torch.device] = None):
    """Check one tensor argument.  The C entry points receive raw pointers and
    take every length from the scalar arguments, so a buffer shorter than
    those lengths, or one on another device, must be caught here."""
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.device.type != "cuda":
        raise ValueError(f"{name} must be a CUDA tensor (got {t.device})")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, the other arguments on {device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype} (got {t.dtype})")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name} must hold {numel} elements (got {t.numel()})")


def _empty_like_phase(n: int, dtype, like: torch.Tensor, period: int) -> torch.Tensor:
    """An empty [n] tensor whose address has the same residue mod `period`
    bytes as `like`'s, so that the kernels' 16-byte vector paths (taken when
    the streams' alignments agree) still apply to sliced inputs."""
    esize = torch.empty(0, dtype=dtype).element_size()
    shift = (like.data_ptr() % period) // esize
    buf = torch.empty(n + period // esize, dtype=dtype, device=like.device)
    off = (shift - buf.data_ptr() % period // esize) % (period // esize)
    return buf[off:off + n]


def _lm_inputs(h_orig, h_hind, w, targets, w_name="w_lmhead"):
    """Validate the operands of a re-scoring call; returns (dtype code, N, d, V, device)."""
    _dev(h_orig, "h_orig")
    dev = h_orig.device
    _dev(h_hind, "h_hind", device=dev)
    _dev(w, w_name, device=dev)
    _dev(targets, "targets", torch.int32, device=dev)
    dt = _hdl_dtype(h_orig)
    if h_hind.dtype != h_orig.dtype or w.dtype != h_orig.dtype:
        raise ValueError(f"h_orig, h_hind and {w_name} must share one dtype")
    if h_orig.dim() != 2 or w.dim() != 2:
        raise ValueError(f"h_orig and {w_name} must be 2-D")
    N, d = h_orig.shape
    V = w.shape[0]
    if h_hind.shape != (N, d) or w.shape != (V, d) or targets.shape != (N,):
        raise ValueError(f"shape mismatch between h_orig, h_hind, {w_name}, targets")
    return dt, N, d, V, dev


def _hdl_dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return HDL_BF16
    if t.dtype == torch.float32:
        return HDL_F32
    raise ValueError(f"hidden states / LM head must be bf16 or fp32 (got {t.dtype})")


# -------------------------------------------------------------- entry points
def hdl_abi_version() -> int:
    return int(lib().hdl_abi_version())


def hdl_status_string(code: int) -> str:
    return lib().hdl_status_string(code).decode()


def hdl_rescore_workspace_bytes(n_tokens: int, d: int, vocab: int, dtype=HDL_BF16) -> int:
    if isinstance(dtype, torch.dtype):
        dtype = HDL_BF16 if dtype == torch.bfloat16 else HDL_F32
    return int(lib().hdl_rescore_workspace_bytes(n_tokens, d, vocab, dtype))


def hdl_rescore(h_orig, h_hind, w_lmhead, targets, logp_orig=None, logp_hind=None,
                delta=None, workspace=None, want_delta=True, stream=None):
    """log p^0(y_t), log p^H(y_t) and |Delta_t| for every token (Eq. div).

    Returns (logp_orig, logp_hind, delta, workspace); outputs not given are
    allocated.  Asynchronous on ``stream``; device-side errors surface through
    :func:`hdl_device_status` on the returned workspace.
    """
    dt, N, d, V, dev = _lm_inputs(h_orig, h_hind, w_lmhead, targets)
    if logp_orig is None:
        logp_orig = torch.empty(N, dtype=torch.float32, device=dev)
    if logp_hind is None:
        logp_hind = torch.empty(N, dtype=torch.float32, device=dev)
    if delta is None and want_delta:
        delta = torch.empty(N, dtype=torch.float32, device=dev)
    for t, n in ((logp_orig, "logp_orig"), (logp_hind, "logp_hind")):
        _dev(t, n, torch.float32, N, dev)
    if delta is not None:
        _dev(delta, "delta", torch.float32, N, dev)
    need = hdl_rescore_workspace_bytes(N, d, V, dt)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    _dev(workspace, "workspace", torch.uint8, device=dev)
    code = lib().hdl_rescore(_ptr(h_orig), _ptr(h_hind), _ptr(w_lmhead), dt, _ptr(targets),
                             N, d, V, _ptr(logp_orig), _ptr(logp_hind), _ptr(delta),
                             _ptr(workspace), workspace.numel(), _stream(stream, dev))
    _check("hdl_rescore", code)
    return logp_orig, logp_hind, delta, workspace


def _opts(entropy_orig=None, entropy_hind=None, wait_timeout_ns=0, fault_inject=0):
    return _RescoreOpts(None if entropy_orig is None else entropy_orig.data_ptr(),
                        None if entropy_hind is None else entropy_hind.data_ptr(),
                        int(wait_timeout_ns), int(fault_inject), 0)


def hdl_rescore_ex_workspace_bytes(n_tokens: int, d: int, vocab: int, dtype=HDL_BF16,
                                   entropy: bool = False) -> int:
    if isinstance(dtype, torch.dtype):
        dtype = HDL_BF16 if dtype == torch.bfloat16 else HDL_F32
    o = _RescoreOpts(1 if entropy else None, None, 0, 0, 0)
    return int(lib().hdl_rescore_ex_workspace_bytes(n_tokens, d, vocab, dtype, ctypes.byref(o)))


def hdl_rescore_ex(h_orig, h_hind, w_lmhead, targets, logp_orig=None, logp_hind=None,
                   delta=None, entropy_orig=None, entropy_hind=None, want_entropy=True,
                   want_entropy_hind=False, wait_timeout_ns=0, fault_inject=0, workspace=None,
                   stream=None):
    """hdl_rescore plus the next-token entropies (Section 4.1, Entropy selector).

    Returns (logp_orig, logp_hind, delta, entropy_orig, entropy_hind, workspace).
    ``fault_inject`` is the library's test hook (see hdl_rescore_opts)."""
    dt, N, d, V, dev = _lm_inputs(h_orig, h_hind, w_lmhead, targets)

    def out(t, want):
        if t is None and want:
            t = torch.empty(N, dtype=torch.float32, device=dev)
        if t is not None:
            _dev(t, "output", torch.float32, N, dev)
        return t
    logp_orig, logp_hind = out(logp_orig, True), out(logp_hind, True)
    delta = out(delta, True)
    entropy_orig = out(entropy_orig, want_entropy)
    entropy_hind = out(entropy_hind, want_entropy_hind)
    o = _opts(entropy_orig, entropy_hind, wait_timeout_ns, fault_inject)
    need = int(lib().hdl_rescore_ex_workspace_bytes(N, d, V, dt, ctypes.byref(o)))
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    _dev(workspace, "workspace", torch.uint8, device=dev)
    code = lib().hdl_rescore_ex(_ptr(h_orig), _ptr(h_hind), _ptr(w_lmhead), dt, _ptr(targets),
                                N, d, V, _ptr(logp_orig), _ptr(logp_hind), _ptr(delta),
                                ctypes.byref(o), _ptr(workspace), workspace.numel(),
                                _stream(stream, dev))
    _check("hdl_rescore_ex", code)
    return logp_orig, logp_hind, delta, entropy_orig, entropy_hind, workspace


def hdl_device_status(workspace, stream=None):
    """(status code, raw status word) of a re-scoring workspace; synchronises.

    ``workspace`` is the workspace tensor of an earlier call, or the scratch
    address that :func:`hdl_rescore_noalloc` returned."""
    if isinstance(workspace, int):
        ptr, size, dev = ctypes.c_void_p(workspace), HDL_STATIC_SCRATCH_BYTES, None
    else:
        _dev(workspace, "workspace", torch.uint8)
        ptr, size, dev = _ptr(workspace), workspace.numel(), workspace.device
    raw = ctypes.c_uint32(0)
    code = lib().hdl_device_status(ptr, size, _stream(stream, dev), ctypes.byref(raw))
    return int(code), int(raw.value)


def hdl_select_branches(delta, valid, root_offsets, k: int, min_gap: int = 0,
                        gap_mode: int = 0, lo: int = 0, hi: int = 0, branch_pos=None,
                        n_selected=None, branch_delta=None, want_delta=True, stream=None):
    """Top-k branch points per root; returns (branch_pos [R,k], n_selected [R], branch_delta)."""
    _dev(delta, "delta", torch.float32)
    dev = delta.device
    if valid is not None:
        _dev(valid, "valid", torch.uint8, delta.numel(), dev)
    _dev(root_offsets, "root_offsets", torch.int64, device=dev)
    R = root_offsets.numel() - 1
    if R < 0:
        raise ValueError("root_offsets needs n_roots + 1 entries")
    if branch_pos is None:
        branch_pos = torch.empty((R, k), dtype=torch.int32, device=dev)
    if n_selected is None:
        n_selected = torch.empty(R, dtype=torch.int32, device=dev)
    if branch_delta is None and want_delta:
        branch_delta = torch.empty((R, k), dtype=torch.float32, device=dev)
    _dev(branch_pos, "branch_pos", torch.int32, R * k, dev)
    _dev(n_selected, "n_selected", torch.int32, R, dev)
    if branch_delta is not None:
        _dev(branch_delta, "branch_delta", torch.float32, R * k, dev)
    opts = _SelectOpts(min_gap, gap_mode, lo, hi)
    code = lib().hdl_select_branches(_ptr(delta), _ptr(valid), delta.numel(),
                                     _ptr(root_offsets), R, k, ctypes.byref(opts),
                                     _ptr(branch_pos), _ptr(n_selected), _ptr(branch_delta),
                                     _stream(stream, dev))
    _check("hdl_select_branches", code)
    return branch_pos, n_selected, branch_delta


def hdl_assign_continuations(n_selected, branch_pos, conts_per_root, extra_to_higher=True,
                             cont_branch=None, n_cont: Optional[int] = None, stream=None):
    """Root-relative branch position of every continuation (root-major)."""
    _dev(branch_pos, "branch_pos", torch.int32)
    dev = branch_pos.device
    if branch_pos.dim() != 2:
        raise ValueError("branch_pos must be [n_roots, k]")
    R, k = branch_pos.shape
    _dev(n_selected, "n_selected", torch.int32, R, dev)
    _dev(conts_per_root, "conts_per_root", torch.int32, R, dev)
    if cont_branch is None:
        if n_cont is None:
            raise ValueError("give cont_branch or n_cont (the total continuation count)")
        cont_branch = torch.empty(n_cont, dtype=torch.int32, device=dev)
    _dev(cont_branch, "cont_branch", torch.int32, device=dev)
    code = lib().hdl_assign_continuations(_ptr(n_selected), _ptr(branch_pos), R, k,
                                          _ptr(conts_per_root), 1 if extra_to_higher else 0,
                                          _ptr(cont_branch), cont_branch.numel(),
                                          _stream(stream, dev))
    _check("hdl_assign_continuations", code)
    return cont_branch


def hdl_suffix_mask(cont_branch, cont_offsets, cont_valid=None, mask=None,
                    mask_len: Optional[int] = None, stream=None):
    """Suffix-only loss mask of packed continuations (uint8)."""
    _dev(cont_branch, "cont_branch", torch.int32)
    dev = cont_branch.device
    C = cont_branch.numel()
    _dev(cont_offsets, "cont_offsets", torch.int64, C + 1, dev)
    if cont_valid is not None:
        _dev(cont_valid, "cont_valid", torch.uint8, device=dev)
    if mask is None:
        if mask_len is None:
            mask_len = cont_valid.numel() if cont_valid is not None else None
        if mask_len is None:
            raise ValueError("give mask, mask_len or cont_valid")
        if cont_valid is not None:
            mask = _empty_like_phase(mask_len, torch.uint8, cont_valid, 16).zero_()
        else:
            mask = torch.zeros(mask_len, dtype=torch.uint8, device=dev)
    _dev(mask, "mask", torch.uint8, device=dev)
    if cont_valid is not None and cont_valid.numel() != mask.numel():
        raise ValueError("cont_valid and mask must have the same length")
    code = lib().hdl_suffix_mask(_ptr(cont_branch), _ptr(cont_offsets), C, _ptr(cont_valid),
                                 _ptr(mask), mask.numel(), _stream(stream, dev))
    _check("hdl_suffix_mask", code)
    return mask


def hdl_rescore_noalloc(h_orig, h_hind, w_lmhead, targets, logp_orig, logp_hind, delta=None,
                        stream=None):
    """hdl_rescore without a workspace, for callers that must not allocate
    device memory while they run (inference-runtime plugins, pool-owned
    device memory, latency-critical loops).  Scratch is one static 64 MiB
    device array shared by all calls: calls that overlap on the GPU race, and
    problems needing more scratch are rejected (HDL_ERR_UNSUPPORTED).  Every
    output tensor must be given; nothing is allocated here either.  Returns
    the device address of the scratch array, which hdl_device_status()
    accepts."""
    dt, N, d, V, dev = _lm_inputs(h_orig, h_hind, w_lmhead, targets)
    for t, n in ((logp_orig, "logp_orig"), (logp_hind, "logp_hind")):
        _dev(t, n, torch.float32, N, dev)
    if delta is not None:
        _dev(delta, "delta", torch.float32, N, dev)
    scratch = ctypes.c_void_p(0)
    code = lib().hdl_rescore_noalloc(_ptr(h_orig), _ptr(h_hind), _ptr(w_lmhead), dt,
                                     _ptr(targets), N, d, V, _ptr(logp_orig), _ptr(logp_hind),
                                     _ptr(delta), ctypes.byref(scratch), _stream(stream, dev))
    _check("hdl_rescore_noalloc", code)
    return scratch.value


def hdl_rescore_shard_workspace_bytes(n_tokens: int, d: int, vocab_shard: int,
                                      dtype=HDL_BF16) -> int:
    if isinstance(dtype, torch.dtype):
        dtype = HDL_BF16 if dtype == torch.bfloat16 else HDL_F32
    return int(lib().hdl_rescore_shard_workspace_bytes(n_tokens, d, vocab_shard, dtype))


def hdl_rescore_shard(h_orig, h_hind, w_shard, targets, vocab_offset: int, stats=None,
                      workspace=None, stream=None):
    """Per-row statistics of one vocabulary shard of the LM head: a
    [2, n_tokens, 4] float tensor (max in log2 units, sum, target logit or NaN,
    entropy numerator), to be exchanged and merged by hdl_merge_vocab_shards."""
    dt, N, d, Vs, dev = _lm_inputs(h_orig, h_hind, w_shard, targets, "w_shard")
    if stats is None:
        stats = torch.empty((2, N, 4), dtype=torch.float32, device=dev)
    _dev(stats, "stats", torch.float32, 2 * N * 4, dev)
    need = hdl_rescore_shard_workspace_bytes(N, d, Vs, dt)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    _dev(workspace, "workspace", torch.uint8, device=dev)
    code = lib().hdl_rescore_shard(_ptr(h_orig), _ptr(h_hind), _ptr(w_shard), dt, _ptr(targets),
                                   N, d, Vs, int(vocab_offset), _ptr(stats), _ptr(workspace),
                                   workspace.numel(), _stream(stream, dev))
    _check("hdl_rescore_shard", code)
    return stats, workspace


def hdl_merge_vocab_shards(stats, logp_orig=None, logp_hind=None, delta=None,
                           entropy_orig=None, entropy_hind=None, want_entropy=True,
                           stream=None):
    """Merge stacked shard statistics [P, 2, n_tokens, 4] into log-probs,
    |Delta| and entropies: returns (logp_orig, logp_hind, delta, H_orig, H_hind)."""
    _dev(stats, "stats", torch.float32)
    P, two, N, four = stats.shape
    if two != 2 or four != 4:
        raise ValueError("stats must be [n_shards, 2, n_tokens, 4]")
    dev = stats.device

    def out(t, want=True):
        if t is None and want:
            t = torch.empty(N, dtype=torch.float32, device=dev)
        if t is not None:
            _dev(t, "output", torch.float32, N, dev)
        return t
    logp_orig, logp_hind, delta = out(logp_orig), out(logp_hind), out(delta)
    entropy_orig, entropy_hind = out(entropy_orig, want_entropy), out(entropy_hind, want_entropy)
    code = lib().hdl_merge_vocab_shards(_ptr(stats), P, N, _ptr(logp_orig), _ptr(logp_hind),
                                        _ptr(delta), _ptr(entropy_orig), _ptr(entropy_hind),
                                        _stream(stream, dev))
    _check("hdl_merge_vocab_shards", code)
    return logp_orig, logp_hind, delta, entropy_orig, entropy_hind


def hdl_grpo_loss_workspace_bytes() -> int:
    return int(lib().hdl_grpo_loss_workspace_bytes())


def hdl_grpo_loss(logp_new, logp_old, mask, traj_offsets, rewards, group_offsets,
                  eps_low: float = 0.2, eps_high: float = 0.28, advantages=None, grad=None,
                  want_grad=True, stats=None, workspace=None, stream=None):
    """Group advantages and the clipped token-level policy loss (Section 4.1).

    Returns (advantages [J], grad [T] or None, stats [4] = loss, masked
    tokens, clipped fraction, mean ratio), all on the device."""
    _dev(logp_new, "logp_new", torch.float32)
    dev = logp_new.device
    T, J, G = logp_new.numel(), traj_offsets.numel() - 1, group_offsets.numel() - 1
    if J < 0 or G < 0:
        raise ValueError("traj_offsets and group_offsets need count + 1 entries")
    _dev(logp_old, "logp_old", torch.float32, T, dev)
    _dev(mask, "mask", torch.uint8, T, dev)
    _dev(traj_offsets, "traj_offsets", torch.int64, device=dev)
    _dev(rewards, "rewards", torch.float32, J, dev)
    _dev(group_offsets, "group_offsets", torch.int32, device=dev)
    if advantages is None:
        advantages = torch.zeros(J, dtype=torch.float32, device=dev)
    if grad is None and want_grad:
        grad = _empty_like_phase(T, torch.float32, logp_new, 16)
    if stats is None:
        stats = torch.empty(4, dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = torch.empty(hdl_grpo_loss_workspace_bytes(), dtype=torch.uint8, device=dev)
    _dev(advantages, "advantages", torch.float32, J, dev)
    if grad is not None:
        _dev(grad, "grad", torch.float32, T, dev)
    _dev(stats, "stats", torch.float32, 4, dev)
    _dev(workspace, "workspace", torch.uint8, device=dev)
    code = lib().hdl_grpo_loss(_ptr(logp_new), _ptr(logp_old), _ptr(mask), T, _ptr(traj_offsets),
                               J, _ptr(rewards), _ptr(group_offsets), G, float(eps_low),
                               float(eps_high), _ptr(advantages), _ptr(grad), _ptr(stats),
                               _ptr(workspace), workspace.numel(), _stream(stream, dev))
    _check("hdl_grpo_loss", code)
    return advantages, grad, stats
