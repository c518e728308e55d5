"""Python binding of libasrspec (ctypes): the C ABI of include/asrspec.h under
the same names.  Argument marshalling only: every step of the computation runs
in the library's CUDA kernels.  Device arrays are torch tensors; with host I/O
enabled, array arguments are numpy arrays.

The library must have been built (``paper_2608_12703_gb300.build.build()``);
loading fails loudly otherwise: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libasrspec.so")

ASR_OK = 0
ERRORS = {-1: "ASR_E_INVAL", -2: "ASR_E_STATE", -3: "ASR_E_CAPACITY", -4: "ASR_E_OOM",
          -5: "ASR_E_CUDA", -6: "ASR_E_DEVICE"}
ST_BAD_TOKEN, ST_BAD_LENS, ST_CAPACITY, ST_WAIT_TIMEOUT, ST_NOT_READY, ST_BAD_TREE, ST_BOUNDS = 1, 2, 4, 8, 16, 32, 64

EXPORTED = [
    "asr_spec_create", "asr_spec_set_host_io", "asr_spec_encode_cache", "asr_spec_prefill",
    "asr_spec_verify", "asr_spec_rollback", "asr_spec_state", "asr_spec_debug_logits",
    "asr_spec_status", "asr_spec_last_error", "asr_spec_destroy", "asr_spec_synth_drafts",
    "asr_spec_test_gemm", "asr_spec_set_graphs", "asr_spec_profile", "asr_spec_profile_read",
    "asr_spec_gemm_noalloc", "asr_spec_timeline", "asr_spec_timeline_read",
    "asr_spec_verify_tree", "asr_spec_restart", "asr_spec_fewrow_trace", "asr_spec_fewrow_trace_read",
    "asr_spec_debug_anchor_profile", "asr_spec_draft_create", "asr_spec_draft_propose",
    "asr_spec_draft_set_threshold",
]
DRAFT_WIN = {"anchor": 0, "shifted": 1, "random": 2, None: 3}
PROF_CLASSES = ["qkv", "resid", "query", "mlp_up", "self_attn", "cross_attn", "lm_head", "layernorm", "other",
                "qkv_self", "query_cross"]
TL_CAP = 65536
TL_GEMM, TL_LN_FUSED = 16, 32
TL_KINDS = {0: "other", 1: "plan", 2: "embed", 3: "layernorm", 4: "attn_self", 5: "attn_cross", 6: "accept_anchor",
            8: "qkv_self", 9: "query_cross"}
TL_GEMM_EPILOGUES = {0: "plain", 1: "qkv", 2: "residual", 3: "query", 4: "gelu", 5: "cross_kv", 6: "argmax"}


def tl_kind_name(kind: int) -> str:
    """Readable name of a timeline launch kind (ASR_TL_* codes)."""
    if kind >= TL_GEMM:
        name = "gemm_" + TL_GEMM_EPILOGUES.get((kind - TL_GEMM) % TL_GEMM, str(kind))
        return name + ("+ln" if kind & TL_LN_FUSED else "")
    return TL_KINDS.get(kind, str(kind))


class AsrModelDims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "n_layers", "d_model", "n_heads", "d_ffn", "vocab", "max_pos", "max_batch", "max_draft",
        "max_enc", "dtype", "anchor_layer")]


class AsrWeights(ctypes.Structure):
    _fields_ = [("blob", ctypes.POINTER(ctypes.c_float)), ("n_floats", ctypes.c_size_t)]


class AsrSpecError(RuntimeError):
    pass


_lib = None


def lib():
    """Load the shared library (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise AsrSpecError(f"libasrspec.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, p32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p
    L.asr_spec_create.argtypes = [ctypes.POINTER(AsrModelDims), ctypes.POINTER(AsrWeights), vp,
                                  ctypes.POINTER(vp)]
    L.asr_spec_set_host_io.argtypes = [vp, ctypes.c_int]
    L.asr_spec_encode_cache.argtypes = [vp, i32, vp, i32, p32]
    L.asr_spec_prefill.argtypes = [vp, p32, i32]
    L.asr_spec_verify.argtypes = [vp, p32, p32, i32, p32, p32, p32, p32]
    L.asr_spec_verify_tree.argtypes = [vp, p32, p32, p32, i32, p32, p32, p32, p32, p32]
    L.asr_spec_rollback.argtypes = [vp, p32, p32]
    L.asr_spec_restart.argtypes = [vp, p32]
    L.asr_spec_draft_create.argtypes = [vp, ctypes.POINTER(AsrWeights)]
    L.asr_spec_draft_propose.argtypes = [vp, i32, i32, p32, p32, p32, p32]
    L.asr_spec_draft_set_threshold.argtypes = [vp, ctypes.c_float]
    L.asr_spec_fewrow_trace.argtypes = [vp, i32]
    L.asr_spec_fewrow_trace_read.argtypes = [vp, vp, ctypes.c_int64, vp]
    L.asr_spec_debug_anchor_profile.argtypes = [vp, vp]
    L.asr_spec_state.argtypes = [vp, p32, p32]
    L.asr_spec_debug_logits.argtypes = [vp, vp, i32]
    L.asr_spec_status.argtypes = [vp]
    L.asr_spec_last_error.argtypes = [vp]
    L.asr_spec_last_error.restype = ctypes.c_char_p
    L.asr_spec_destroy.argtypes = [vp]
    L.asr_spec_destroy.restype = None
    L.asr_spec_synth_drafts.argtypes = [vp, p32, p32, p32, i32, p32, i32, p32, p32]
    L.asr_spec_test_gemm.argtypes = [i32, vp, vp, vp, i32, i32, i32, vp]
    L.asr_spec_set_graphs.argtypes = [vp, ctypes.c_int]
    L.asr_spec_profile.argtypes = [vp, ctypes.c_int]
    L.asr_spec_profile_read.argtypes = [vp, vp, vp, vp]
    L.asr_spec_gemm_noalloc.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp]
    L.asr_spec_timeline.argtypes = [vp, i32]
    L.asr_spec_timeline_read.argtypes = [vp, vp, vp, i32, vp]
    for name in EXPORTED:
        if name not in ("asr_spec_last_error", "asr_spec_destroy"):
            getattr(L, name).restype = ctypes.c_int
    _lib = L
    return L


def ptr(x) -> Optional[int]:
    """Address of a torch tensor or numpy array (contiguous), or None."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("array must be contiguous")
        return x.ctypes.data
    if not x.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return x.data_ptr()


def _check(h, rc, what):
    if rc < 0:
        msg = lib().asr_spec_last_error(h).decode() if h else ""
        raise AsrSpecError(f"{what}: {ERRORS.get(rc, rc)} {msg}")
    return rc


def asr_spec_create(dims: dict, blob: np.ndarray, stream=None) -> int:
    d = AsrModelDims(**dims)
    blob = np.ascontiguousarray(blob, dtype=np.float32)
    w = AsrWeights(blob.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), blob.size)
    h = ctypes.c_void_p()
    st = None if stream is None else ctypes.c_void_p(stream)
    _check(None, lib().asr_spec_create(ctypes.byref(d), ctypes.byref(w), st, ctypes.byref(h)), "asr_spec_create")
    return h.value


def asr_spec_set_host_io(h, host_io: bool):
    return _check(h, lib().asr_spec_set_host_io(h, int(host_io)), "asr_spec_set_host_io")


def asr_spec_encode_cache(h, B, enc_states, t_max, enc_lens):
    return _check(h, lib().asr_spec_encode_cache(h, B, ptr(enc_states), t_max, ptr(enc_lens)),
                  "asr_spec_encode_cache")


def asr_spec_prefill(h, prompt, P0):
    return _check(h, lib().asr_spec_prefill(h, ptr(prompt), P0), "asr_spec_prefill")


def asr_spec_verify(h, draft, lens, k, accepted, bonus, kv_len, anchor):
    return _check(h, lib().asr_spec_verify(h, ptr(draft), ptr(lens), k, ptr(accepted), ptr(bonus),
                                           ptr(kv_len), ptr(anchor)), "asr_spec_verify")


def asr_spec_verify_tree(h, tokens, parent, lens, n, accepted, bonus, kv_len, anchor, path):
    return _check(h, lib().asr_spec_verify_tree(h, ptr(tokens), ptr(parent), ptr(lens), n, ptr(accepted), ptr(bonus),
                                                ptr(kv_len), ptr(anchor), ptr(path)), "asr_spec_verify_tree")


def asr_spec_restart(h, restart):
    return _check(h, lib().asr_spec_restart(h, ptr(restart)), "asr_spec_restart")


def asr_spec_draft_create(h, blob: np.ndarray):
    blob = np.ascontiguousarray(blob, dtype=np.float32)
    w = AsrWeights(blob.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), blob.size)
    return _check(h, lib().asr_spec_draft_create(h, ctypes.byref(w)), "asr_spec_draft_create")


def asr_spec_draft_propose(h, k, window, centers, total_len, draft_out, lens_out):
    return _check(h, lib().asr_spec_draft_propose(h, k, window, ptr(centers), ptr(total_len), ptr(draft_out),
                                                  ptr(lens_out)), "asr_spec_draft_propose")


def asr_spec_draft_set_threshold(h, threshold: float):
    return _check(h, lib().asr_spec_draft_set_threshold(h, float(threshold)), "asr_spec_draft_set_threshold")


def asr_spec_debug_anchor_profile(h, out):
    return _check(h, lib().asr_spec_debug_anchor_profile(h, ptr(out)), "asr_spec_debug_anchor_profile")


def asr_spec_rollback(h, new_len, new_pending):
    return _check(h, lib().asr_spec_rollback(h, ptr(new_len), ptr(new_pending)), "asr_spec_rollback")


def asr_spec_state(h, kv_len, pending):
    return _check(h, lib().asr_spec_state(h, ptr(kv_len), ptr(pending)), "asr_spec_state")


def asr_spec_debug_logits(h, out, max_rows):
    return _check(h, lib().asr_spec_debug_logits(h, ptr(out), max_rows), "asr_spec_debug_logits")


def asr_spec_status(h) -> int:
    return _check(h, lib().asr_spec_status(h), "asr_spec_status")


def asr_spec_last_error(h) -> str:
    return lib().asr_spec_last_error(h).decode()


def asr_spec_destroy(h):
    lib().asr_spec_destroy(h)


def asr_spec_synth_drafts(h, truth, total_len, repl, k_repl, shift, k, draft_out, lens_out):
    return _check(h, lib().asr_spec_synth_drafts(h, ptr(truth), ptr(total_len), ptr(repl), k_repl, ptr(shift),
                                                 k, ptr(draft_out), ptr(lens_out)), "asr_spec_synth_drafts")


def asr_spec_test_gemm(impl, A, B, C, M, N, K, stream=None):
    return _check(None, lib().asr_spec_test_gemm(impl, ptr(A), ptr(B), ptr(C), M, N, K,
                                                 None if stream is None else ctypes.c_void_p(stream)),
                  "asr_spec_test_gemm")


def asr_spec_set_graphs(h, enable: bool):
    return _check(h, lib().asr_spec_set_graphs(h, int(enable)), "asr_spec_set_graphs")


def asr_spec_profile(h, enable: bool):
    return _check(h, lib().asr_spec_profile(h, int(enable)), "asr_spec_profile")


def asr_spec_profile_read(h):
    """Returns (ms per class, launches per class, traffic counters)."""
    ms = np.zeros(len(PROF_CLASSES), dtype=np.float64)
    launches = np.zeros(len(PROF_CLASSES), dtype=np.int64)
    traffic = np.zeros(8, dtype=np.uint64)
    _check(h, lib().asr_spec_profile_read(h, ms.ctypes.data, launches.ctypes.data, traffic.ctypes.data),
           "asr_spec_profile_read")
    return ms, launches, traffic


def asr_spec_timeline(h, enable: bool):
    return _check(h, lib().asr_spec_timeline(h, 1 if enable else 0), "asr_spec_timeline")


def asr_spec_timeline_read(h):
    """Returns (ns [n][4] = start, past the wait, midpoint, end; kinds [n]) of the recorded launches."""
    ns = np.zeros((TL_CAP, 4), dtype=np.uint64)
    kinds = np.zeros(TL_CAP, dtype=np.int32)
    count = ctypes.c_int32(0)
    _check(h, lib().asr_spec_timeline_read(h, ns.ctypes.data, kinds.ctypes.data, TL_CAP, ctypes.byref(count)),
           "asr_spec_timeline_read")
    n = min(count.value, TL_CAP)
    return ns[:n].copy(), kinds[:n].copy()


FR_TRACE_CTAS, FR_TRACE_PHASES = 320, 12


def asr_spec_fewrow_trace(h, enable: bool):
    return _check(h, lib().asr_spec_fewrow_trace(h, 1 if enable else 0), "asr_spec_fewrow_trace")


def asr_spec_fewrow_trace_read(h):
    """Per-CTA phase stamps (ns) of the last traced call's few-row launches,
    [n_launches][320][12] (entry, past wait, rows ready, weights landed,
    reduced, exchange landed, attention done, exit, first K/V chunk landed,
    first chunk combined, merge inputs landed; 0 = none)."""
    n = ctypes.c_int32(0)
    _check(h, lib().asr_spec_fewrow_trace_read(h, None, 0, ctypes.byref(n)), "asr_spec_fewrow_trace_read")
    out = np.zeros((n.value, FR_TRACE_CTAS, FR_TRACE_PHASES), dtype=np.uint64)
    _check(h, lib().asr_spec_fewrow_trace_read(h, out.ctypes.data, out.size, ctypes.byref(n)),
           "asr_spec_fewrow_trace_read")
    return out


def asr_spec_gemm_noalloc(A, B, C, M, N, K, splits, stream=None):
    """Split-K GEMM whose scratch is a fixed device array (no allocation)."""
    return _check(None, lib().asr_spec_gemm_noalloc(ptr(A), ptr(B), ptr(C), M, N, K, splits,
                                                    None if stream is None else ctypes.c_void_p(stream)),
                  "asr_spec_gemm_noalloc")
