"""ctypes binding of libgs (include/gs.h): same names, argument marshalling only.

Every step of the decoding path runs in libgs's CUDA kernels; this module only
converts Python values to the C structs and pointers.  PyTorch supplies device
memory and streams.  Importing this module fails loudly if libgs.so has not
been built (``python -c "import __graft_entry__ as g; g.build()"``).
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgs.so")

GS_OK = 0
GS_ERR_INVALID_ARG = 1
GS_ERR_OOM = 2
GS_ERR_UNSUPPORTED = 3
GS_ERR_CUDA = 4
GS_ERR_DEVICE_CHECK = 5
GS_ERR_TIMEOUT = 6
GS_ACCEPT_GREEDY = 0
GS_ACCEPT_STOCHASTIC = 1
EPI_STORE_F16, EPI_RESID_F32, EPI_SWIGLU, EPI_ARGMAX = 0, 1, 2, 3
ATTN_DRAFT, ATTN_VERIFY = 0, 1
KIND_NAMES = ("window", "embed", "qkv", "attention", "o_proj", "gate_up", "down", "lm_head",
              "accept")

ERROR_NAMES = {0: "GS_OK", 1: "GS_ERR_INVALID_ARG", 2: "GS_ERR_OOM", 3: "GS_ERR_UNSUPPORTED",
               4: "GS_ERR_CUDA", 5: "GS_ERR_DEVICE_CHECK", 6: "GS_ERR_TIMEOUT"}


class GsError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERROR_NAMES.get(code, code)}: {msg}")
        self.code = code


class gs_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in
                ("n_layers", "d_model", "n_heads", "n_kv_heads", "head_dim", "d_ffn", "vocab")] + [
        ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float)] + [
        (n, ctypes.c_int) for n in ("mask_token_id", "eos_token_id", "max_batch", "max_ctx",
                                    "max_K", "max_prefill", "kv_pages", "split_pages")]


_PP = ctypes.POINTER(ctypes.c_void_p)


class gs_weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("lm_head", ctypes.c_void_p),
                ("final_norm", ctypes.c_void_p), ("attn_norm", _PP), ("w_qkv", _PP),
                ("w_o", _PP), ("ffn_norm", _PP), ("w_gate_up", _PP), ("w_down", _PP)]


class gs_force(ctypes.Structure):
    _fields_ = [("teacher", ctypes.c_void_p), ("teacher_stride", ctypes.c_int64),
                ("L_sched", ctypes.c_void_p), ("L_stride", ctypes.c_int64)]


class gs_debug(ctypes.Structure):
    _fields_ = [("draft_tok", ctypes.c_void_p), ("verify_in", ctypes.c_void_p),
                ("verify_tok", ctypes.c_void_p), ("draft_logits", ctypes.c_void_p),
                ("verify_logits", ctypes.c_void_p)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libgs.so not built at {LIB_PATH}; run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    sig = {
        "gs_workspace_bytes": (sz, [ctypes.POINTER(gs_config)]),
        "gs_create": (i32, [ctypes.POINTER(gs_config), ctypes.POINTER(gs_weights), vp, sz, vp,
                            ctypes.POINTER(vp)]),
        "gs_destroy": (i32, [vp]),
        "gs_last_error": (ctypes.c_char_p, [vp]),
        "gs_prefill": (i32, [vp, i32, vp, i32, vp, i32, i32, vp]),
        "gs_round": (i32, [vp, vp, i32, i32, i32, ctypes.POINTER(gs_force), vp, vp, vp,
                           ctypes.POINTER(gs_debug)]),
        "gs_seq_restore": (i32, [vp, i32, i32, i32, i32, i32, i32, i32]),
        "gs_set_sampling": (i32, [vp, ctypes.c_float, ctypes.c_uint64]),
        "gs_diffusion_block": (i32, [vp, vp, i32, i32, ctypes.c_float, vp, vp, vp, vp]),
        "gs_round_refined": (i32, [vp, vp, i32, i32, ctypes.c_float, ctypes.POINTER(gs_force), vp,
                                   vp, vp, vp]),
        "gs_round_launches": (i32, [vp]),
        "gs_round_profile": (i32, [vp, vp, i32, i32, ctypes.POINTER(gs_force), vp, vp, vp, i32,
                                   ctypes.POINTER(ctypes.c_float), ctypes.POINTER(i32),
                                   ctypes.POINTER(i32)]),
        "gs_seq_state": (i32, [vp, i32] + [ctypes.POINTER(i32)] * 5),
        "gs_release": (i32, [vp, i32]),
        "gs_sync_check": (i32, [vp]),
        "gs_wait_probe": (i32, [vp, i32]),
        "gs_attention_scratch_bytes": (sz, [i32] * 6),
        "gs_attention": (i32, [i32, vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, vp, vp, sz, i32,
                               vp]),
        "gs_linear_scratch_bytes": (sz, [i32, i32, i32]),
        "gs_linear": (i32, [vp, vp, vp, i32, i32, i32, i32, i32, vp, sz, vp]),
        "gs_linear_noalloc": (i32, [vp, vp, vp, i32, i32, i32, i32, i32, vp]),
        "gs_linear_noalloc_status": (i32, [vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


_lib = _load()
EXPORTED = ("gs_workspace_bytes", "gs_create", "gs_destroy", "gs_last_error", "gs_prefill",
            "gs_round", "gs_set_sampling", "gs_diffusion_block", "gs_round_refined", "gs_seq_restore", "gs_round_launches", "gs_round_profile", "gs_seq_state",
            "gs_release", "gs_sync_check", "gs_wait_probe",
            "gs_attention_scratch_bytes", "gs_attention", "gs_linear_scratch_bytes", "gs_linear",
            "gs_linear_noalloc", "gs_linear_noalloc_status")


def lib():
    return _lib


def _check(handle, rc: int) -> None:
    if rc != GS_OK:
        msg = _lib.gs_last_error(handle)
        raise GsError(rc, msg.decode() if msg else "")


# ------------------------------------------------------------------ same-name wrappers
def gs_workspace_bytes(cfg: gs_config) -> int:
    return int(_lib.gs_workspace_bytes(ctypes.byref(cfg)))


def gs_create(cfg: gs_config, w: gs_weights, workspace_ptr: int, ws_bytes: int, stream_ptr: int):
    h = ctypes.c_void_p()
    rc = _lib.gs_create(ctypes.byref(cfg), ctypes.byref(w), workspace_ptr, ws_bytes, stream_ptr,
                        ctypes.byref(h))
    _check(None, rc)
    return h


def gs_destroy(h) -> None:
    _check(None, _lib.gs_destroy(h))


def gs_last_error(h) -> str:
    m = _lib.gs_last_error(h)
    return m.decode() if m else ""


def gs_prefill(h, slot: int, vis_ptr: int, n_vis: int, text_ptr: int, n_text: int, max_new: int,
               x0_ptr: int = 0) -> None:
    _check(h, _lib.gs_prefill(h, slot, vis_ptr or None, n_vis, text_ptr or None, n_text, max_new,
                              x0_ptr or None))


def gs_round(h, slots_ptr: int, n_seq: int, K: int, rule: int, force: gs_force | None,
             out_tok_ptr: int, out_cnt_ptr: int, out_done_ptr: int, dbg: gs_debug | None = None):
    _check(h, _lib.gs_round(h, slots_ptr, n_seq, K, rule,
                            ctypes.byref(force) if force is not None else None,
                            out_tok_ptr, out_cnt_ptr, out_done_ptr,
                            ctypes.byref(dbg) if dbg is not None else None))


def gs_set_sampling(h, temperature: float, seed: int) -> None:
    _check(h, _lib.gs_set_sampling(h, temperature, seed))


def gs_diffusion_block(h, slots_ptr: int, n_seq: int, B: int, tau_c: float, out_tok_ptr: int,
                       out_cnt_ptr: int, out_done_ptr: int, out_steps_ptr: int = 0) -> None:
    _check(h, _lib.gs_diffusion_block(h, slots_ptr, n_seq, B, tau_c, out_tok_ptr, out_cnt_ptr,
                                      out_done_ptr, out_steps_ptr or None))


def gs_round_refined(h, slots_ptr: int, n_seq: int, K: int, tau_d: float, force: gs_force | None,
                     out_tok_ptr: int, out_cnt_ptr: int, out_done_ptr: int,
                     out_steps_ptr: int = 0) -> None:
    _check(h, _lib.gs_round_refined(h, slots_ptr, n_seq, K, tau_d,
                                    ctypes.byref(force) if force is not None else None,
                                    out_tok_ptr, out_cnt_ptr, out_done_ptr, out_steps_ptr or None))


def gs_seq_restore(h, slot: int, seq_len: int, x0: int, n_out: int, max_new: int, done: int,
                   rounds: int) -> None:
    _check(h, _lib.gs_seq_restore(h, slot, seq_len, x0, n_out, max_new, done, rounds))


def gs_round_launches(h) -> int:
    return int(_lib.gs_round_launches(h))


def gs_round_profile(h, slots_ptr: int, n_seq: int, K: int, force: gs_force | None,
                     out_tok_ptr: int, out_cnt_ptr: int, out_done_ptr: int,
                     max_launches: int = 4096) -> list[tuple[int, float]]:
    """(kind, device ms) per kernel launch of one eagerly enqueued round."""
    ms = (ctypes.c_float * max_launches)()
    kind = (ctypes.c_int * max_launches)()
    n = ctypes.c_int()
    _check(h, _lib.gs_round_profile(h, slots_ptr, n_seq, K,
                                    ctypes.byref(force) if force is not None else None,
                                    out_tok_ptr, out_cnt_ptr, out_done_ptr, max_launches, ms, kind,
                                    ctypes.byref(n)))
    return [(int(kind[i]), float(ms[i])) for i in range(n.value)]


def gs_seq_state(h, slot: int) -> dict:
    v = [ctypes.c_int() for _ in range(5)]
    _check(h, _lib.gs_seq_state(h, slot, *[ctypes.byref(x) for x in v]))
    return dict(zip(("seq_len", "x0", "n_out", "done", "rounds"), (x.value for x in v)))


def gs_release(h, slot: int) -> None:
    _check(h, _lib.gs_release(h, slot))


def gs_sync_check(h) -> None:
    _check(h, _lib.gs_sync_check(h))


def gs_wait_probe(h, limit_us: int) -> None:
    _check(h, _lib.gs_wait_probe(h, limit_us))


def gs_attention_scratch_bytes(n_seq, W, n_heads, n_kv_heads, max_pages, split_pages) -> int:
    return int(_lib.gs_attention_scratch_bytes(n_seq, W, n_heads, n_kv_heads, max_pages, split_pages))


def gs_attention(mode, q_ptr, kv_ptr, n_pages, pt_ptr, pt_stride, n_ptr, n_seq, W, n_heads,
                 n_kv_heads, out_ptr, scratch_ptr, scratch_bytes, split_pages, stream_ptr) -> None:
    rc = _lib.gs_attention(mode, q_ptr, kv_ptr, n_pages, pt_ptr, pt_stride, n_ptr, n_seq, W,
                           n_heads, n_kv_heads, out_ptr, scratch_ptr, scratch_bytes, split_pages,
                           stream_ptr)
    if rc != GS_OK:
        raise GsError(rc, "gs_attention")


def gs_linear_scratch_bytes(M, N, split_k) -> int:
    return int(_lib.gs_linear_scratch_bytes(M, N, split_k))


def gs_linear(x_ptr, w_ptr, y_ptr, M, N, K, epilogue, split_k, scratch_ptr, scratch_bytes,
              stream_ptr) -> None:
    rc = _lib.gs_linear(x_ptr, w_ptr, y_ptr, M, N, K, epilogue, split_k, scratch_ptr, scratch_bytes,
                        stream_ptr)
    if rc != GS_OK:
        raise GsError(rc, "gs_linear")


NOALLOC_SCRATCH_BYTES = 8 << 20


def gs_linear_noalloc(x_ptr, w_ptr, y_ptr, M, N, K, epilogue, split_k, stream_ptr) -> None:
    """gs_linear with its scratch in the library's fixed device array (no allocation).
    Calls that overlap on the GPU race on that array; the first call on a device
    must come before any stream capture."""
    rc = _lib.gs_linear_noalloc(x_ptr, w_ptr, y_ptr, M, N, K, epilogue, split_k, stream_ptr)
    if rc != GS_OK:
        raise GsError(rc, "gs_linear_noalloc")


def gs_linear_noalloc_status(stream_ptr) -> int:
    """GS_OK or the kernel-side failure code of the last gs_linear_noalloc (synchronises)."""
    return int(_lib.gs_linear_noalloc_status(stream_ptr))
