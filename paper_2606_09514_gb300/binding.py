"""ctypes binding of libbuddy (include/buddy.h).  Argument marshalling only:
every step of the decode path runs in the library's CUDA kernels; PyTorch
provides device memory and streams.  Raises if the library is missing."""
from __future__ import annotations

import ctypes
import os
from typing import Dict, List, Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libbuddy.so")

BUDDY_OK, BUDDY_ERR_ARG, BUDDY_ERR_RANGE, BUDDY_ERR_CUDA, BUDDY_ERR_DEVICE, BUDDY_ERR_STATE = range(6)
BUDDY_DTYPE_F32, BUDDY_DTYPE_BF16 = 0, 1
BUDDY_FEATURE = {"v": 0, "k": 1, "kv": 2}
BUDDY_SKIP = {"zero": 0, "masked": 1}
BUDDY_DEV_BAD_BUDGET, BUDDY_DEV_BAD_POSITION, BUDDY_DEV_BAD_SEQ, BUDDY_DEV_TIMEOUT = 1, 2, 4, 8

EXPORTED = ["buddy_create", "buddy_destroy", "buddy_set_weights", "buddy_kv_append", "buddy_route",
            "buddy_decode_step", "buddy_decode_step_host", "buddy_set_options",
            "buddy_device_status", "buddy_budget_to_k", "buddy_error_string", "buddy_version",
            "buddy_set_profiling", "buddy_profile_read", "buddy_profile_class_name",
            "buddy_route_noalloc", "buddy_set_budget_predictor", "buddy_get_paths", "buddy_prefill",
            "buddy_set_wait_limit"]
PROF_CLASSES = ["check", "rmsnorm", "gemm_qkv", "qkv_finalize", "attention", "gemm_o", "gemm_gate_up",
                "gemm_down", "route", "compact", "other", "gemm_fixup",
                "pf_gemm", "pf_attention", "pf_other"]

c_p = ctypes.c_void_p
c_i32 = ctypes.c_int32


class buddy_config(ctypes.Structure):
    _fields_ = [("n_layers", c_i32), ("d_model", c_i32), ("n_q_heads", c_i32), ("n_kv_heads", c_i32),
                ("head_dim", c_i32), ("ffn_dim", c_i32), ("dm_hidden", c_i32), ("dtype", c_i32),
                ("max_batch", c_i32), ("max_pos", c_i32), ("qkv_bias", c_i32),
                ("feature", c_i32), ("ctx_layer", c_i32), ("skip_kv", c_i32), ("max_prefill_tokens", c_i32),
                ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)]


class buddy_layer_weights(ctypes.Structure):
    _fields_ = [("attn_norm", c_p), ("w_qkv", c_p), ("b_qkv", c_p), ("w_o", c_p), ("ffn_norm", c_p),
                ("w_gate_up", c_p), ("w_down", c_p)]


class buddy_dm_weights(ctypes.Structure):
    _fields_ = [("w1", c_p), ("b1", c_p), ("w2", c_p), ("b2", c_p), ("prior", c_p),
                ("omega", ctypes.c_float)]


class buddy_predictor_weights(ctypes.Structure):
    _fields_ = [("w1", c_p), ("b1", c_p), ("w2", c_p), ("b2", c_p), ("hidden", c_i32)]


class buddy_kv_state(ctypes.Structure):
    _fields_ = [("k_cache", ctypes.POINTER(c_p)), ("v_cache", ctypes.POINTER(c_p)), ("seq_off", c_p),
                ("cap", c_p), ("len", c_p), ("pool_sum", c_p), ("batch", c_i32), ("layer_len", c_p)]


class BuddyError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: libbuddy error {code}")
        self.code = code


_lib = None


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Loads libbuddy.so (built by __graft_entry__.build()); raises if absent."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libbuddy.so not found at {p}: run __graft_entry__.build() first")
    lib = ctypes.CDLL(p)
    lib.buddy_create.argtypes = [ctypes.POINTER(buddy_config), ctypes.POINTER(c_p)]
    lib.buddy_destroy.argtypes = [c_p]
    lib.buddy_destroy.restype = None
    lib.buddy_set_weights.argtypes = [c_p, ctypes.POINTER(buddy_layer_weights), ctypes.POINTER(buddy_dm_weights)]
    lib.buddy_kv_append.argtypes = [c_p, ctypes.POINTER(buddy_kv_state), c_i32, c_i32, c_p, c_i32, c_p, c_p,
                                    c_i32, c_p]
    lib.buddy_route.argtypes = [c_p, ctypes.POINTER(buddy_kv_state), c_i32, c_p, c_p, c_p, c_p, c_p, c_p]
    lib.buddy_decode_step.argtypes = [c_p, ctypes.POINTER(buddy_kv_state), c_i32, c_p, c_p, c_p, c_p, c_p,
                                      c_p, c_p, c_p]
    lib.buddy_decode_step_host.argtypes = [c_p, ctypes.POINTER(buddy_kv_state), c_i32, c_p, c_p, c_p, c_p,
                                           c_p]
    lib.buddy_set_options.argtypes = [c_p, c_i32]
    lib.buddy_device_status.argtypes = [c_p, c_p, ctypes.POINTER(c_i32)]
    lib.buddy_budget_to_k.argtypes = [ctypes.c_float, c_i32]
    lib.buddy_budget_to_k.restype = c_i32
    lib.buddy_error_string.argtypes = [c_i32]
    lib.buddy_error_string.restype = ctypes.c_char_p
    lib.buddy_version.restype = c_i32
    lib.buddy_set_profiling.argtypes = [c_p, c_i32]
    lib.buddy_profile_read.argtypes = [c_p, c_i32, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(c_i32)]
    lib.buddy_profile_class_name.argtypes = [c_i32]
    lib.buddy_profile_class_name.restype = ctypes.c_char_p
    lib.buddy_route_noalloc.argtypes = [c_i32, c_i32, c_i32, c_i32, c_i32, c_i32, ctypes.POINTER(buddy_dm_weights),
                                        c_i32, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p]
    lib.buddy_route_noalloc.restype = ctypes.c_int
    lib.buddy_set_budget_predictor.argtypes = [c_p, ctypes.POINTER(buddy_predictor_weights)]
    lib.buddy_set_budget_predictor.restype = ctypes.c_int
    lib.buddy_get_paths.argtypes = [c_p, ctypes.POINTER(c_i32), c_i32]
    lib.buddy_get_paths.restype = ctypes.c_int
    lib.buddy_prefill.argtypes = [c_p, ctypes.POINTER(buddy_kv_state), c_i32, ctypes.POINTER(c_i32), c_p, c_p, c_p,
                                  c_p, c_p, c_p]
    lib.buddy_prefill.restype = ctypes.c_int
    lib.buddy_set_wait_limit.argtypes = [c_p, ctypes.c_int64]
    lib.buddy_set_wait_limit.restype = ctypes.c_int
    for name in ("buddy_create", "buddy_set_weights", "buddy_kv_append", "buddy_route", "buddy_decode_step",
                 "buddy_decode_step_host", "buddy_set_options", "buddy_device_status", "buddy_set_profiling",
                 "buddy_profile_read"):
        getattr(lib, name).restype = ctypes.c_int
    if path is None:
        _lib = lib
    return lib


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(rc: int, what: str):
    if rc != BUDDY_OK:
        raise BuddyError(rc, what)


def buddy_budget_to_k(b: float, n_layers: int) -> int:
    return int(load_library().buddy_budget_to_k(float(b), int(n_layers)))


def buddy_route_noalloc(shape, dm: Dict[str, torch.Tensor], pool_sum: torch.Tensor, length: torch.Tensor,
                        h1: torch.Tensor, k: torch.Tensor, sel_out=None, mask_out=None, scores_out=None,
                        flags_out=None, prior: Optional[torch.Tensor] = None, omega: float = 0.0,
                        stream=None):
    """Context-free router (no device allocation); see include/buddy.h."""
    lib = load_library()
    dmw = buddy_dm_weights(dm["w1"].data_ptr(), dm["b1"].data_ptr(), dm["w2"].data_ptr(), dm["b2"].data_ptr(),
                           None if prior is None else prior.data_ptr(), float(omega))
    _check(lib.buddy_route_noalloc(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads,
                                   shape.head_dim, shape.dm_hidden, ctypes.byref(dmw), h1.shape[0],
                                   _ptr(pool_sum), _ptr(length), _ptr(h1), _ptr(k), _ptr(sel_out),
                                   _ptr(mask_out), _ptr(scores_out), _ptr(flags_out), _stream(stream)),
           "buddy_route_noalloc")


class KVCache:
    """Per-layer K/V caches in the library's layout (head-major block of cap_i
    positions per sequence), positions len_i and the pooled first-layer sums."""

    def __init__(self, n_layers: int, n_kv: int, head_dim: int, caps: Sequence[int], dtype, device,
                 masked: bool = False):
        caps = [int(c) for c in caps]
        self.batch = len(caps)
        self.n_kv, self.head_dim = n_kv, head_dim
        off, o = [], 0
        for c in caps:
            off.append(o)
            o += c
        self.total_pos = o
        n_el = o * n_kv * head_dim
        self.k = [torch.zeros(n_el, dtype=dtype, device=device) for _ in range(n_layers)]
        self.v = [torch.zeros(n_el, dtype=dtype, device=device) for _ in range(n_layers)]
        self.seq_off = torch.tensor(off, dtype=torch.int64, device=device)
        self.cap = torch.tensor(caps, dtype=torch.int32, device=device)
        self.len = torch.zeros(self.batch, dtype=torch.int32, device=device)
        self.pool_sum = torch.zeros(self.batch, n_kv * head_dim, dtype=torch.float32, device=device)
        # masked skip variant: positions each layer holds
        self.layer_len = (torch.zeros(n_layers, self.batch, dtype=torch.int32, device=device) if masked
                          else None)
        self._caps = caps
        self._off = off
        self._kp = (c_p * n_layers)(*[t.data_ptr() for t in self.k])
        self._vp = (c_p * n_layers)(*[t.data_ptr() for t in self.v])
        self.state = buddy_kv_state(self._kp, self._vp, self.seq_off.data_ptr(), self.cap.data_ptr(),
                                    self.len.data_ptr(), self.pool_sum.data_ptr(), self.batch,
                                    None if self.layer_len is None else self.layer_len.data_ptr())

    def view(self, which: str, layer: int, seq: int) -> torch.Tensor:
        """[n_kv, cap_i, hd] view of one sequence's block."""
        buf = (self.k if which == "k" else self.v)[layer]
        n = self._caps[seq] * self.n_kv * self.head_dim
        s = self._off[seq] * self.n_kv * self.head_dim
        return buf[s:s + n].view(self.n_kv, self._caps[seq], self.head_dim)


def pack_layer(w: Dict[str, torch.Tensor]) -> Dict[str, torch.Tensor]:
    """Fused layouts the library takes: W_qkv = [W_q; W_k; W_v], W_gate_up = [W_gate; W_up]."""
    out = {"attn_norm": w["attn_norm"].contiguous(), "ffn_norm": w["ffn_norm"].contiguous(),
           "w_qkv": torch.cat([w["w_q"], w["w_k"], w["w_v"]], 0).contiguous(),
           "w_o": w["w_o"].contiguous(),
           "w_gate_up": torch.cat([w["w_gate"], w["w_up"]], 0).contiguous(),
           "w_down": w["w_down"].contiguous()}
    if w.get("b_q") is not None:
        out["b_qkv"] = torch.cat([w["b_q"], w["b_k"], w["b_v"]], 0).contiguous()
    return out


class Context:
    """Owns a buddy_ctx handle; keeps the registered weight tensors alive."""

    def __init__(self, *, n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn_dim, dm_hidden, dtype,
                 max_batch, max_pos, qkv_bias, rms_eps, rope_theta, feature="v", ctx_layer=0, skip_kv="zero",
                 max_prefill_tokens=0):
        self.lib = load_library()
        cfg = buddy_config(n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn_dim, dm_hidden,
                           BUDDY_DTYPE_BF16 if dtype == "bf16" else BUDDY_DTYPE_F32, max_batch, max_pos,
                           1 if qkv_bias else 0, BUDDY_FEATURE[feature], int(ctx_layer), BUDDY_SKIP[skip_kv],
                           int(max_prefill_tokens), rms_eps, rope_theta)
        h = c_p()
        _check(self.lib.buddy_create(ctypes.byref(cfg), ctypes.byref(h)), "buddy_create")
        self.handle = h
        self.cfg = cfg
        self._keep: List = []

    @classmethod
    def for_shape(cls, shape, max_batch: int, max_pos: int, max_prefill_tokens: int = 0) -> "Context":
        return cls(n_layers=shape.n_layers, d_model=shape.d_model, n_q_heads=shape.n_q_heads,
                   n_kv_heads=shape.n_kv_heads, head_dim=shape.head_dim, ffn_dim=shape.ffn_dim,
                   dm_hidden=shape.dm_hidden, dtype=shape.dtype, max_batch=max_batch, max_pos=max_pos,
                   qkv_bias=shape.qkv_bias, rms_eps=shape.rms_eps, rope_theta=shape.rope_theta,
                   feature=shape.feature, ctx_layer=shape.ctx_layer, skip_kv=shape.skip_kv,
                   max_prefill_tokens=max_prefill_tokens)

    def close(self):
        if self.handle is not None and self.handle.value:
            self.lib.buddy_destroy(self.handle)
        self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def buddy_set_weights(self, layers: List[Dict[str, torch.Tensor]], dm: Dict[str, torch.Tensor],
                          prior: Optional[torch.Tensor] = None, omega: float = 0.0):
        n = len(layers)
        arr = (buddy_layer_weights * n)()
        for l, w in enumerate(layers):
            arr[l] = buddy_layer_weights(w["attn_norm"].data_ptr(), w["w_qkv"].data_ptr(),
                                         w["b_qkv"].data_ptr() if w.get("b_qkv") is not None else None,
                                         w["w_o"].data_ptr(), w["ffn_norm"].data_ptr(),
                                         w["w_gate_up"].data_ptr(), w["w_down"].data_ptr())
        dmw = buddy_dm_weights(dm["w1"].data_ptr(), dm["b1"].data_ptr(), dm["w2"].data_ptr(),
                               dm["b2"].data_ptr(), None if prior is None else prior.data_ptr(), float(omega))
        _check(self.lib.buddy_set_weights(self.handle, arr, ctypes.byref(dmw)), "buddy_set_weights")
        self._keep = [layers, dm, prior]

    def buddy_set_budget_predictor(self, pw: Optional[Dict[str, torch.Tensor]]):
        """Registers the Budget Predictor ({"w1", "b1", "w2", "b2"}), or removes it (None)."""
        if pw is None:
            _check(self.lib.buddy_set_budget_predictor(self.handle, None), "buddy_set_budget_predictor")
            return
        bp = buddy_predictor_weights(pw["w1"].data_ptr(), pw["b1"].data_ptr(), pw["w2"].data_ptr(),
                                     pw["b2"].data_ptr(), int(pw["w1"].shape[0]))
        _check(self.lib.buddy_set_budget_predictor(self.handle, ctypes.byref(bp)), "buddy_set_budget_predictor")
        self._pred = pw

    def buddy_get_paths(self) -> Dict[str, str]:
        """Which kernels this context runs (see include/buddy.h)."""
        v = (c_i32 * 4)()
        _check(self.lib.buddy_get_paths(self.handle, v, 4), "buddy_get_paths")
        return {"gemm": "tcgen05 bf16 (TMA, TMEM)" if v[0] else "CUDA-core fp32",
                "attention": ["CUDA-core", "mma.sync tensor-core, warp shares over the GPU (in-kernel span merge)",
                              "mma.sync tensor-core, one cluster per stream (DSMEM merge)"][v[1]],
                "rmsnorm": "inside the QKV and gate/up GEMMs" if v[2] else "separate kernel",
                "split_k_fixup": "separate kernel" if v[3] else "last-arriving CTA"}

    def buddy_set_wait_limit(self, ns: int):
        _check(self.lib.buddy_set_wait_limit(self.handle, int(ns)), "buddy_set_wait_limit")

    def buddy_set_options(self, use_graph: bool):
        _check(self.lib.buddy_set_options(self.handle, 1 if use_graph else 0), "buddy_set_options")

    def buddy_kv_append(self, kv: KVCache, layer: int, seq_ids: torch.Tensor, k_new: torch.Tensor,
                        v_new: torch.Tensor, advance: bool, stream=None):
        n_seq = seq_ids.numel()
        n_new = k_new.shape[1] if k_new.numel() else 0
        _check(self.lib.buddy_kv_append(self.handle, ctypes.byref(kv.state), layer, n_seq, _ptr(seq_ids),
                                        n_new, _ptr(k_new), _ptr(v_new), 1 if advance else 0,
                                        _stream(stream)), "buddy_kv_append")

    def buddy_route(self, kv: KVCache, h1: torch.Tensor, k: torch.Tensor, sel_out=None, mask_out=None,
                    scores_out=None, stream=None):
        _check(self.lib.buddy_route(self.handle, ctypes.byref(kv.state), h1.shape[0], _ptr(h1), _ptr(k),
                                    _ptr(sel_out), _ptr(mask_out), _ptr(scores_out), _stream(stream)),
               "buddy_route")

    def buddy_decode_step(self, kv: KVCache, h_in: torch.Tensor, k: torch.Tensor, h_out: torch.Tensor,
                          mask_out=None, rows_out=None, count_out=None, scores_out=None, stream=None):
        _check(self.lib.buddy_decode_step(self.handle, ctypes.byref(kv.state), h_in.shape[0], _ptr(h_in),
                                          _ptr(k), _ptr(h_out), _ptr(mask_out), _ptr(rows_out),
                                          _ptr(count_out), _ptr(scores_out), _stream(stream)),
               "buddy_decode_step")

    def buddy_prefill(self, kv: KVCache, n_tok: Sequence[int], x: torch.Tensor, k: torch.Tensor,
                      h_out: torch.Tensor, mask_out=None, scores_out=None, stream=None):
        """Routed prefill: x / h_out [sum(n_tok), d] fp32 device, n_tok host lengths."""
        nt = (c_i32 * len(n_tok))(*[int(v) for v in n_tok])
        _check(self.lib.buddy_prefill(self.handle, ctypes.byref(kv.state), len(n_tok), nt, _ptr(x), _ptr(k),
                                      _ptr(h_out), _ptr(mask_out), _ptr(scores_out), _stream(stream)),
               "buddy_prefill")

    def buddy_decode_step_host(self, kv: KVCache, h_in_host: torch.Tensor, k_host: torch.Tensor,
                               h_out_host: torch.Tensor, mask_host=None, stream=None):
        _check(self.lib.buddy_decode_step_host(self.handle, ctypes.byref(kv.state), h_in_host.shape[0],
                                               _ptr(h_in_host), _ptr(k_host), _ptr(h_out_host),
                                               _ptr(mask_host), _stream(stream)), "buddy_decode_step_host")

    def buddy_set_profiling(self, on: bool):
        _check(self.lib.buddy_set_profiling(self.handle, 1 if on else 0), "buddy_set_profiling")

    def buddy_profile_read(self) -> Dict[str, tuple]:
        """{class name: (milliseconds, launches)} since the last read."""
        n = len(PROF_CLASSES)
        ms = (ctypes.c_float * n)()
        la = (c_i32 * n)()
        _check(self.lib.buddy_profile_read(self.handle, n, ms, la), "buddy_profile_read")
        return {PROF_CLASSES[i]: (float(ms[i]), int(la[i])) for i in range(n)}

    def buddy_device_status(self, stream=None) -> int:
        flags = c_i32(0)
        rc = self.lib.buddy_device_status(self.handle, _stream(stream), ctypes.byref(flags))
        if rc not in (BUDDY_OK, BUDDY_ERR_DEVICE):
            _check(rc, "buddy_device_status")
        return int(flags.value)
