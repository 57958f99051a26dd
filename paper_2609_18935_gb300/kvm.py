"""Thin Python binding of libkvm (include/kvm.h).

Argument marshalling only: every step of the maintenance path runs in the
library's CUDA kernels.  Tensors are torch CUDA tensors (device memory and
streams come from PyTorch); host-side index arrays are numpy int32/int64.
The binding has no fallback: if libkvm.so has not been built, loading it
raises immediately.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.environ.get("KVM_LIB", os.path.join(_PKG, "_build", "libkvm.so"))

KVM_OK, KVM_E_INVAL, KVM_E_SPAN, KVM_E_CAPACITY, KVM_E_CUDA, KVM_E_DEVICE, KVM_E_UNSUPPORTED = range(7)
LAYER_GDN, LAYER_ATTN = 0, 1
PLAN_GDN_FUSED, PLAN_GDN_STATE_CHAIN = 0, 1

_ERRNAMES = {1: "KVM_E_INVAL", 2: "KVM_E_SPAN", 3: "KVM_E_CAPACITY", 4: "KVM_E_CUDA",
             5: "KVM_E_DEVICE", 6: "KVM_E_UNSUPPORTED"}


class KvmError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{_ERRNAMES.get(code, code)}: {msg}")
        self.code = code


class ModelDesc(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("layer_kind", C.POINTER(C.c_int32)),
                ("n_q_heads", C.c_int32), ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32),
                ("rotary_dim", C.c_int32), ("rope_theta", C.c_double), ("n_gdn_heads", C.c_int32),
                ("d_k", C.c_int32), ("d_v", C.c_int32), ("conv_kernel", C.c_int32)]


class Round(C.Structure):
    _fields_ = [("span_cu", C.POINTER(C.c_int32)), ("span_begin", C.POINTER(C.c_int32)),
                ("span_end", C.POINTER(C.c_int32)), ("tail_cu", C.POINTER(C.c_int32)),
                ("q", C.POINTER(C.c_void_p)), ("k", C.POINTER(C.c_void_p)), ("v", C.POINTER(C.c_void_p)),
                ("alpha", C.POINTER(C.c_void_p)), ("beta", C.POINTER(C.c_void_p)),
                ("out", C.POINTER(C.c_void_p)), ("io_on_host", C.c_int32),
                ("gather_out", C.c_void_p), ("tail_pos", C.POINTER(C.c_int32)),
                ("delim_cu", C.POINTER(C.c_int32)), ("delim_begin", C.POINTER(C.c_int32)),
                ("delim_end", C.POINTER(C.c_int32))]


# name -> (restype, argtypes)
_SIGS = {
    "kvm_create": (C.c_int, [C.POINTER(ModelDesc), C.c_int32, C.POINTER(C.c_int32), C.c_int32,
                             C.POINTER(C.c_void_p)]),
    "kvm_destroy": (C.c_int, [C.c_void_p]),
    "kvm_last_error": (C.c_char_p, []),
    "kvm_load_prefix": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_int64, C.POINTER(C.c_int32),
                                  C.c_void_p]),
    "kvm_set_kv": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p]),
    "kvm_get_kv": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p]),
    "kvm_get_positions": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_set_state": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_get_state": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_set_conv_weights": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_get_conv_state": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_set_conv_state": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_get_live": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int32), C.POINTER(C.c_int64)]),
    "kvm_spans_from_positions": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.POINTER(C.c_int64),
                                           C.POINTER(C.c_int64), C.POINTER(C.c_int32),
                                           C.POINTER(C.c_int32)]),
    "kvm_kv_compact": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                 C.POINTER(C.c_int32), C.c_void_p, C.c_void_p]),
    "kvm_tail_attn_prefill": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int32), C.c_void_p,
                                        C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "kvm_gdn_chunk_scan_from_state": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int32), C.c_void_p,
                                                C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                                C.c_void_p, C.c_void_p]),
    "kvm_advance": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32)]),
    "kvm_tail_attn_prefill_at": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                           C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "kvm_advance_at": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "kvm_rerotate_keys": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.POINTER(C.c_int32),
                                    C.c_void_p]),
    "kvm_update_round": (C.c_int, [C.c_void_p, C.POINTER(Round), C.c_void_p]),
    "kvm_check": (C.c_int, [C.c_void_p, C.c_void_p]),
    "kvm_launch_count": (C.c_int64, [C.c_void_p]),
    "kvm_fork": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "kvm_plan_removal": (C.c_int, [C.c_int32, C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                   C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "kvm_plan_spans_from_positions": (C.c_int, [C.c_int32, C.POINTER(C.c_int32), C.c_int32, C.POINTER(C.c_int64),
                                                C.POINTER(C.c_int64), C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "kvm_plan_attention": (C.c_int, [C.c_int32, C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.c_int32, C.c_int32,
                                     C.c_int32, C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                     C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "kvm_plan_partition": (C.c_int, [C.c_int32, C.POINTER(C.c_int64), C.c_int32, C.POINTER(C.c_int32),
                                     C.POINTER(C.c_int64)]),
    "kvm_kv_compact_noalloc": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int64, C.c_int32,
                                         C.c_int32, C.c_int32, C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                         C.POINTER(C.c_int32), C.c_void_p]),
    "kvm_kv_compact_noalloc_check": (C.c_int, [C.c_void_p]),
    "kvm_debug_compact_wait": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32]),
    "kvm_debug_poke_canary": (C.c_int, [C.c_void_p]),
    "kvm_set_plan": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32]),
    "kvm_attn_probe": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                 C.c_int32, C.c_void_p, C.c_void_p]),
    "kvm_effective_group_count": (C.c_int, [C.c_int32, C.POINTER(C.c_double), C.POINTER(C.c_double)]),
    "kvm_total_variation": (C.c_int, [C.c_int32, C.POINTER(C.c_double), C.POINTER(C.c_double),
                                      C.POINTER(C.c_double)]),
    "kvm_profile_enable": (C.c_int, [C.c_void_p, C.c_int32]),
    "kvm_profile_read": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int64), C.POINTER(C.c_double),
                                   C.c_int32]),
}

# kernel families of kvm_profile_read
K_COMPACT, K_ROPE_APPEND, K_ATTENTION, K_ATTN_COMBINE, K_GDN, K_GATHER, K_GDN_PREP, K_GDN_CONV = range(8)
KERNEL_NAMES = ["kv_compact", "rope_append", "tail_attention", "attn_combine", "gdn_chunk_scan", "gather_map",
                "gdn_chunk_prep", "gdn_conv"]

_lib = None


def load_library(path: str | None = None):
    """Load libkvm.so once; raises OSError if it is missing (no fallback)."""
    global _lib
    if _lib is None:
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise OSError(f"libkvm.so not found at {p}; build it with "
                          "`python -m paper_2609_18935_gb300.build_lib`")
        lib = C.CDLL(p)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _check(status: int):
    if status != KVM_OK:
        raise KvmError(status, _lib.kvm_last_error().decode())


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _p32(a: np.ndarray):
    return a.ctypes.data_as(C.POINTER(C.c_int32))


def _dptr(t, dtype=None) -> int:
    """Device address of a contiguous torch CUDA tensor (0 for None)."""
    if t is None:
        return 0
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"expected {dtype}, got {t.dtype}")
    return t.data_ptr()


def _stream(stream) -> int:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def kv_compact_noalloc(K, V, positions, live, span_begin, span_end, stream=None) -> int:
    """kvm_kv_compact_noalloc on caller-owned buffers (no allocation anywhere).

    K, V: CUDA bf16 tensors [n_slabs][slab_rows][head_dim]; positions: CUDA
    int32 [slab_rows] or None.  Returns the new live length."""
    import torch
    load_library()
    if K.dim() != 3:
        raise ValueError("K must be [n_slabs][slab_rows][head_dim]")
    n_slabs, rows, D = K.shape
    if tuple(V.shape) != tuple(K.shape):
        raise ValueError(f"V has shape {tuple(V.shape)}, K has {tuple(K.shape)}")
    dev = torch.cuda.current_device()
    for name, t in (("K", K), ("V", V), ("positions", positions)):
        if t is not None and (not t.is_cuda or t.device.index != dev):
            raise ValueError(f"{name} must live on the current CUDA device (cuda:{dev})")
    if positions is not None and positions.numel() < rows:
        raise ValueError(f"positions holds {positions.numel()} entries, need >= slab_rows = {rows}")
    sb, se = _i32(span_begin), _i32(span_end)
    if len(sb) != len(se):
        raise ValueError("span_begin and span_end differ in length")
    new_live = C.c_int32()
    _check(_lib.kvm_kv_compact_noalloc(_dptr(K, torch.bfloat16), _dptr(V, torch.bfloat16),
                                       _dptr(positions, torch.int32), n_slabs, rows, D, int(live), len(sb),
                                       _p32(sb), _p32(se), C.byref(new_live), _stream(stream)))
    return new_live.value


def kv_compact_noalloc_check(stream=None):
    """kvm_kv_compact_noalloc_check: raise KvmError (KVM_E_DEVICE) if an
    allocation-free compaction on the current device reported a failure
    since the last check (the check clears it)."""
    load_library()
    _check(_lib.kvm_kv_compact_noalloc_check(_stream(stream)))


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def effective_group_count(mass) -> float:
    """kvm_effective_group_count: exp(entropy) of the normalised group masses."""
    load_library()
    m = _f64(mass)
    out = C.c_double()
    _check(_lib.kvm_effective_group_count(len(m), m.ctypes.data_as(C.POINTER(C.c_double)), C.byref(out)))
    return out.value


def total_variation(p, q) -> float:
    """kvm_total_variation: 0.5 * sum |p - q| over matched entries."""
    load_library()
    a, b = _f64(p), _f64(q)
    if a.shape != b.shape:
        raise ValueError("p and q differ in length")
    out = C.c_double()
    _check(_lib.kvm_total_variation(len(a), a.ctypes.data_as(C.POINTER(C.c_double)),
                                    b.ctypes.data_as(C.POINTER(C.c_double)), C.byref(out)))
    return out.value


def plan_removal(live, span_cu, span_begin, span_end):
    """kvm_plan_removal: (new live lengths, first moved index) per character;
    raises KvmError with the library's status on invalid spans."""
    load_library()
    L = _i32(live)
    cu, sb, se = _i32(span_cu), _i32(span_begin), _i32(span_end)
    new_live, first = np.zeros(len(L), np.int32), np.zeros(len(L), np.int32)
    _check(_lib.kvm_plan_removal(len(L), _p32(L), _p32(cu), _p32(sb) if len(sb) else None,
                                 _p32(se) if len(se) else None, _p32(new_live), _p32(first)))
    return new_live, first


def plan_spans_from_positions(positions, pos_begin, pos_end):
    """kvm_plan_spans_from_positions: live-index spans (begin, end) of the
    position ranges [pos_begin, pos_end) over one character's live positions."""
    load_library()
    P = _i32(positions)
    pb = np.ascontiguousarray(np.asarray(pos_begin, dtype=np.int64))
    pe = np.ascontiguousarray(np.asarray(pos_end, dtype=np.int64))
    sb, se = np.zeros(len(pb), np.int32), np.zeros(len(pb), np.int32)
    p64 = lambda a: a.ctypes.data_as(C.POINTER(C.c_int64))
    _check(_lib.kvm_plan_spans_from_positions(len(P), _p32(P) if len(P) else None, len(pb), p64(pb), p64(pe),
                                              _p32(sb), _p32(se)))
    return sb, se


def plan_attention(live, tail_cu, n_q_heads, n_kv_heads, max_blocks):
    """kvm_plan_attention: the attention's work partition for one layer."""
    load_library()
    L, cu = _i32(live), _i32(tail_cu)
    tile, key = np.zeros(max_blocks + 1, np.int32), np.zeros(max_blocks + 1, np.int32)
    split = np.zeros(max_blocks, np.int32)
    nb, nt, ns = C.c_int32(), C.c_int32(), C.c_int32()
    _check(_lib.kvm_plan_attention(len(L), _p32(L), _p32(cu), int(n_q_heads), int(n_kv_heads), int(max_blocks),
                                   C.byref(nb), C.byref(nt), _p32(tile), _p32(key), C.byref(ns), _p32(split)))
    n = nb.value
    return {"n_blocks": n, "n_tiles": nt.value, "block_tile": tile[:n + 1].copy(), "block_key": key[:n + 1].copy(),
            "split_first_block": split[:ns.value].copy()}


def round_cost(live_after_removal, tails):
    """Per-character cost of a round's attention, M_b (L'_b + (M_b + 1) / 2),
    in units of query-key pairs (the partitioner's balance target)."""
    return [int(m) * int(l) + int(m) * (int(m) + 1) // 2 for l, m in zip(live_after_removal, tails)]


def plan_partition(cost, n_ranks):
    """kvm_plan_partition: (rank of each character, summed cost per rank)."""
    load_library()
    c = np.ascontiguousarray(np.asarray(cost, dtype=np.int64))
    rank_of = np.zeros(len(c), np.int32)
    loads = np.zeros(int(n_ranks), np.int64)
    p64 = lambda a: a.ctypes.data_as(C.POINTER(C.c_int64))
    _check(_lib.kvm_plan_partition(len(c), p64(c) if len(c) else None, int(n_ranks),
                                   _p32(rank_of) if len(c) else None, p64(loads)))
    return rank_of, loads


def pinned_layer_inputs(inputs):
    """Copy per-layer inputs into one pinned host arena per layer.

    inputs[layer] = dict(q, k, v[, alpha, beta]) (CPU or CUDA tensors).
    Returns the same structure with views into a pinned arena per layer,
    laid out q, k, v, alpha, beta back to back (each piece padded to 16
    bytes), which lets a host-resident update_round move a layer's inputs in
    one copy."""
    import torch
    out = {}
    for layer, x in inputs.items():
        keys = [k for k in ("q", "k", "v", "alpha", "beta") if x.get(k) is not None]
        sizes = [x[k].numel() * x[k].element_size() for k in keys]
        padded = [(n + 15) // 16 * 16 for n in sizes]
        arena = torch.empty(sum(padded), dtype=torch.uint8).pin_memory()
        views, off = {}, 0
        for k, n, pn in zip(keys, sizes, padded):
            t = x[k]
            v = arena[off:off + n].view(t.dtype).view(t.shape)
            v.copy_(t.cpu())
            views[k] = v
            off += pn
        out[layer] = views
    return out


class Context:
    """A population of character states on the current CUDA device (kvm_create)."""

    def __init__(self, layer_kind, n_q_heads, n_kv_heads, head_dim, rotary_dim, rope_theta,
                 n_gdn_heads, d_k, d_v, capacity, max_tail_tokens, conv_kernel=0):
        lib = load_library()
        self.layer_kind = [int(x) for x in layer_kind]
        self._kinds = _i32(self.layer_kind)
        self.desc = ModelDesc(len(self.layer_kind), _p32(self._kinds), n_q_heads, n_kv_heads, head_dim,
                              rotary_dim, float(rope_theta), n_gdn_heads, d_k, d_v, int(conv_kernel))
        self.conv_kernel = int(conv_kernel)
        self.n_chars = len(capacity)
        self.Hq, self.Hkv, self.D, self.R = n_q_heads, n_kv_heads, head_dim, rotary_dim
        self.H, self.dk, self.dv = n_gdn_heads, d_k, d_v
        caps = _i32(capacity)
        h = C.c_void_p()
        _check(lib.kvm_create(C.byref(self.desc), self.n_chars, _p32(caps), int(max_tail_tokens), C.byref(h)))
        self._h = h

    def destroy(self):
        if self._h:
            _check(_lib.kvm_destroy(self._h))
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass

    # ---------------------------------------------------------------- state
    def load_prefix(self, b, live, cursor, positions, stream=None):
        pos = _i32(positions)
        _check(_lib.kvm_load_prefix(self._h, b, int(live), int(cursor), _p32(pos), _stream(stream)))

    def set_kv(self, layer, b, k, v, stream=None):
        import torch
        _check(_lib.kvm_set_kv(self._h, layer, b, _dptr(k, torch.bfloat16), _dptr(v, torch.bfloat16),
                               _stream(stream)))

    def get_kv(self, layer, b, stream=None):
        import torch
        live, _ = self.get_live(b)
        k = torch.empty((self.Hkv, live, self.D), dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        _check(_lib.kvm_get_kv(self._h, layer, b, _dptr(k), _dptr(v), _stream(stream)))
        return k, v

    def get_positions(self, b, stream=None):
        import torch
        live, _ = self.get_live(b)
        out = torch.empty(live, dtype=torch.int32, device="cuda")
        _check(_lib.kvm_get_positions(self._h, b, _dptr(out), _stream(stream)))
        return out

    def set_state(self, layer, S, stream=None):
        import torch
        _check(_lib.kvm_set_state(self._h, layer, _dptr(S, torch.float32), _stream(stream)))

    def get_state(self, layer, stream=None):
        import torch
        S = torch.empty((self.n_chars, self.H, self.dv, self.dk), dtype=torch.float32, device="cuda")
        _check(_lib.kvm_get_state(self._h, layer, _dptr(S), _stream(stream)))
        return S

    def set_conv_weights(self, layer, w, stream=None):
        """kvm_set_conv_weights: w CUDA fp32 [channels][4]."""
        import torch
        _check(_lib.kvm_set_conv_weights(self._h, layer, _dptr(w, torch.float32), _stream(stream)))

    def get_conv_state(self, layer, stream=None):
        """kvm_get_conv_state: CUDA bf16 [n_chars][3][channels]."""
        import torch
        C_ = self.H * (2 * self.dk + self.dv)
        out = torch.empty((self.n_chars, 3, C_), dtype=torch.bfloat16, device="cuda")
        _check(_lib.kvm_get_conv_state(self._h, layer, _dptr(out), _stream(stream)))
        return out

    def set_conv_state(self, layer, state, stream=None):
        import torch
        _check(_lib.kvm_set_conv_state(self._h, layer, _dptr(state, torch.bfloat16), _stream(stream)))

    def get_live(self, b):
        live, cur = C.c_int32(), C.c_int64()
        _check(_lib.kvm_get_live(self._h, b, C.byref(live), C.byref(cur)))
        return live.value, cur.value

    def spans_from_positions(self, b, pos_begin, pos_end):
        pb = np.ascontiguousarray(pos_begin, dtype=np.int64)
        pe = np.ascontiguousarray(pos_end, dtype=np.int64)
        n = len(pb)
        sb = np.zeros(n, np.int32)
        se = np.zeros(n, np.int32)
        _check(_lib.kvm_spans_from_positions(self._h, b, n, pb.ctypes.data_as(C.POINTER(C.c_int64)),
                                             pe.ctypes.data_as(C.POINTER(C.c_int64)), _p32(sb), _p32(se)))
        return sb, se

    # ---------------------------------------------------------------- hot path
    def kv_compact(self, span_cu, span_begin, span_end, gather_out=None, stream=None):
        import torch
        cu, sb, se = _i32(span_cu), _i32(span_begin), _i32(span_end)
        _check(_lib.kvm_kv_compact(self._h, _p32(cu), _p32(sb), _p32(se), _dptr(gather_out, torch.int32),
                                   _stream(stream)))

    def tail_attn_prefill(self, layer, tail_cu, q, k_new, v_new, out, tail_pos=None, stream=None):
        """kvm_tail_attn_prefill, or kvm_tail_attn_prefill_at when tail_pos
        (host int32 [sum M], one position id per tail token) is given."""
        import torch
        cu = _i32(tail_cu)
        bf = torch.bfloat16
        if tail_pos is None:
            _check(_lib.kvm_tail_attn_prefill(self._h, layer, _p32(cu), _dptr(q, bf), _dptr(k_new, bf),
                                              _dptr(v_new, bf), _dptr(out, bf), _stream(stream)))
        else:
            tp = _i32(tail_pos)
            _check(_lib.kvm_tail_attn_prefill_at(self._h, layer, _p32(cu), _p32(tp), _dptr(q, bf),
                                                 _dptr(k_new, bf), _dptr(v_new, bf), _dptr(out, bf),
                                                 _stream(stream)))

    def rerotate_keys(self, b, live_begin, live_end, new_pos, stream=None):
        """kvm_rerotate_keys: turn the stored keys of live entries
        [live_begin, live_end) of character b to the position ids new_pos."""
        np_ = _i32(new_pos)
        _check(_lib.kvm_rerotate_keys(self._h, int(b), int(live_begin), int(live_end),
                                      _p32(np_) if len(np_) else None, _stream(stream)))

    def gdn_chunk_scan_from_state(self, layer, tail_cu, q, k, v, alpha, beta, out, stream=None):
        import torch
        cu = _i32(tail_cu)
        bf, f = torch.bfloat16, torch.float32
        _check(_lib.kvm_gdn_chunk_scan_from_state(self._h, layer, _p32(cu), _dptr(q, bf), _dptr(k, bf),
                                                  _dptr(v, bf), _dptr(alpha, f), _dptr(beta, f),
                                                  _dptr(out, bf), _stream(stream)))

    def advance(self, tail_cu, tail_pos=None):
        cu = _i32(tail_cu)
        if tail_pos is None:
            _check(_lib.kvm_advance(self._h, _p32(cu)))
        else:
            tp = _i32(tail_pos)
            _check(_lib.kvm_advance_at(self._h, _p32(cu), _p32(tp)))

    def update_round(self, span_cu, span_begin, span_end, tail_cu, inputs, outputs,
                     io_on_host=False, gather_out=None, stream=None, tail_pos=None, delim=None):
        """One whole round (kvm_update_round).

        inputs[layer] = dict(q, k, v[, alpha, beta]) and outputs[layer] = tensor,
        CUDA tensors (io_on_host=False) or pinned CPU tensors (io_on_host=True).
        tail_pos: optional host int32 [sum M] position ids of the tail tokens.
        delim: optional (delim_cu, delim_begin, delim_end), tail-index ranges
        of maintenance delimiters whose KV leave the caches after the round."""
        n = len(self.layer_kind)
        arr = lambda: (C.c_void_p * n)()
        q, k, v, al, be, out = arr(), arr(), arr(), arr(), arr(), arr()
        ptr = (lambda t: t.data_ptr() if t is not None else 0)
        for l in range(n):
            x = inputs[l]
            q[l], k[l], v[l] = ptr(x["q"]), ptr(x["k"]), ptr(x["v"])
            al[l], be[l] = ptr(x.get("alpha")), ptr(x.get("beta"))
            out[l] = ptr(outputs[l])
        cu, sb, se, tc = _i32(span_cu), _i32(span_begin), _i32(span_end), _i32(tail_cu)
        tp = _i32(tail_pos) if tail_pos is not None else None
        dl = tuple(_i32(x) for x in delim) if delim is not None else None
        r = Round(_p32(cu), _p32(sb), _p32(se), _p32(tc), q, k, v, al, be, out, int(bool(io_on_host)),
                  ptr(gather_out), _p32(tp) if tp is not None else None,
                  *((_p32(dl[0]), _p32(dl[1]), _p32(dl[2])) if dl is not None else (None, None, None)))
        self._keep = (cu, sb, se, tc, q, k, v, al, be, out, tp, dl)
        _check(_lib.kvm_update_round(self._h, C.byref(r), _stream(stream)))

    def attn_probe(self, layer, b, q, group_of=None, n_groups=0, stream=None):
        """kvm_attn_probe: the probe distribution over character b's live
        entries (CUDA fp32 [live]) for the unrotated queries q (CUDA bf16
        [n_q][Hq][D]) of its last n_q live entries, and the per-group mass
        (CUDA fp32 [n_groups]) when group_of (CUDA int32 [live]) is given."""
        import torch
        live, _ = self.get_live(b)
        probs = torch.empty(live, dtype=torch.float32, device="cuda")
        mass = torch.empty(max(1, n_groups), dtype=torch.float32, device="cuda") if group_of is not None else None
        _check(_lib.kvm_attn_probe(self._h, int(layer), int(b), int(q.shape[0]), _dptr(q, torch.bfloat16),
                                   _dptr(probs), _dptr(group_of, torch.int32), int(n_groups), _dptr(mass),
                                   _stream(stream)))
        return probs, mass

    def check(self, stream=None):
        _check(_lib.kvm_check(self._h, _stream(stream)))

    def debug_compact_wait(self, polls=0, stall=False):
        """kvm_debug_compact_wait: compaction wait limit (0 = default) and the
        failure-detection stall (every later compaction block waits on a word
        nothing sets and gives up after `polls` polls)."""
        _check(_lib.kvm_debug_compact_wait(self._h, int(polls), int(bool(stall))))

    def set_gdn_fusion(self, enable=True):
        """kvm_set_plan(KVM_PLAN_GDN_FUSED): prep and chain of a delta-rule
        layer in one launch when it applies, or always separate launches."""
        _check(_lib.kvm_set_plan(self._h, PLAN_GDN_FUSED, int(bool(enable))))

    def set_gdn_state_chain(self, enable=True):
        """kvm_set_plan(KVM_PLAN_GDN_STATE_CHAIN): the chain carries only the
        state and the outputs follow in a parallel pass (d_k = d_v = 128)."""
        _check(_lib.kvm_set_plan(self._h, PLAN_GDN_STATE_CHAIN, int(bool(enable))))

    def debug_poke_canary(self):
        """kvm_debug_poke_canary (debug builds): spoil one canary byte."""
        _check(_lib.kvm_debug_poke_canary(self._h))

    def launch_count(self) -> int:
        return int(_lib.kvm_launch_count(self._h))

    def fork_from(self, src: "Context", stream=None):
        """Overwrite this context's state with a copy of `src` (kvm_fork)."""
        _check(_lib.kvm_fork(self._h, src._h, _stream(stream)))

    def profile_enable(self, enable=True):
        _check(_lib.kvm_profile_enable(self._h, int(bool(enable))))

    def profile_read(self, kernel, reset=False):
        """(launches, total device ms) of one kernel family since the last reset."""
        n, ms = C.c_int64(), C.c_double()
        _check(_lib.kvm_profile_read(self._h, kernel, C.byref(n), C.byref(ms), int(bool(reset))))
        return n.value, ms.value
