"""Python binding of libtriemask.so (C ABI in include/triemask.h).

Argument marshalling only: every step of the trie automaton runs in the
library (host trie builder + sm_103a kernels). Host arrays are numpy arrays;
device buffers are torch CUDA tensors, passed by pointer together with the
current torch stream. There is no fallback: if the library has not been
built, the first call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

TRIE_OK, TRIE_EINVAL, TRIE_ENOMEM, TRIE_ECUDA, TRIE_ESTATE = 0, -1, -2, -3, -4
TRIE_DTYPE_F32, TRIE_DTYPE_BF16 = 0, 1
TRIE_STATE_DEAD, TRIE_STATE_FINISHED = -1, -2

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtriemask.so")
_lock = threading.Lock()
_lib = None

# every symbol include/triemask.h declares: (restype, argtypes)
_P, _I32, _I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
SIGNATURES = {
    "trie_build": (ctypes.c_int, [_P, _P, _I32, _P]),
    "trie_build_many": (ctypes.c_int, [_P, _P, _P, _I32, _P]),
    "trie_build_many_device": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "trie_num_nodes": (_I32, [_P]),
    "trie_root": (_I32, [_P, _I32]),
    "trie_copy_roots": (ctypes.c_int, [_P, _P]),
    "trie_num_sets": (_I32, [_P]),
    "trie_num_chars": (_I64, [_P]),
    "trie_max_depth": (_I32, [_P]),
    "trie_get_csr": (ctypes.c_int, [_P, _P, _P, _P, _P]),
    "trie_compile_masks": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "trie_compile_masks_pairwise": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "trie_compile_masks_noalloc": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "trie_compile_lists": (ctypes.c_int, [_P, _P, _P, _I32, _P]),
    "trie_vocab_create": (ctypes.c_int, [_P, _P, _I32, _P]),
    "trie_vocab_size": (_I32, [_P]),
    "trie_vocab_destroy": (None, [_P]),
    "trie_compile_masks_vocab": (ctypes.c_int, [_P, _P, _P, _P]),
    "trie_compile_lists_vocab": (ctypes.c_int, [_P, _P, _P]),
    "trie_num_valid": (_I64, [_P]),
    "trie_copy_lists": (ctypes.c_int, [_P, _P, _P, _P]),
    "trie_apply_lists": (ctypes.c_int, [_P, _P, ctypes.c_int, _P, _I32, _I32, _P]),
    "trie_advance_apply_lists": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, ctypes.c_int, _I32, _I32, _P]),
    "trie_advance": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "trie_advance_apply": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, ctypes.c_int, _I32, _I32, _P]),
    "trie_apply_mask": (ctypes.c_int, [_P, _P, ctypes.c_int, _P, _I32, _I32, _P]),
    "trie_lazy_init": (ctypes.c_int, [_P, _P, _P, _I32, _I32, _I32]),
    "trie_lazy_apply": (ctypes.c_int, [_P, _P, ctypes.c_int, _P, _I32, _I32, _P]),
    "trie_lazy_advance_apply": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, ctypes.c_int, _I32, _I32, _P]),
    "trie_lazy_rows": (ctypes.c_int, [_P, _P, _I32, _P, _P]),
    "trie_lazy_stats": (ctypes.c_int, [_P, _P, _P]),
    "fmt_build": (ctypes.c_int, [_P, _I32, _P]),
    "fmt_length": (_I32, [_P]),
    "fmt_compile_masks": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "fmt_advance": (ctypes.c_int, [_P, _P, _P, _I32, _P, _P]),
    "fmt_apply_mask": (ctypes.c_int, [_P, _P, ctypes.c_int, _P, _I32, _I32, _P]),
    "fmt_destroy": (ctypes.c_int, [_P]),
    "trie_destroy": (ctypes.c_int, [_P]),
    "trie_destroy_async": (ctypes.c_int, [_P, _P]),
    "trie_last_error": (ctypes.c_char_p, []),
}


class TrieError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"libtriemask error {code}: {msg}")
        self.code = code


def load_library(path: str = LIB_PATH):
    """Load libtriemask.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise RuntimeError(f"{path} is missing: build it with "
                                   "`python -c 'import __graft_entry__ as g; g.build()'`")
            lib = ctypes.CDLL(path)
            for name, (res, args) in SIGNATURES.items():
                f = getattr(lib, name)
                f.restype = res
                f.argtypes = args
            _lib = lib
    return _lib


def trie_last_error() -> str:
    return load_library().trie_last_error().decode(errors="replace")


def _check(rc: int) -> None:
    if rc != TRIE_OK:
        raise TrieError(rc, trie_last_error())


def _host(a, dtype) -> np.ndarray:
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


def _hp(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data) if a.size else None


def _stream(stream, device=None) -> ctypes.c_void_p:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t, dtypes, name: str):
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype not in dtypes:
        raise TypeError(f"{name} must have dtype in {dtypes}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


class Trie:
    """Owns one trie handle (released by trie_destroy or garbage collection)."""

    def __init__(self, handle: ctypes.c_void_p):
        self._lib = load_library()
        self.handle = handle

    @property
    def num_nodes(self) -> int:
        return self._lib.trie_num_nodes(self.handle)

    @property
    def num_sets(self) -> int:
        return self._lib.trie_num_sets(self.handle)

    @property
    def num_chars(self) -> int:
        return self._lib.trie_num_chars(self.handle)

    @property
    def max_depth(self) -> int:
        return self._lib.trie_max_depth(self.handle)

    def root(self, i: int = 0) -> int:
        r = self._lib.trie_root(self.handle, i)
        if r < 0:
            raise IndexError(i)
        return r

    def roots(self) -> np.ndarray:
        out = np.empty(self.num_sets, np.int32)
        _check(self._lib.trie_copy_roots(self.handle, _hp(out)))
        return out

    def csr(self) -> dict[str, np.ndarray]:
        n = self.num_nodes
        out = {"parent": np.empty(n, np.int32), "label": np.empty(n, np.uint8),
               "terminal": np.empty(n, np.uint8), "first_child": np.empty(n, np.int32)}
        _check(self._lib.trie_get_csr(self.handle, *(_hp(out[k]) for k in
                                                     ("parent", "label", "terminal", "first_child"))))
        return out

    def destroy(self) -> None:
        if self.handle:
            self._lib.trie_destroy(self.handle)
            self.handle = None

    def destroy_async(self, stream=None) -> None:
        """Release the handle; its device memory is freed in stream order."""
        import torch
        if self.handle:
            h, self.handle = self.handle, None
            _check(self._lib.trie_destroy_async(h, _stream(stream, torch.cuda.current_device())))

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


class Vocab:
    """Owns one vocabulary handle: the vocabulary packed and uploaded once on
    a device, named by later compiles without comparing its arrays again."""

    def __init__(self, handle: ctypes.c_void_p, device: int):
        self._lib = load_library()
        self.handle = handle
        self.device = device

    @property
    def V(self) -> int:
        return self._lib.trie_vocab_size(self.handle)

    def destroy(self) -> None:
        if self.handle:
            self._lib.trie_vocab_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def trie_vocab_create(vocab_bytes, vocab_offsets, V: int) -> Vocab:
    """Pack and upload the vocabulary on the current CUDA device (host-synchronous)."""
    import torch
    lib = load_library()
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    h = ctypes.c_void_p()
    _check(lib.trie_vocab_create(_hp(vb), _hp(vo), V, ctypes.byref(h)))
    return Vocab(h, torch.cuda.current_device())


def _vocab_handle(v: Vocab):
    if not isinstance(v, Vocab) or not v.handle:
        raise ValueError("expected a live Vocab")
    return v.handle


def mask_words(V: int) -> int:
    return (V + 31) // 32


def trie_build(set_bytes, set_offsets) -> Trie:
    """Byte trie of the K strings set_bytes[set_offsets[i]:set_offsets[i+1]]."""
    lib = load_library()
    b = _host(set_bytes, np.uint8)
    o = _host(set_offsets, np.int64)
    h = ctypes.c_void_p()
    _check(lib.trie_build(_hp(b), _hp(o), len(o) - 1, ctypes.byref(h)))
    return Trie(h)


def trie_build_many(set_bytes, set_offsets, set_index) -> Trie:
    """Forest of M tries; set i owns strings set_index[i]:set_index[i+1]."""
    lib = load_library()
    b = _host(set_bytes, np.uint8)
    o = _host(set_offsets, np.int64)
    si = _host(set_index, np.int32)
    h = ctypes.c_void_p()
    _check(lib.trie_build_many(_hp(b), _hp(o), _hp(si), len(si) - 1, ctypes.byref(h)))
    return Trie(h)


def trie_build_many_device(set_bytes, set_offsets, set_index, stream=None) -> Trie:
    """trie_build_many with the level loop on the current CUDA device (same node layout)."""
    import torch
    lib = load_library()
    b = _host(set_bytes, np.uint8)
    o = _host(set_offsets, np.int64)
    si = _host(set_index, np.int32)
    h = ctypes.c_void_p()
    _check(lib.trie_build_many_device(_hp(b), _hp(o), _hp(si), len(si) - 1,
                                      _stream(stream, torch.cuda.current_device()), ctypes.byref(h)))
    return Trie(h)


def trie_num_nodes(h: Trie) -> int:
    return h.num_nodes


def trie_root(h: Trie, i: int = 0) -> int:
    return h.root(i)


def alloc_mask(h: Trie, V: int, device=None):
    """Uninitialised [num_nodes, ceil(V/32)] int32 device tensor for trie_compile_masks."""
    import torch
    return torch.empty((h.num_nodes, mask_words(V)), dtype=torch.int32,
                       device=device if device is not None else "cuda")


def trie_compile_masks(h: Trie, vocab_bytes, vocab_offsets, V: int, d_mask, stream=None) -> None:
    """Fill d_mask ([num_nodes, ceil(V/32)] int32, CUDA) with every node's valid set."""
    import torch
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    p = _dev(d_mask, (torch.int32,), "d_mask")
    if d_mask.numel() < h.num_nodes * mask_words(V):
        raise ValueError("d_mask is smaller than num_nodes * ceil(V/32) words")
    _check(h._lib.trie_compile_masks(h.handle, _hp(vb), _hp(vo), V, p,
                                     _stream(stream, d_mask.device)))


def trie_compile_masks_vocab(h: Trie, vocab: Vocab, d_mask, stream=None) -> None:
    """trie_compile_masks with the vocabulary of a Vocab handle."""
    import torch
    vh = _vocab_handle(vocab)
    p = _dev(d_mask, (torch.int32,), "d_mask")
    if d_mask.numel() < h.num_nodes * mask_words(vocab.V):
        raise ValueError("d_mask is smaller than num_nodes * ceil(V/32) words")
    _check(h._lib.trie_compile_masks_vocab(h.handle, vh, p, _stream(stream, d_mask.device)))


def trie_compile_masks_pairwise(h: Trie, vocab_bytes, vocab_offsets, V: int, d_mask, stream=None) -> None:
    """The dense mask evaluated pair by pair (one token per lane, a warp ballot per word)."""
    import torch
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    p = _dev(d_mask, (torch.int32,), "d_mask")
    if d_mask.numel() < h.num_nodes * mask_words(V):
        raise ValueError("d_mask is smaller than num_nodes * ceil(V/32) words")
    _check(h._lib.trie_compile_masks_pairwise(h.handle, _hp(vb), _hp(vo), V, p,
                                              _stream(stream, d_mask.device)))


def trie_compile_masks_noalloc(h: Trie, vocab_bytes, vocab_offsets, V: int, d_mask, stream=None) -> None:
    """trie_compile_masks without device allocation (fixed 32 MiB library scratch)."""
    import torch
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    p = _dev(d_mask, (torch.int32,), "d_mask")
    if d_mask.numel() < h.num_nodes * mask_words(V):
        raise ValueError("d_mask is smaller than num_nodes * ceil(V/32) words")
    _check(h._lib.trie_compile_masks_noalloc(h.handle, _hp(vb), _hp(vo), V, p,
                                             _stream(stream, d_mask.device)))


def trie_advance(h: Trie, d_states, d_tokens, d_err=None, stream=None) -> None:
    """states <- delta*(states, bytes(tokens)) in place (int32 CUDA tensors of length B)."""
    import torch
    B = d_states.numel()
    if d_tokens.numel() != B:
        raise ValueError("states and tokens differ in length")
    ps = _dev(d_states, (torch.int32,), "d_states")
    pt = _dev(d_tokens, (torch.int32,), "d_tokens")
    pe = _dev(d_err, (torch.int32,), "d_err") if d_err is not None else None
    _check(h._lib.trie_advance(h.handle, ps, pt, B, pe, _stream(stream, d_states.device)))


def trie_advance_apply(h: Trie, d_states_in, d_tokens, d_states_out, d_logits, d_err=None, stream=None) -> None:
    """states_out <- delta*(states_in, tokens); then mask d_logits ([B, V]) by states_out."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    for t, name in ((d_states_in, "d_states_in"), (d_tokens, "d_tokens"), (d_states_out, "d_states_out")):
        if t.numel() != B:
            raise ValueError(f"{name} must have B entries")
    pe = _dev(d_err, (torch.int32,), "d_err") if d_err is not None else None
    _check(h._lib.trie_advance_apply(h.handle, _dev(d_states_in, (torch.int32,), "d_states_in"),
                                     _dev(d_tokens, (torch.int32,), "d_tokens"),
                                     _dev(d_states_out, (torch.int32,), "d_states_out"), pe,
                                     _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits"), dtype, B, V,
                                     _stream(stream, d_logits.device)))


def trie_apply_mask(h: Trie, d_logits, d_states, stream=None) -> None:
    """-inf into disallowed entries of d_logits ([B, V] fp32 or bf16, CUDA), in place."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    if d_states.numel() != B:
        raise ValueError("d_states must have B entries")
    pl = _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits")
    ps = _dev(d_states, (torch.int32,), "d_states")
    _check(h._lib.trie_apply_mask(h.handle, pl, dtype, ps, B, V, _stream(stream, d_logits.device)))


def trie_compile_lists(h: Trie, vocab_bytes, vocab_offsets, V: int, stream=None, device=None,
                       count: bool = True) -> int | None:
    """Build the handle's sparse valid lists on the GPU (asynchronous on the
    stream). Returns the number of entries, which waits for the build; with
    count=False it returns None and does not wait."""
    import torch
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    _check(h._lib.trie_compile_lists(h.handle, _hp(vb), _hp(vo), V,
                                     _stream(stream, device if device is not None else torch.cuda.current_device())))
    return h._lib.trie_num_valid(h.handle) if count else None


def trie_compile_lists_vocab(h: Trie, vocab: Vocab, stream=None, count: bool = True) -> int | None:
    """trie_compile_lists with the vocabulary of a Vocab handle."""
    vh = _vocab_handle(vocab)
    _check(h._lib.trie_compile_lists_vocab(h.handle, vh, _stream(stream, vocab.device)))
    return h._lib.trie_num_valid(h.handle) if count else None


def trie_num_valid(h: Trie) -> int:
    return h._lib.trie_num_valid(h.handle)


def trie_copy_lists(h: Trie, device=None, stream=None):
    """(offsets int64[N+1], tokens int32[n_valid]) device tensors with the handle's lists."""
    import torch
    n = trie_num_valid(h)
    if n < 0:
        raise TrieError(TRIE_ESTATE, "no valid lists on this handle")
    dev = device if device is not None else "cuda"
    off = torch.empty(h.num_nodes + 1, dtype=torch.int64, device=dev)
    tok = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    _check(h._lib.trie_copy_lists(h.handle, ctypes.c_void_p(off.data_ptr()), ctypes.c_void_p(tok.data_ptr()),
                                  _stream(stream, off.device)))
    return off, tok[:n]


def trie_apply_lists(h: Trie, d_logits, d_states, stream=None) -> None:
    """trie_apply_mask driven by the handle's valid lists."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    if d_states.numel() != B:
        raise ValueError("d_states must have B entries")
    pl = _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits")
    ps = _dev(d_states, (torch.int32,), "d_states")
    _check(h._lib.trie_apply_lists(h.handle, pl, dtype, ps, B, V, _stream(stream, d_logits.device)))


def trie_lazy_init(h: Trie, vocab_bytes, vocab_offsets, V: int, cache_rows: int, max_batch: int) -> None:
    """Set up lazily computed rows with an LRU cache of cache_rows rows (current device)."""
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    _check(h._lib.trie_lazy_init(h.handle, _hp(vb), _hp(vo), V, cache_rows, max_batch))


def _logits_dtype(d_logits) -> int:
    import torch
    if d_logits.dim() != 2:
        raise ValueError("d_logits must be [B, V]")
    dtype = {torch.float32: TRIE_DTYPE_F32, torch.bfloat16: TRIE_DTYPE_BF16}.get(d_logits.dtype)
    if dtype is None:
        raise TypeError("d_logits must be float32 or bfloat16")
    return dtype


def trie_lazy_apply(h: Trie, d_logits, d_states, stream=None) -> None:
    """trie_apply_mask with rows computed on first use and cached."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    if d_states.numel() != B:
        raise ValueError("d_states must have B entries")
    _check(h._lib.trie_lazy_apply(h.handle, _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits"), dtype,
                                  _dev(d_states, (torch.int32,), "d_states"), B, V,
                                  _stream(stream, d_logits.device)))


def trie_lazy_advance_apply(h: Trie, d_states_in, d_tokens, d_states_out, d_logits, d_err=None,
                            stream=None) -> None:
    """states_out <- delta*(states_in, tokens); then mask d_logits by lazily computed rows."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    for t, name in ((d_states_in, "d_states_in"), (d_tokens, "d_tokens"), (d_states_out, "d_states_out")):
        if t.numel() != B:
            raise ValueError(f"{name} must have B entries")
    pe = _dev(d_err, (torch.int32,), "d_err") if d_err is not None else None
    _check(h._lib.trie_lazy_advance_apply(h.handle, _dev(d_states_in, (torch.int32,), "d_states_in"),
                                          _dev(d_tokens, (torch.int32,), "d_tokens"),
                                          _dev(d_states_out, (torch.int32,), "d_states_out"), pe,
                                          _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits"), dtype, B,
                                          V, _stream(stream, d_logits.device)))


def trie_lazy_rows(h: Trie, d_states, V: int, out=None, stream=None):
    """The rows ([B, ceil(V/32)] int32 CUDA tensor) of the states, computed or taken from the cache."""
    import torch
    B = d_states.numel()
    if out is None:
        out = torch.empty((B, mask_words(V)), dtype=torch.int32, device=d_states.device)
    if out.shape != (B, mask_words(V)):
        raise ValueError("out must be [B, ceil(V/32)]")
    _check(h._lib.trie_lazy_rows(h.handle, _dev(d_states, (torch.int32,), "d_states"), B,
                                 _dev(out, (torch.int32,), "out"), _stream(stream, d_states.device)))
    return out


def trie_lazy_stats(h: Trie) -> tuple[int, int]:
    """(hits, misses) of the lazy-row cache since trie_lazy_init."""
    hits, misses = ctypes.c_int64(0), ctypes.c_int64(0)
    _check(h._lib.trie_lazy_stats(h.handle, ctypes.byref(hits), ctypes.byref(misses)))
    return hits.value, misses.value


def trie_advance_apply_lists(h: Trie, d_states_in, d_tokens, d_states_out, d_logits, d_err=None,
                             stream=None) -> None:
    """states_out <- delta*(states_in, tokens); then mask d_logits ([B, V]) by the lists of states_out."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    for t, name in ((d_states_in, "d_states_in"), (d_tokens, "d_tokens"), (d_states_out, "d_states_out")):
        if t.numel() != B:
            raise ValueError(f"{name} must have B entries")
    pe = _dev(d_err, (torch.int32,), "d_err") if d_err is not None else None
    _check(h._lib.trie_advance_apply_lists(h.handle, _dev(d_states_in, (torch.int32,), "d_states_in"),
                                           _dev(d_tokens, (torch.int32,), "d_tokens"),
                                           _dev(d_states_out, (torch.int32,), "d_states_out"), pe,
                                           _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits"), dtype, B,
                                           V, _stream(stream, d_logits.device)))


def trie_destroy(h: Trie) -> None:
    h.destroy()


def trie_destroy_async(h: Trie, stream=None) -> None:
    h.destroy_async(stream)


# ------------------------------------------------------------ fixed formats

class Fmt:
    """A fixed format (character-position masks): an owned library handle."""

    def __init__(self, handle: ctypes.c_void_p):
        self.handle = handle
        self._lib = load_library()
        self.L = self._lib.fmt_length(handle)

    def destroy(self) -> None:
        if self.handle:
            self._lib.fmt_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def fmt_build(classes) -> Fmt:
    """classes: uint8 [L, 32] bitmaps (byte c allowed at position i iff bit c % 8 of classes[i, c // 8])."""
    c = np.ascontiguousarray(classes, dtype=np.uint8).reshape(-1, 32)
    h = ctypes.c_void_p()
    lib = load_library()
    _check(lib.fmt_build(_hp(c), c.shape[0], ctypes.byref(h)))
    return Fmt(h)


def fmt_alloc_mask(f: Fmt, V: int, device=None):
    import torch
    return torch.zeros((f.L + 1, mask_words(V)), dtype=torch.int32, device=device if device is not None else "cuda")


def fmt_compile_masks(f: Fmt, vocab_bytes, vocab_offsets, V: int, d_mask, stream=None) -> None:
    import torch
    vb = _host(vocab_bytes, np.uint8)
    vo = _host(vocab_offsets, np.int64)
    if len(vo) != V + 1:
        raise ValueError("vocab_offsets must have V+1 entries")
    p = _dev(d_mask, (torch.int32,), "d_mask")
    if d_mask.numel() < (f.L + 1) * mask_words(V):
        raise ValueError("d_mask is smaller than (L + 1) * ceil(V/32) words")
    _check(f._lib.fmt_compile_masks(f.handle, _hp(vb), _hp(vo), V, p, _stream(stream, d_mask.device)))


def fmt_advance(f: Fmt, d_states, d_tokens, d_err=None, stream=None) -> None:
    """Positions in place by one token each (int32 CUDA tensors of length B)."""
    import torch
    B = d_states.numel()
    if d_tokens.numel() != B:
        raise ValueError("states and tokens differ in length")
    pe = _dev(d_err, (torch.int32,), "d_err") if d_err is not None else None
    _check(f._lib.fmt_advance(f.handle, _dev(d_states, (torch.int32,), "d_states"),
                              _dev(d_tokens, (torch.int32,), "d_tokens"), B, pe, _stream(stream, d_states.device)))


def fmt_apply_mask(f: Fmt, d_logits, d_states, stream=None) -> None:
    """-inf into the logits ([B, V] fp32 or bf16) of tokens not allowed at each position."""
    import torch
    dtype = _logits_dtype(d_logits)
    B, V = d_logits.shape
    if d_states.numel() != B:
        raise ValueError("d_states must have B entries")
    _check(f._lib.fmt_apply_mask(f.handle, _dev(d_logits, (torch.float32, torch.bfloat16), "d_logits"), dtype,
                                 _dev(d_states, (torch.int32,), "d_states"), B, V, _stream(stream, d_logits.device)))

