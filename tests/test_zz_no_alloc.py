"""trie_compile_masks_noalloc against trie_compile_masks, through the C ABI.

The no-alloc entry point is for callers that cannot let the library call
cudaMalloc: an engine that has handed all free device memory to its own pool,
a process held to a fixed device-memory budget, or a loop in which an
allocation's implicit device synchronisation is not allowed. It must return
exactly the mask of trie_compile_masks while every call reuses the same fixed
scratch array, so two different workloads are compiled back to back and each
is compared with the allocating entry point.

This file is collected last; it needs nothing from the other tests and runs
alone as well.
"""
from __future__ import annotations

import ctypes

import numpy as np
import pytest

from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_12574_gb300 import _build
    _build.build()
    return torch.device("cuda:0")


def _noalloc(lib, h, vb, vo, V, out, stream):
    vb = np.ascontiguousarray(vb, np.uint8)
    vo = np.ascontiguousarray(vo, np.int64)
    return lib.trie_compile_masks_noalloc(h.handle, ctypes.c_void_p(vb.ctypes.data),
                                          ctypes.c_void_p(vo.ctypes.data), V,
                                          ctypes.c_void_p(out.data_ptr()),
                                          ctypes.c_void_p(stream.cuda_stream))


def test_noalloc_equals_compile_on_consecutive_calls(cuda):
    import torch
    lib = T.load_library()
    stream = torch.cuda.current_stream(cuda)
    # two calls in a row on different tries and vocabularies (the second one
    # larger, then the first again) sharing the one scratch array
    for cfg in (1, 3, 1):
        w = W.config(cfg)
        h = T.trie_build(w.set_bytes, w.set_offsets)
        ref = T.alloc_mask(h, w.V, cuda)
        T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, ref)
        out = torch.full_like(ref, -1)  # every word must be written
        rc = _noalloc(lib, h, w.vocab_bytes, w.vocab_offsets, w.V, out, stream)
        assert rc == T.TRIE_OK, T.trie_last_error()
        torch.cuda.synchronize()
        assert torch.equal(out, ref), f"workload {w.name}: no-alloc mask differs"


def test_noalloc_back_to_back_without_sync(cuda):
    """Calls queued on one stream with no synchronisation between them: each
    call rewrites the shared host staging buffer only after the previous
    call's copy out of it has completed, so both masks must be right."""
    import torch
    lib = T.load_library()
    stream = torch.cuda.Stream(cuda)
    ws = [W.config(c) for c in (3, 1, 2)]
    hs = [T.trie_build(w.set_bytes, w.set_offsets) for w in ws]
    refs = []
    for w, h in zip(ws, hs):
        ref = T.alloc_mask(h, w.V, cuda)
        T.trie_compile_masks(h, w.vocab_bytes, w.vocab_offsets, w.V, ref)
        refs.append(ref)
    torch.cuda.synchronize()
    outs = [torch.full_like(r, -1) for r in refs]
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        # a long kernel ahead of the first copy keeps the stream busy
        big = torch.empty(1 << 28, dtype=torch.int32, device=cuda)
        big.fill_(7)
        for w, h, out in zip(ws, hs, outs):
            rc = _noalloc(lib, h, w.vocab_bytes, w.vocab_offsets, w.V, out, stream)
            assert rc == T.TRIE_OK, T.trie_last_error()
    stream.synchronize()
    for w, out, ref in zip(ws, outs, refs):
        assert torch.equal(out, ref), f"workload {w.name}: queued no-alloc mask differs"


def test_noalloc_device_built_forest(cuda):
    """A forest built on the device keeps its trie only in device memory; the
    no-alloc compile copies those arrays within the device."""
    import torch
    lib = T.load_library()
    stream = torch.cuda.current_stream(cuda)
    w = W.config(1)
    names = W.unpack(w.set_bytes, w.set_offsets)
    sets = [names[:30], names[30:31] + [b""], names[31:], names[5:60]]
    fb, fo = W.pack([x for s in sets for x in s])
    fi = np.cumsum([0] + [len(s) for s in sets]).astype(np.int32)
    for _ in range(2):  # two calls in a row
        hd = T.trie_build_many_device(fb, fo, fi)
        hh = T.trie_build_many(fb, fo, fi)
        ref = T.alloc_mask(hh, w.V, cuda)
        T.trie_compile_masks(hh, w.vocab_bytes, w.vocab_offsets, w.V, ref)
        out = torch.full_like(ref, -1)
        rc = _noalloc(lib, hd, w.vocab_bytes, w.vocab_offsets, w.V, out, stream)
        assert rc == T.TRIE_OK, T.trie_last_error()
        torch.cuda.synchronize()
        assert hd.num_nodes == hh.num_nodes
        assert torch.equal(out, ref), "no-alloc mask of the device-built forest differs"
        hd.destroy()
        hh.destroy()


def test_noalloc_rejects_oversized_input(cuda):
    import torch
    lib = T.load_library()
    long_string = np.full(6_000_000, ord("a"), np.uint8)      # 6M nodes > 32 MiB of scratch
    h = T.trie_build(long_string, np.array([0, long_string.size], np.int64))
    vb, vo = W.pack([b"a", b""])
    out = torch.zeros(1, dtype=torch.int32, device=cuda)
    rc = _noalloc(lib, h, vb, vo, 2, out, torch.cuda.current_stream(cuda))
    assert rc == T.TRIE_EINVAL
    assert "no-alloc scratch" in T.trie_last_error()
    assert int(out.item()) == 0   # nothing was launched
