"""CPU-only checks of libtriemask: exported symbols, the host trie builder and
argument validation (no device call is made here)."""
from __future__ import annotations

import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W
from pins import prefix_ids, random_case

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "triemask.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_12574_gb300 import _build
    _build.build()
    return T.load_library()


def declared_functions() -> list[str]:
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]+?\b((?:trie|fmt)_\w+)\s*\(", src, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for f in ("trie_build", "trie_compile_masks", "trie_advance", "trie_apply_mask", "trie_destroy",
              "trie_build_many", "trie_last_error"):
        assert f in names


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    for name in names:
        assert hasattr(lib, name), name
        assert name in T.SIGNATURES, f"binding does not declare {name}"
    assert sorted(T.SIGNATURES) == names


def _csr_matches_oracle(strings):
    sb, so = W.pack(strings)
    h = T.trie_build(sb, so)
    ot = oracle.Trie(sb, so)
    c = h.csr()
    assert h.num_nodes == ot.num_nodes
    assert np.array_equal(c["parent"], ot.parent)
    assert np.array_equal(c["label"], ot.label)
    assert np.array_equal(c["terminal"], ot.terminal)
    assert h.num_chars == ot.num_chars
    assert h.max_depth == (int(ot.depth.max()) if ot.num_nodes else 0)
    # first child: smallest id whose parent is the node, -1 for leaves
    fc = np.full(ot.num_nodes, -1, np.int64)
    for c_ in range(ot.num_nodes - 1, 0, -1):
        fc[ot.parent[c_]] = c_
    assert np.array_equal(c["first_child"], fc)
    return h


@pytest.mark.parametrize("seed", range(40))
def test_host_builder_matches_oracle_small(lib, oracle_lib, seed):
    strings, _ = random_case(seed)
    _csr_matches_oracle(strings)


@pytest.mark.parametrize("cfg", [1, 2, 3, 4])
def test_host_builder_matches_oracle_configs(lib, oracle_lib, cfg):
    w = W.config(cfg)
    _csr_matches_oracle(W.unpack(w.set_bytes, w.set_offsets))


def test_host_builder_closed_form_ids(lib):
    strings = [b"get_user", b"get", b"", b"\x00\xff", b"get_user", b"got"]
    sb, so = W.pack(strings)
    h = T.trie_build(sb, so)
    ids, E = prefix_ids(strings)
    c = h.csr()
    inv = {i: p for p, i in ids.items()}
    for i in range(h.num_nodes):
        p = inv[i]
        assert c["terminal"][i] == (p in E)
        if i:
            assert c["label"][i] == p[-1] and c["parent"][i] == ids[p[:-1]]


def test_forest_is_concatenation(lib, oracle_lib):
    sets = [[b"ab", b"ac"], [], [b""], [b"xyz", b"x", b"xy"], [b"ab"]]
    flat = [s for st in sets for s in st]
    index = np.cumsum([0] + [len(s) for s in sets]).astype(np.int32)
    sb, so = W.pack(flat)
    h = T.trie_build_many(sb, so, index)
    assert h.num_sets == len(sets)
    c = h.csr()
    for i, st in enumerate(sets):
        r = h.root(i)
        ot = oracle.Trie(*W.pack(st))
        n = ot.num_nodes
        assert c["parent"][r] == -1
        par = c["parent"][r:r + n].astype(np.int64)
        par[par >= 0] -= r
        assert np.array_equal(par, ot.parent)
        assert np.array_equal(c["label"][r:r + n], ot.label)
        assert np.array_equal(c["terminal"][r:r + n], ot.terminal)
        nxt = h.root(i + 1) if i + 1 < len(sets) else h.num_nodes
        assert nxt - r == n
    with pytest.raises(IndexError):
        h.root(len(sets))


def test_forest_of_config5_prefix(lib, oracle_lib):
    w = W.dynamic_requests(6)
    h = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
    strings = W.unpack(w.set_bytes, w.set_offsets)
    total = 0
    for i in range(6):
        st = strings[w.set_index[i]:w.set_index[i + 1]]
        total += len(prefix_ids(st)[0])
    assert h.num_nodes == total


def _rc(lib, *args):
    return lib.trie_build(*args)


def test_build_argument_errors(lib):
    h = ctypes.c_void_p()
    offs = np.array([0, 3, 2], np.int64)
    b = np.frombuffer(b"abc", np.uint8).copy()
    assert lib.trie_build(b.ctypes.data, offs.ctypes.data, 2, ctypes.byref(h)) == T.TRIE_EINVAL
    assert "non-decreasing" in T.trie_last_error()
    assert lib.trie_build(b.ctypes.data, offs.ctypes.data, -1, ctypes.byref(h)) == T.TRIE_EINVAL
    assert lib.trie_build(b.ctypes.data, offs.ctypes.data, 1, None) == T.TRIE_EINVAL
    assert lib.trie_build(None, None, 1, ctypes.byref(h)) == T.TRIE_EINVAL
    neg = np.array([-1, 2], np.int64)
    assert lib.trie_build(b.ctypes.data, neg.ctypes.data, 1, ctypes.byref(h)) == T.TRIE_EINVAL
    # K = 0: a lone root, offsets may be NULL
    assert lib.trie_build(None, None, 0, ctypes.byref(h)) == T.TRIE_OK
    assert lib.trie_num_nodes(h) == 1
    assert lib.trie_destroy(h) == T.TRIE_OK


def test_build_many_argument_errors(lib):
    h = ctypes.c_void_p()
    b = np.frombuffer(b"abcd", np.uint8).copy()
    offs = np.array([0, 2, 4], np.int64)
    bad_first = np.array([1, 2], np.int32)
    bad_order = np.array([0, 2, 1], np.int32)
    assert lib.trie_build_many(b.ctypes.data, offs.ctypes.data, bad_first.ctypes.data, 1,
                               ctypes.byref(h)) == T.TRIE_EINVAL
    assert lib.trie_build_many(b.ctypes.data, offs.ctypes.data, bad_order.ctypes.data, 2,
                               ctypes.byref(h)) == T.TRIE_EINVAL
    assert lib.trie_build_many(b.ctypes.data, offs.ctypes.data, None, 1, ctypes.byref(h)) == T.TRIE_EINVAL
    ok = np.array([0, 2], np.int32)
    assert lib.trie_build_many(b.ctypes.data, offs.ctypes.data, ok.ctypes.data, 0,
                               ctypes.byref(h)) == T.TRIE_EINVAL


def test_build_many_device_argument_errors(lib):
    """Bad arguments are rejected before any device call (none is made here)."""
    h = ctypes.c_void_p()
    b = np.frombuffer(b"abcd", np.uint8).copy()
    offs = np.array([0, 2, 4], np.int64)
    bad_first = np.array([1, 2], np.int32)
    bad_order = np.array([0, 2, 1], np.int32)
    ok = np.array([0, 2], np.int32)
    f = lib.trie_build_many_device
    assert f(b.ctypes.data, offs.ctypes.data, bad_first.ctypes.data, 1, None, ctypes.byref(h)) == T.TRIE_EINVAL
    assert f(b.ctypes.data, offs.ctypes.data, bad_order.ctypes.data, 2, None, ctypes.byref(h)) == T.TRIE_EINVAL
    assert f(b.ctypes.data, offs.ctypes.data, None, 1, None, ctypes.byref(h)) == T.TRIE_EINVAL
    assert f(b.ctypes.data, offs.ctypes.data, ok.ctypes.data, 0, None, ctypes.byref(h)) == T.TRIE_EINVAL
    assert f(b.ctypes.data, offs.ctypes.data, ok.ctypes.data, 1, None, None) == T.TRIE_EINVAL
    # offsets[0] < 0 or offsets[K] < offsets[0]: caught on the host (the rest on the device)
    neg = np.array([-1, 2, 4], np.int64)
    assert f(b.ctypes.data, neg.ctypes.data, ok.ctypes.data, 1, None, ctypes.byref(h)) == T.TRIE_EINVAL
    back = np.array([3, 4, 2], np.int64)
    assert f(b.ctypes.data, back.ctypes.data, ok.ctypes.data, 1, None, ctypes.byref(h)) == T.TRIE_EINVAL
    assert "non-decreasing" in T.trie_last_error()
    assert f(None, offs.ctypes.data, ok.ctypes.data, 1, None, ctypes.byref(h)) == T.TRIE_EINVAL
    assert h.value is None


def test_null_handle_queries(lib):
    assert lib.trie_num_nodes(None) == -1
    assert lib.trie_root(None, 0) == -1
    assert lib.trie_destroy(None) == T.TRIE_OK
    assert lib.trie_compile_masks(None, None, None, 10, None, None) == T.TRIE_EINVAL
    assert lib.trie_advance(None, None, None, 1, None, None) == T.TRIE_EINVAL
    assert lib.trie_apply_mask(None, None, 0, None, 1, 10, None) == T.TRIE_EINVAL


def test_vocab_handle_calls_checked_before_any_device_work(lib):
    """Vocabulary handles: NULL handles and bad arguments come back before the GPU is touched."""
    assert lib.trie_vocab_size(None) == -1
    lib.trie_vocab_destroy(None)  # a no-op
    out = ctypes.c_void_p(12345)
    vo = np.array([0, 1, 1], np.int64)
    vb = np.frombuffer(b"a", np.uint8).copy()
    assert lib.trie_vocab_create(vb.ctypes.data, vo.ctypes.data, 2, None) == T.TRIE_EINVAL      # out NULL
    assert lib.trie_vocab_create(vb.ctypes.data, None, 2, ctypes.byref(out)) == T.TRIE_EINVAL   # offsets NULL
    assert out.value is None                                                                     # cleared
    out = ctypes.c_void_p(12345)
    assert lib.trie_vocab_create(vb.ctypes.data, vo.ctypes.data, 1, ctypes.byref(out)) == T.TRIE_EINVAL  # V < 2
    assert out.value is None
    sb, so = W.pack([b"ab"])
    h = T.trie_build(sb, so)
    assert lib.trie_compile_masks_vocab(None, None, 16, None) == T.TRIE_EINVAL        # trie handle NULL
    assert lib.trie_compile_masks_vocab(h.handle, None, None, None) == T.TRIE_EINVAL  # d_mask NULL
    assert lib.trie_compile_masks_vocab(h.handle, None, 2, None) == T.TRIE_EINVAL     # misaligned
    assert lib.trie_compile_masks_vocab(h.handle, None, 16, None) == T.TRIE_EINVAL    # vocabulary NULL
    assert lib.trie_compile_lists_vocab(None, None, None) == T.TRIE_EINVAL
    assert lib.trie_compile_lists_vocab(h.handle, None, None) == T.TRIE_EINVAL
    assert "vocabulary handle is NULL" in T.trie_last_error()


def test_device_calls_checked_before_any_device_work(lib):
    """Argument errors and call-order errors come back before the GPU is touched."""
    sb, so = W.pack([b"ab"])
    h = T.trie_build(sb, so)
    L = lib
    assert L.trie_compile_masks(h.handle, None, None, 1, None, None) == T.TRIE_EINVAL      # V < 2
    vo = np.array([0, 1, 1], np.int64)
    vb = np.frombuffer(b"a", np.uint8).copy()
    assert L.trie_compile_masks(h.handle, vb.ctypes.data, vo.ctypes.data, 2, None, None) == T.TRIE_EINVAL
    assert L.trie_compile_masks(h.handle, vb.ctypes.data, vo.ctypes.data, 2, 2, None) == T.TRIE_EINVAL  # misaligned
    # advance / apply before compile
    assert L.trie_advance(h.handle, 16, 16, 1, None, None) == T.TRIE_ESTATE
    assert L.trie_apply_mask(h.handle, 16, 0, 16, 1, 2, None) == T.TRIE_ESTATE
    assert L.trie_apply_mask(h.handle, 16, 7, 16, 1, 2, None) == T.TRIE_EINVAL           # dtype
    assert L.trie_advance(h.handle, 16, 16, -1, None, None) == T.TRIE_EINVAL


def test_lazy_calls_checked_before_any_device_work(lib):
    """Lazy-row calls: argument and call-order errors before the GPU is touched."""
    sb, so = W.pack([b"ab"])
    h = T.trie_build(sb, so)
    L = lib
    vo = np.array([0, 1, 1], np.int64)
    vb = np.frombuffer(b"a", np.uint8).copy()
    assert L.trie_lazy_apply(h.handle, 16, 0, 16, 1, 2, None) == T.TRIE_ESTATE
    assert L.trie_lazy_advance_apply(h.handle, 16, 16, 32, None, 16, 0, 1, 2, None) == T.TRIE_ESTATE
    assert L.trie_lazy_rows(h.handle, 16, 1, 16, None) == T.TRIE_ESTATE
    assert L.trie_lazy_stats(h.handle, None, None) == T.TRIE_ESTATE
    assert L.trie_lazy_init(h.handle, vb.ctypes.data, vo.ctypes.data, 1, 8, 8) == T.TRIE_EINVAL       # V < 2
    assert L.trie_lazy_init(h.handle, vb.ctypes.data, vo.ctypes.data, 600000, 8, 8) == T.TRIE_EINVAL  # V too big
    assert L.trie_lazy_init(h.handle, vb.ctypes.data, vo.ctypes.data, 2, -1, 8) == T.TRIE_EINVAL      # cache_rows
    for rows in ((1 << 30) + 1, 2**31 - 1):                  # rounding up must not overflow int32
        assert L.trie_lazy_init(h.handle, vb.ctypes.data, vo.ctypes.data, 2, rows, 8) == T.TRIE_EINVAL
        assert "cache_rows" in T.trie_last_error()
    assert L.trie_lazy_init(h.handle, vb.ctypes.data, vo.ctypes.data, 2, 8, 0) == T.TRIE_EINVAL       # max_batch
    assert L.trie_lazy_init(h.handle, vb.ctypes.data, vo.ctypes.data, 2, 8, 4097) == T.TRIE_EINVAL
    assert L.trie_lazy_init(h.handle, vb.ctypes.data, None, 2, 8, 8) == T.TRIE_EINVAL
    for f, args in (("trie_lazy_init", (None, None, 2, 8, 8)), ("trie_lazy_apply", (16, 0, 16, 1, 2, None)),
                    ("trie_lazy_rows", (16, 1, 16, None)), ("trie_lazy_stats", (None, None))):
        assert getattr(L, f)(None, *args) == T.TRIE_EINVAL


def test_fmt_calls_checked_before_any_device_work(lib):
    """Fixed formats: argument and call-order errors before the GPU is touched."""
    L = lib
    h = ctypes.c_void_p()
    cls = W.format_classes("####-##-##")
    assert L.fmt_build(cls.ctypes.data, 1025, ctypes.byref(h)) == T.TRIE_EINVAL
    assert L.fmt_build(cls.ctypes.data, -1, ctypes.byref(h)) == T.TRIE_EINVAL
    assert L.fmt_build(None, 3, ctypes.byref(h)) == T.TRIE_EINVAL
    assert L.fmt_build(cls.ctypes.data, 10, None) == T.TRIE_EINVAL
    f = T.fmt_build(cls)
    assert f.L == 10 and L.fmt_length(None) == -1
    assert L.fmt_advance(f.handle, 16, 16, 1, None, None) == T.TRIE_ESTATE
    assert L.fmt_apply_mask(f.handle, 16, 0, 16, 1, 2, None) == T.TRIE_ESTATE
    assert L.fmt_apply_mask(f.handle, 16, 9, 16, 1, 2, None) == T.TRIE_EINVAL           # dtype
    assert L.fmt_compile_masks(f.handle, None, None, 1, None, None) == T.TRIE_EINVAL      # V < 2
    assert L.fmt_destroy(None) == T.TRIE_OK
    f0 = T.fmt_build(np.zeros((0, 32), np.uint8))                                        # L = 0
    assert f0.L == 0


def test_format_patterns():
    """The four formats of App. K's comparison as class bitmaps."""
    for name, pat in W.FORMATS.items():
        c = W.format_classes(pat)
        assert c.shape == (len(pat), 32)
        sizes = np.unpackbits(c, axis=1).sum(axis=1)
        for ch, n in zip(pat, sizes):
            assert n == {"#": 10, "x": 16, "y": 4}.get(ch, 1), (name, ch)
    assert len(W.FORMATS["UUID v4"]) == 36 and len(W.FORMATS["datetime.ms"]) == 23


def test_binding_fails_loudly_without_library(tmp_path):
    import importlib
    mod = importlib.import_module("paper_2608_12574_gb300.triemask")
    with pytest.raises(RuntimeError, match="missing"):
        old = mod._lib
        mod._lib = None
        try:
            mod.load_library(str(tmp_path / "nope.so"))
        finally:
            mod._lib = old


def test_concurrent_builds_equal_serial(lib):
    """Forests built from 6 threads at once (each build itself multi-threaded,
    all sharing the builder's cache of large blocks) equal a build on its own,
    array for array; every handle is destroyed while the others build."""
    import threading
    w = W.config(5)
    so = w.set_index[:97].astype(np.int32)     # the first 96 sets of the forest workload
    ref = T.trie_build_many(w.set_bytes, w.set_offsets, so)
    want = ref.csr()
    want_roots = ref.roots()
    errors = []

    def work(k):
        try:
            for _ in range(3):
                h = T.trie_build_many(w.set_bytes, w.set_offsets, so)
                got = h.csr()
                for name, arr in want.items():
                    if not np.array_equal(got[name], arr):
                        errors.append((k, name))
                if not np.array_equal(h.roots(), want_roots):
                    errors.append((k, "roots"))
                h.destroy()
        except Exception as e:  # pragma: no cover - reported below
            errors.append((k, repr(e)))

    th = [threading.Thread(target=work, args=(k,)) for k in range(6)]
    for t in th:
        t.start()
    for t in th:
        t.join()
    assert not errors, errors[:5]
