"""GPU: forests built on the device (trie_build_many_device) against the CPU
oracle's tries and the host builder, through the C ABI.

The node numbering is part of the ABI (breadth-first per set, siblings by
ascending byte, sets concatenated in order), so a device-built forest must
equal the host-built one array for array, and every set must equal the
oracle's own trie of that set. The downstream calls (valid lists, lazy rows,
the no-alloc compile, the fused decode step) must then give the same results
on either handle.
"""
from __future__ import annotations

import random

import numpy as np
import pytest

import oracle
from paper_2608_12574_gb300 import triemask as T
from paper_2608_12574_gb300 import workloads as W
from pins import random_case

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="session")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_12574_gb300 import _build
    _build.build()
    T.load_library()
    oracle.build()
    return torch.device("cuda:0")


def _np_u32(t):
    import torch
    return t.cpu().contiguous().view(torch.int32).numpy().view(np.uint32)


def _forest(sets):
    flat = [s for st in sets for s in st]
    index = np.cumsum([0] + [len(s) for s in sets]).astype(np.int32)
    sb, so = W.pack(flat)
    return sb, so, index


def _check_against_oracle(h, sets):
    """Every set of h equals the oracle's trie of that set, at its root."""
    c = h.csr()
    assert h.num_sets == len(sets)
    chars, depth = 0, 0
    for i, st in enumerate(sets):
        r = h.root(i)
        ot = oracle.Trie(*W.pack(st))
        n = ot.num_nodes
        nxt = h.root(i + 1) if i + 1 < len(sets) else h.num_nodes
        assert nxt - r == n, f"set {i}: {nxt - r} nodes, oracle {n}"
        par = c["parent"][r:r + n].astype(np.int64)
        par[par >= 0] -= r
        assert np.array_equal(par, ot.parent), f"set {i}"
        assert np.array_equal(c["label"][r:r + n], ot.label), f"set {i}"
        assert np.array_equal(c["terminal"][r:r + n], ot.terminal), f"set {i}"
        chars += ot.num_chars
        depth = max(depth, int(ot.depth.max()))
    assert h.num_chars == chars
    assert h.max_depth == depth


def _same_handles(a, b):
    assert a.num_nodes == b.num_nodes and a.num_sets == b.num_sets
    assert np.array_equal(a.roots(), b.roots())
    assert a.num_chars == b.num_chars and a.max_depth == b.max_depth
    ca, cb = a.csr(), b.csr()
    for k in ca:
        assert np.array_equal(ca[k], cb[k]), k


def _random_sets(seed):
    r = random.Random(seed)
    sets = []
    for j in range(r.randint(1, 12)):
        if r.random() < 0.15:
            sets.append([])  # a set with no strings: a lone, non-terminal root
            continue
        strings, _ = random_case(seed * 100 + j)
        sets.append(strings)
    return sets


@pytest.mark.parametrize("seed", range(40))
def test_device_forest_small_random(cuda, seed):
    """Random forests (empty sets, empty strings, duplicates, prefixes of
    other strings, bytes 0x00 / 0xFF): each set equals the oracle's trie, and
    the whole forest equals the host builder's."""
    sets = _random_sets(seed)
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _check_against_oracle(d, sets)
    _same_handles(d, T.trie_build_many(sb, so, index))


@pytest.mark.parametrize("big", [4096, 4097, 9000])
def test_device_forest_set_size_paths(cuda, big):
    """Sets of up to 4,096 strings are built one CTA per set (levels in shared
    memory), larger ones by the level path over all sets: both sides of the
    boundary, with small random sets beside the big one."""
    r = random.Random(big)
    alpha = [0x00, 0x41, 0x61, 0x5F, 0xFF]
    big_set = [bytes(r.choice(alpha) for _ in range(r.randint(0, 9))) for _ in range(big)]
    sets = _random_sets(big)[:3] + [big_set] + _random_sets(big + 1)[:3]
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _check_against_oracle(d, sets)
    _same_handles(d, T.trie_build_many(sb, so, index))


def test_device_forest_level_path_codes(cuda):
    """The K = 10,000 ICD-style codes as one set (level path), between two
    small sets."""
    w = W.config(3)
    codes = W.unpack(w.set_bytes, w.set_offsets)
    sets = [[b"A01.1", b"A01"], codes, [b"", b"Z"]]
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _check_against_oracle(d, sets)
    _same_handles(d, T.trie_build_many(sb, so, index))


@pytest.mark.parametrize("sets", [[[]], [[], [], []], [[b""]], [[], [b""], []]])
def test_device_forest_without_bytes(cuda, sets):
    """Forests without a single string byte: lone roots (terminal where the
    set holds the empty string)."""
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _check_against_oracle(d, sets)
    _same_handles(d, T.trie_build_many(sb, so, index))


def test_device_forest_more_sets_than_strings(cuda):
    """5,000 sets holding 3 strings in all: the root level is the widest."""
    sets = [[] for _ in range(5000)]
    sets[7] = [b"ab"]
    sets[4000] = [b"", b"abc"]
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _same_handles(d, T.trie_build_many(sb, so, index))
    c = d.csr()
    assert d.num_nodes == 5000 + 2 + 3
    assert d.root(7) == 7 and d.root(8) == 10 and c["terminal"][d.root(4000)] == 1


def test_device_forest_offsets_checked_on_the_device(cuda):
    """Offsets that decrease, or go negative, inside the list are found by the
    staging kernel: TRIE_EINVAL, and no handle."""
    import ctypes
    lib = T.load_library()
    b = np.frombuffer(b"abcdefgh", np.uint8).copy()
    so = np.array([0, 3], np.int32)
    h = ctypes.c_void_p()
    for offs in ([0, 5, 2, 8], [0, 3, -1, 8], [0, 9, 4, 8]):
        o = np.array(offs, np.int64)
        rc = lib.trie_build_many_device(b.ctypes.data, o.ctypes.data, so.ctypes.data, 1, None, ctypes.byref(h))
        assert rc == T.TRIE_EINVAL, offs
        assert "non-decreasing" in T.trie_last_error()
        assert h.value is None


@pytest.mark.parametrize("shift", [0, 1, 5, 15])
def test_device_forest_unaligned_bytes(cuda, shift):
    """Byte arrays that start at any alignment, and offsets that do not start
    at 0: the staged image keeps the source's alignment."""
    sets = _random_sets(7) + [[b"get", b"get_user", b"", b"set"]]
    sb, so, index = _forest(sets)
    buf = np.zeros(len(sb) + 64, np.uint8)
    view = buf[shift:shift + len(sb) + 3]
    view[3:3 + len(sb)] = sb
    d = T.trie_build_many_device(view, so + 3, index)
    _check_against_oracle(d, sets)


def test_device_forest_copy_path(cuda):
    """The path for devices that cannot read pageable host memory (copies,
    then the same checks on the device), forced in a fresh process."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    code = (
        "import sys; sys.path[:0] = [%r, %r]\n"
        "import numpy as np\n"
        "from paper_2608_12574_gb300 import triemask as T\n"
        "import test_gpu_device_build as t\n"
        "for seed in range(12):\n"
        "    sets = t._random_sets(seed)\n"
        "    sb, so, index = t._forest(sets)\n"
        "    d = T.trie_build_many_device(sb, so, index)\n"
        "    t._check_against_oracle(d, sets)\n"
        "    t._same_handles(d, T.trie_build_many(sb, so, index))\n"
        "print('ok')\n" % (root, os.path.join(root, "tests")))
    env = dict(os.environ, TRIEMASK_HOST_READ="copy")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout + r.stderr


def test_device_forest_repeated_builds_reuse_memory(cuda):
    """Build, use and destroy forests of different sizes in turn, as a server
    does per batch: every build is still equal to the host builder's (blocks
    that the library's pool hands out again carry nothing over), and the
    device memory in use stops growing once the pool holds its blocks."""
    import torch
    w = W.dynamic_requests(24)
    small = [_forest(_random_sets(s)) for s in (41, 42)]
    free = []
    for it in range(6):
        sb, so, index = (w.set_bytes, w.set_offsets, w.set_index) if it % 2 == 0 else small[it // 2 % 2]
        d = T.trie_build_many_device(sb, so, index)
        T.trie_compile_lists(d, w.vocab_bytes, w.vocab_offsets, w.V)
        if it < 2 or it == 5:
            h = T.trie_build_many(sb, so, index)
            _same_handles(d, h)
            T.trie_compile_lists(h, w.vocab_bytes, w.vocab_offsets, w.V)
            od, td = T.trie_copy_lists(d)
            oh, th = T.trie_copy_lists(h)
            assert torch.equal(od, oh)
            rows = np.repeat(np.arange(d.num_nodes, dtype=np.int64), np.diff(od.cpu().numpy()))
            assert np.array_equal(np.sort(rows * w.V + td.cpu().numpy()), np.sort(rows * w.V + th.cpu().numpy()))
            h.destroy()
        d.destroy()
        torch.cuda.synchronize()
        free.append(torch.cuda.mem_get_info()[0])
    # after the first large build the pool serves the later ones
    assert free[-2] >= free[2] - (64 << 20), free


def test_device_forest_single_set_mask_equals_oracle(cuda):
    """A forest of one set (the K=100 tool names): the dense mask compiled on
    the device-built handle equals the oracle's mask."""
    import os
    w = W.config(1)
    d = T.trie_build_many_device(w.set_bytes, w.set_offsets, np.array([0, len(w.set_offsets) - 1], np.int32))
    _same_handles(d, T.trie_build(w.set_bytes, w.set_offsets))
    m = T.alloc_mask(d, w.V, cuda)
    T.trie_compile_masks(d, w.vocab_bytes, w.vocab_offsets, w.V, m)
    want = oracle.mask_all(oracle.Trie(w.set_bytes, w.set_offsets), oracle.Vocab(w.vocab_bytes, w.vocab_offsets),
                           nthreads=os.cpu_count() or 1)
    assert np.array_equal(_np_u32(m), want)


def test_device_forest_long_strings_use_the_host_builder(cuda):
    """Strings longer than the level loop's limit (1,024 bytes) go to the host
    builder; the result is the same forest."""
    rng = np.random.default_rng(11)
    long = bytes(rng.integers(0, 3, 1500, dtype=np.uint8))
    sets = [[long, long[:700], b"xy"], [long[:1100]]]
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _check_against_oracle(d, sets)
    assert d.max_depth == 1500


def test_device_forest_noalloc_compile(cuda):
    """The no-alloc compile reads a device-built trie's arrays on the device;
    its mask equals trie_compile_masks on the same handle."""
    sets = _random_sets(3) + [[b"get", b"get_user", b"set"]]
    sb, so, index = _forest(sets)
    d = T.trie_build_many_device(sb, so, index)
    _, toks = random_case(77)
    vb, vo = W.pack(toks)
    V = len(toks)
    m1 = T.alloc_mask(d, V, cuda)
    m2 = T.alloc_mask(d, V, cuda)
    m2.fill_(-1)
    T.trie_compile_masks(d, vb, vo, V, m1)
    T.trie_compile_masks_noalloc(d, vb, vo, V, m2)
    assert np.array_equal(_np_u32(m1), _np_u32(m2))


def test_device_forest_config5(cuda):
    """The 256-request forest (4.8M nodes): equal to the host builder's; the
    valid lists, lazy rows of sampled states and four fused list-driven
    decode steps equal those of the host-built forest."""
    import torch
    w = W.config(5)
    d = T.trie_build_many_device(w.set_bytes, w.set_offsets, w.set_index)
    hst = T.trie_build_many(w.set_bytes, w.set_offsets, w.set_index)
    _same_handles(d, hst)
    # sampled sets against the oracle
    strings = W.unpack(w.set_bytes, w.set_offsets)
    sel = [0, 1, 100, 255]
    c = d.csr()
    for i in sel:
        ot = oracle.Trie(*W.pack(strings[w.set_index[i]:w.set_index[i + 1]]))
        r, n = d.root(i), ot.num_nodes
        assert np.array_equal(c["label"][r:r + n], ot.label)
        assert np.array_equal(c["terminal"][r:r + n], ot.terminal)

    T.trie_compile_lists(d, w.vocab_bytes, w.vocab_offsets, w.V)
    T.trie_compile_lists(hst, w.vocab_bytes, w.vocab_offsets, w.V)
    od, td = T.trie_copy_lists(d)
    oh, th = T.trie_copy_lists(hst)
    assert torch.equal(od, oh)
    rows = np.repeat(np.arange(d.num_nodes, dtype=np.int64), np.diff(od.cpu().numpy()))
    # the tokens of a row are in no particular order
    assert np.array_equal(np.sort(rows * w.V + td.cpu().numpy()), np.sort(rows * w.V + th.cpu().numpy()))

    B = 256
    st = torch.as_tensor(d.roots()[:B].astype(np.int32), device=cuda)
    sd, sh = st.clone(), st.clone()
    tok = None
    for step in range(5):
        lg = W.logits(w, step, device="cuda", batch=B)
        xd, xh = lg.clone(), lg.clone()
        if tok is None:
            T.trie_apply_lists(d, xd, sd)
            T.trie_apply_lists(hst, xh, sh)
        else:
            nd, nh = torch.empty_like(sd), torch.empty_like(sh)
            T.trie_advance_apply_lists(d, sd, tok, nd, xd)
            T.trie_advance_apply_lists(hst, sh, tok, nh, xh)
            assert torch.equal(nd, nh), f"step {step}"
            sd, sh = nd, nh
        assert torch.equal(xd.view(torch.int16), xh.view(torch.int16)), f"step {step}"
        tok = torch.argmax(xd, dim=1).to(torch.int32)
    assert int((sd >= 0).sum()) > 0  # the greedy walk stayed inside the tries

    rng = np.random.default_rng(5)
    states = rng.integers(0, d.num_nodes, 2048).astype(np.int32)
    rows = []
    for h in (d, hst):
        T.trie_lazy_init(h, w.vocab_bytes, w.vocab_offsets, w.V, cache_rows=1024, max_batch=2048)
        rows.append(_np_u32(T.trie_lazy_rows(h, torch.as_tensor(states, device=cuda), w.V)))
    assert np.array_equal(rows[0], rows[1])


def _link_sets():
    """Sets whose tries stress the child links: empty sets and lone terminal
    roots next to each other, a root with all 256 children, a chain of 70
    nodes, parents whose children run past a warp's 32 consecutive nodes
    (100 and 256 siblings), and many one-child parents."""
    return [[], [b""], [bytes([i]) for i in range(256)], [], [b"x" * 70],
            [bytes([i, j]) for i in range(3) for j in range(0, 200, 2)], [b"a"], [],
            [bytes([97 + i % 26]) * (1 + i % 9) + bytes([i]) for i in range(60)],
            [bytes([i, 255 - i]) for i in range(256)], [b""], []]


@pytest.mark.parametrize("builder", ["host", "device"])
def test_child_links_walk_every_byte(cuda, builder):
    """The child links built on the device (first child and 256-bit child-label
    set of every node) move every (node, byte) pair to the child that the
    parent and label arrays give, and every other pair to DEAD: trie_advance
    by single-byte tokens walks exactly one link."""
    import torch
    sets = _link_sets()
    sb, so, index = _forest(sets)
    h = (T.trie_build_many_device(sb, so, index) if builder == "device"
         else T.trie_build_many(sb, so, index))
    _check_against_oracle(h, sets)
    vb, vo = W.pack([bytes([b]) for b in range(256)] + [b""])  # token 256: EOS
    T.trie_compile_lists(h, vb, vo, 257)
    c = h.csr()
    n = h.num_nodes
    child = np.full((n, 256), T.TRIE_STATE_DEAD, np.int32)
    for x in range(n):
        if c["parent"][x] >= 0:
            child[c["parent"][x], c["label"][x]] = x
    states = torch.as_tensor(np.repeat(np.arange(n, dtype=np.int32), 256), device=cuda)
    tokens = torch.as_tensor(np.tile(np.arange(256, dtype=np.int32), n), device=cuda)
    err = torch.zeros(1, dtype=torch.int32, device=cuda)
    T.trie_advance(h, states, tokens, err)
    got = states.cpu().numpy().reshape(n, 256)
    assert np.array_equal(got, child)
    assert int(err.item()) == int((child == T.TRIE_STATE_DEAD).sum())
    h.destroy()
