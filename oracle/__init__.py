"""CPU oracle for the trie automaton: brute force, from the paper's definitions.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the
bench's CPU-baseline leg may import this package. It shares no code with the
CUDA path and imports nothing from it.

The arithmetic lives in ``oracle.c`` (a plain C library, each function citing
the passage it follows); this module loads it with ctypes and adds the decode
loop (Eq. 1: mask, greedy choice, state advance), which only calls those
functions in order. ``ac.c`` adds the paper's own Aho-Corasick precomputation
(``AhoCorasick``), used as a third check of the masks and as the stronger
timed CPU baseline.

Pins (``tests/test_oracle_pins.py``): the worked example of App. G.1 and the
Fig. 2 example (``tests/golden/``), exhaustive comparison with the prefix-set
enumeration of the App. G.5 proof on small random sets, and the invariants of
Sec. 4.2 / App. G.5 (tokenization paths allowed, leaves admit only EOS,
prefix closure, padding bits zero, ...). ``Format`` (the character-position
masks of App. K) is pinned in ``tests/test_fmt_oracle.py`` to the same
prefix-set definition on the enumerated strings of small formats, to a closed
form and to a date format worked by hand.
"""
from __future__ import annotations

import contextlib
import ctypes
import os
import subprocess
import threading

import numpy as np

DEAD = -1
FINISHED = -2
_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SRC_AC = os.path.join(_HERE, "ac.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c and ac.c into liboracle.so (gcc, OpenMP) if missing or stale."""
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_SRC_AC))
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < newest:
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=c99",
                               "-o", tmp, _SRC, _SRC_AC])
        os.replace(tmp, _LIB)
    return _LIB


def load_library(path: str):
    """Load one build of oracle.c and declare its signatures."""
    lib = ctypes.CDLL(path)
    P, I32, I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    lib.oracle_trie_build.restype = P
    lib.oracle_trie_build.argtypes = [P, P, I32]
    lib.oracle_trie_free.argtypes = [P]
    lib.oracle_trie_num_nodes.restype = I32
    lib.oracle_trie_num_nodes.argtypes = [P]
    lib.oracle_trie_num_chars.restype = I64
    lib.oracle_trie_num_chars.argtypes = [P]
    lib.oracle_trie_child.restype = I32
    lib.oracle_trie_child.argtypes = [P, I32, I32]
    lib.oracle_trie_info.argtypes = [P, P, P, P, P]
    lib.oracle_mask_rows.argtypes = [P, P, P, I32, P, I64, P, I32]
    lib.oracle_advance.restype = I64
    lib.oracle_advance.argtypes = [P, P, P, I32, P, P, I64]
    lib.oracle_apply.argtypes = [P, P, P, I32, P, I32, P, I64]
    lib.oracle_argmax.argtypes = [P, I32, I64, I32, P]
    lib.oracle_fmt_mask_rows.argtypes = [P, I32, P, P, I32, P, I64, P]
    lib.oracle_fmt_advance.restype = I64
    lib.oracle_fmt_advance.argtypes = [P, I32, P, P, I32, P, P, I64]
    if hasattr(lib, "ac_build"):
        lib.ac_build.restype = P
        lib.ac_build.argtypes = [P, P, I32]
        lib.ac_free.argtypes = [P]
        lib.ac_num_states.restype = I32
        lib.ac_num_states.argtypes = [P]
        lib.ac_valid_pairs.restype = I64
        lib.ac_valid_pairs.argtypes = [P, I32, P, P, P, P, P, I64, I32]
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = load_library(build())
    return _lib


@contextlib.contextmanager
def use_library(path: str):
    """Route oracle calls to another build of oracle.c (the mutation tests plant
    mistakes in a copy of the source and check that the pins catch them)."""
    global _lib
    _load()
    old = _lib
    _lib = load_library(path)
    try:
        yield
    finally:
        _lib = old


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def n_words(V: int) -> int:
    return (V + 31) // 32


class Trie:
    """Byte trie of a string set, node ids in breadth-first / ascending-byte order."""

    def __init__(self, set_bytes: np.ndarray, set_offsets: np.ndarray):
        self._lib = _load()
        self._b = np.ascontiguousarray(set_bytes, dtype=np.uint8)
        self._o = np.ascontiguousarray(set_offsets, dtype=np.int64)
        if self._b.size == 0:
            self._b = np.zeros(1, dtype=np.uint8)
        h = self._lib.oracle_trie_build(_p(self._b), _p(self._o), len(self._o) - 1)
        if not h:
            raise MemoryError("oracle_trie_build failed")
        self._h = ctypes.c_void_p(h)
        self.num_nodes = self._lib.oracle_trie_num_nodes(self._h)
        self.num_chars = self._lib.oracle_trie_num_chars(self._h)
        n = self.num_nodes
        self.parent = np.empty(n, np.int32)
        self.label = np.empty(n, np.uint8)
        self.terminal = np.empty(n, np.uint8)
        self.depth = np.empty(n, np.int32)
        self._lib.oracle_trie_info(self._h, _p(self.parent), _p(self.label), _p(self.terminal),
                                   _p(self.depth))

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            self._lib.oracle_trie_free(h)
            self._h = None

    def child(self, node: int, byte: int) -> int:
        return self._lib.oracle_trie_child(self._h, node, byte)

    def prefix(self, node: int) -> bytes:
        out = bytearray()
        while node > 0:
            out.append(int(self.label[node]))
            node = int(self.parent[node])
        return bytes(reversed(out))


class Vocab:
    def __init__(self, vocab_bytes: np.ndarray, vocab_offsets: np.ndarray):
        self.b = np.ascontiguousarray(vocab_bytes, dtype=np.uint8)
        if self.b.size == 0:
            self.b = np.zeros(1, dtype=np.uint8)
        self.o = np.ascontiguousarray(vocab_offsets, dtype=np.int64)
        self.V = len(self.o) - 1
        self.eos = self.V - 1


def mask_rows(t: Trie, voc: Vocab, rows, nthreads: int = 1) -> np.ndarray:
    """uint32[len(rows), ceil(V/32)] mask rows (App. G.5 proof conditions, EOS at terminals)."""
    rows = np.ascontiguousarray(rows, dtype=np.int32)
    out = np.zeros((rows.size, n_words(voc.V)), dtype=np.uint32)
    t._lib.oracle_mask_rows(t._h, _p(voc.b), _p(voc.o), voc.V, _p(rows), rows.size, _p(out),
                            nthreads)
    return out


def mask_all(t: Trie, voc: Vocab, nthreads: int = 1) -> np.ndarray:
    return mask_rows(t, voc, np.arange(t.num_nodes, dtype=np.int32), nthreads)


def advance(t: Trie, voc: Vocab, states: np.ndarray, tokens: np.ndarray) -> tuple[np.ndarray, int]:
    """(next states, number of new DEAD moves) for one batch of tokens."""
    s = np.ascontiguousarray(states, dtype=np.int32).copy()
    tk = np.ascontiguousarray(tokens, dtype=np.int32)
    err = t._lib.oracle_advance(t._h, _p(voc.b), _p(voc.o), voc.V, _p(s), _p(tk), s.size)
    return s, int(err)


def _bits(logits: np.ndarray) -> tuple[np.ndarray, int]:
    if logits.dtype == np.uint32:
        return np.ascontiguousarray(logits), 0
    if logits.dtype == np.uint16:
        return np.ascontiguousarray(logits), 1
    raise TypeError("pass logits as raw bits: uint32 (fp32) or uint16 (bf16)")


def apply(t: Trie, voc: Vocab, logits_bits: np.ndarray, states: np.ndarray) -> np.ndarray:
    """Masked copy of [B, V] raw-bit logits (uint32 = fp32, uint16 = bf16)."""
    x, dt = _bits(logits_bits)
    x = x.copy()
    st = np.ascontiguousarray(states, dtype=np.int32)
    t._lib.oracle_apply(t._h, _p(voc.b), _p(voc.o), voc.V, _p(x), dt, _p(st), st.size)
    return x


def argmax(logits_bits: np.ndarray) -> np.ndarray:
    x, dt = _bits(logits_bits)
    B, V = x.shape
    out = np.empty(B, np.int32)
    _load().oracle_argmax(_p(x), dt, B, V, _p(out))
    return out


class AhoCorasick:
    """The paper's automaton over the vocabulary (ac.c): built once per
    tokenizer, then run over any trie (Sec. 4.2; App. H.4 Phases 3-4)."""

    def __init__(self, voc: Vocab):
        self._lib = _load()
        self.voc = voc
        h = self._lib.ac_build(_p(voc.b), _p(voc.o), voc.V)
        if not h:
            raise MemoryError("ac_build failed")
        self._h = ctypes.c_void_p(h)
        self.num_states = self._lib.ac_num_states(self._h)

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            self._lib.ac_free(h)
            self._h = None

    def pairs(self, t: Trie, nthreads: int = 1) -> tuple[np.ndarray, np.ndarray]:
        """(start node, token) of every allowed pair, EOS excluded."""
        args = (self._h, t.num_nodes, _p(t.parent), _p(t.label), _p(t.depth))
        n = self._lib.ac_valid_pairs(*args, None, None, 0, nthreads)
        if n < 0:
            raise MemoryError("ac_valid_pairs failed")
        rows = np.empty(max(n, 1), np.int32)
        toks = np.empty(max(n, 1), np.int32)
        self._lib.ac_valid_pairs(*args, _p(rows), _p(toks), n, nthreads)
        return rows[:n], toks[:n]

    def mask(self, t: Trie, nthreads: int = 1) -> np.ndarray:
        """Dense [N, ceil(V/32)] mask from the pairs, EOS at terminal nodes (App. G.5)."""
        rows, toks = self.pairs(t, nthreads)
        V = self.voc.V
        m = np.zeros((t.num_nodes, n_words(V)), np.uint32)
        np.bitwise_or.at(m, (rows, toks >> 5), (np.uint32(1) << (toks & 31).astype(np.uint32)))
        term = np.nonzero(t.terminal)[0]
        m[term, (V - 1) >> 5] |= np.uint32(1 << ((V - 1) & 31))
        return m


def decode(t: Trie, voc: Vocab, logits_per_step, states0: np.ndarray):
    """Greedy constrained decode (Eq. 1 with greedy choice): per step mask -> argmax -> advance.

    ``logits_per_step`` yields [B, V] raw-bit arrays. Returns per-step lists of
    (masked logits, tokens, states after the step) and the total error count.
    """
    states = np.ascontiguousarray(states0, dtype=np.int32).copy()
    masked, toks, sts = [], [], []
    errors = 0
    for lg in logits_per_step:
        m = apply(t, voc, lg, states)
        tk = argmax(m)
        states, e = advance(t, voc, states, tk)
        errors += e
        masked.append(m)
        toks.append(tk)
        sts.append(states.copy())
    return masked, toks, sts, errors


class Format:
    """A fixed format for the character-position masks (App. K): L byte
    classes, classes[i] a 32-byte bitmap (byte c allowed iff bit c % 8 of
    classes[i][c // 8]). States are the positions 0..L."""

    def __init__(self, classes: np.ndarray):
        self.classes = np.ascontiguousarray(classes, dtype=np.uint8).reshape(-1, 32)
        self.L = self.classes.shape[0]
        self._lib = _load()

    def mask_rows(self, voc: Vocab, rows) -> np.ndarray:
        rows = np.ascontiguousarray(rows, dtype=np.int32)
        out = np.zeros((rows.size, n_words(voc.V)), np.uint32)
        self._lib.oracle_fmt_mask_rows(_p(self.classes), self.L, _p(voc.b), _p(voc.o), voc.V, _p(rows), rows.size,
                                       _p(out))
        return out

    def mask_all(self, voc: Vocab) -> np.ndarray:
        return self.mask_rows(voc, np.arange(self.L + 1, dtype=np.int32))

    def advance(self, voc: Vocab, states: np.ndarray, tokens: np.ndarray) -> tuple[np.ndarray, int]:
        s = np.array(states, dtype=np.int32, copy=True)
        tk = np.ascontiguousarray(tokens, dtype=np.int32)
        err = self._lib.oracle_fmt_advance(_p(self.classes), self.L, _p(voc.b), _p(voc.o), voc.V, _p(s), _p(tk),
                                           s.size)
        return s, int(err)

    def apply(self, voc: Vocab, logits_bits: np.ndarray, states: np.ndarray) -> np.ndarray:
        """-inf (fp32 0xFF800000 / bf16 0xFF80) where the row of the state's
        position clears the token (Sec. 4.2 last paragraph, App. H.3)."""
        x = np.array(logits_bits, copy=True)
        rows = self.mask_rows(voc, states)
        allowed = np.unpackbits(rows.view(np.uint8), axis=1, bitorder="little")[:, :voc.V].astype(bool)
        x[~allowed] = np.uint32(0xFF800000) if x.dtype == np.uint32 else np.uint16(0xFF80)
        return x

