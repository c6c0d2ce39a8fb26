"""Seeded synthetic inputs: enum sets, byte vocabularies and logits.

This module only draws input data. It holds none of the trie-automaton
arithmetic and is the one module that both the CUDA path and the CPU oracle
are fed from. Every draw comes from a counter-based splitmix64 stream, so the
same seed gives the same bytes on any machine and with any numpy version.

Workloads stand in for the paper's inputs (Sec. 5 and App. C: tool-name sets,
the ICD-10-CM code list, tokenizers of 32K-262K tokens), none of which ship
with this library:

* ``tool_names``: snake_case names, 8-32 bytes, built from shared stems of
  2-3 synthetic words plus suffix words (prefix sharing r ~ 0.4, Table
  prefix_sharing reports r = 0.40 for the paper's synthetic tools).
* ``icd_codes``: uppercase letter + 2 digits [+ '.' + 0-4 of A-Z0-9], the
  category drawn Zipf-skewed over the 2,600 letter+2-digit prefixes (r ~ 0.2,
  the paper reports r = 0.19 for ICD-10-CM).
* ``byte_vocab``: ids 0-255 are the 256 single bytes, the middle ids are
  distinct multi-byte tokens, and id V-1 is EOS with no bytes.

Sets and vocabularies are returned as (bytes: uint8[], offsets: int64[K+1]).
"""
from __future__ import annotations

import dataclasses
import numpy as np

_M64 = np.uint64(0xFFFFFFFFFFFFFFFF)
_GOLDEN = np.uint64(0x9E3779B97F4A7C15)


class SplitMix64:
    """Counter-based splitmix64 (Steele, Lea & Flood, OOPSLA 2014).

    Output i of a stream with seed s is mix(s + (i+1) * 0x9E3779B97F4A7C15).
    """

    def __init__(self, seed: int):
        self.state = np.uint64(seed & 0xFFFFFFFFFFFFFFFF)

    def u64(self, n: int) -> np.ndarray:
        with np.errstate(over="ignore"):
            ctr = np.arange(1, n + 1, dtype=np.uint64) * _GOLDEN + self.state
            self.state = self.state + np.uint64(n) * _GOLDEN
            z = ctr
            z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
            z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
            z = z ^ (z >> np.uint64(31))
        return z

    def random(self, n: int) -> np.ndarray:
        """n doubles uniform in [0, 1)."""
        return (self.u64(n) >> np.uint64(11)).astype(np.float64) * (1.0 / (1 << 53))

    def integers(self, lo: int, hi: int, n: int) -> np.ndarray:
        """n int64 uniform in [lo, hi)."""
        return lo + np.floor(self.random(n) * (hi - lo)).astype(np.int64)

    def choice(self, n: int, p: np.ndarray) -> np.ndarray:
        """n indices drawn from the discrete distribution p."""
        cdf = np.cumsum(p / p.sum())
        cdf[-1] = 1.0
        return np.searchsorted(cdf, self.random(n), side="right").astype(np.int64)


# English-like letter weights (our choice; any fixed table serves).
_LETTERS = b"abcdefghijklmnopqrstuvwxyz"
_LETTER_W = np.array([8.2, 1.5, 2.8, 4.3, 12.7, 2.2, 2.0, 6.1, 7.0, 0.2, 0.8, 4.0, 2.4,
                      6.7, 7.5, 1.9, 0.1, 6.0, 6.3, 9.1, 2.8, 1.0, 2.4, 0.2, 2.0, 0.1])
_VOWELS = set(b"aeiou")


def _words(rng: SplitMix64, n: int, lo: int = 3, hi: int = 8) -> list[bytes]:
    """n distinct pronounceable lower-case words of lo..hi letters."""
    vw = np.array([w if c in _VOWELS else 0.0 for c, w in zip(_LETTERS, _LETTER_W)])
    cw = np.array([0.0 if c in _VOWELS else w for c, w in zip(_LETTERS, _LETTER_W)])
    out: list[bytes] = []
    seen: set[bytes] = set()
    while len(out) < n:
        m = 2 * (n - len(out)) + 8
        lens = rng.integers(lo, hi + 1, m)
        total = int(lens.sum())
        u = rng.random(total)
        vc = rng.choice(total, vw)
        cc = rng.choice(total, cw)
        pos = 0
        for L in lens:
            w = bytearray()
            prev_vowel = u[pos] < 0.5
            for j in range(L):
                # alternate consonant / vowel with a bias, as a crude letter model
                want_vowel = (u[pos + j] < 0.6) if not prev_vowel else (u[pos + j] < 0.2)
                c = _LETTERS[vc[pos + j]] if want_vowel else _LETTERS[cc[pos + j]]
                w.append(c)
                prev_vowel = want_vowel
            pos += int(L)
            b = bytes(w)
            if b not in seen:
                seen.add(b)
                out.append(b)
                if len(out) == n:
                    break
    return out


def pack(strings: list[bytes]) -> tuple[np.ndarray, np.ndarray]:
    """Concatenate byte strings into (uint8 bytes, int64 offsets[K+1])."""
    offs = np.zeros(len(strings) + 1, dtype=np.int64)
    if strings:
        offs[1:] = np.cumsum([len(s) for s in strings])
    data = np.frombuffer(b"".join(strings), dtype=np.uint8).copy()
    return data, offs


def unpack(data: np.ndarray, offs: np.ndarray) -> list[bytes]:
    raw = data.tobytes()
    return [raw[offs[i]:offs[i + 1]] for i in range(len(offs) - 1)]


# ---------------------------------------------------------------- enum sets

def tool_stems(seed: int, n_stems: int) -> list[bytes]:
    """n_stems distinct stems of 2-3 words joined by '_'."""
    rng = SplitMix64(seed * 1000003 + 11)
    words = _words(rng, max(3 * n_stems, 64))
    stems: list[bytes] = []
    seen: set[bytes] = set()
    i = 0
    while len(stems) < n_stems:
        k = int(rng.integers(2, 4, 1)[0])
        idx = rng.integers(0, len(words), k)
        s = b"_".join(words[j] for j in idx)
        if len(s) <= 24 and s not in seen:
            seen.add(s)
            stems.append(s)
        i += 1
    return stems


def tool_names(seed: int, K: int, n_stems: int, lo: int = 8, hi: int = 32) -> list[bytes]:
    """K distinct snake_case names: a shared stem + 1-3 suffix words, lo..hi bytes."""
    stems = tool_stems(seed, n_stems)
    rng = SplitMix64(seed * 1000003 + 29)
    suffix_words = _words(rng, max(4 * n_stems, 200))
    # stems are used Zipf-ish so that some namespaces are much larger than others
    sw = 1.0 / np.arange(1, n_stems + 1) ** 0.8
    out: list[bytes] = []
    seen: set[bytes] = set()
    while len(out) < K:
        m = 2 * (K - len(out)) + 16
        st = rng.choice(m, sw)
        nsuf = rng.integers(1, 4, m)
        wi = rng.integers(0, len(suffix_words), 3 * m)
        for r in range(m):
            s = stems[st[r]] + b"".join(b"_" + suffix_words[wi[3 * r + j]] for j in range(nsuf[r]))
            if lo <= len(s) <= hi and s not in seen:
                seen.add(s)
                out.append(s)
                if len(out) == K:
                    break
    return out


_UPPER = b"ABCDEFGHIJKLMNOPQRSTUVWXYZ"
_DIGITS = b"0123456789"
_ALNUM_UP = _UPPER + _DIGITS


def icd_codes(seed: int, K: int, max_suffix: int, zipf_s: float = 1.1) -> list[bytes]:
    """K distinct codes: letter + 2 digits, then '.' + 1..max_suffix of [A-Z0-9].

    A zero-length suffix gives the bare category ("A12"), which is then both a
    value and a proper prefix of its longer codes. The category is drawn from
    a Zipf(s) law over a seeded ranking of the 26*100 categories.
    """
    rng = SplitMix64(seed * 1000003 + 47)
    cats = [bytes([L]) + b"%02d" % d for L in _UPPER for d in range(100)]
    perm = np.argsort(rng.random(len(cats)), kind="stable")
    ranked = [cats[i] for i in perm]
    w = 1.0 / np.arange(1, len(cats) + 1) ** zipf_s
    out: list[bytes] = []
    seen: set[bytes] = set()
    while len(out) < K:
        m = 2 * (K - len(out)) + 16
        c = rng.choice(m, w)
        sl = rng.integers(0, max_suffix + 1, m)
        ch = rng.integers(0, len(_ALNUM_UP), m * max(max_suffix, 1))
        for r in range(m):
            s = ranked[c[r]]
            if sl[r] > 0:
                s = s + b"." + bytes(_ALNUM_UP[ch[r * max_suffix + j]] for j in range(sl[r]))
            if s not in seen:
                seen.add(s)
                out.append(s)
                if len(out) == K:
                    break
    return out


# ------------------------------------------------------------- vocabularies

_PUNCT = b".,-:;!?()'\"/"
_SPACE = b" "


def _char_table(upper: bool, mixed: bool) -> tuple[bytes, np.ndarray]:
    chars = bytearray(_LETTERS)
    w = list(_LETTER_W / _LETTER_W.sum() * 0.62)
    if upper or mixed:
        chars += _UPPER
        w += list(_LETTER_W / _LETTER_W.sum() * (0.25 if mixed else 0.18))
    chars += _DIGITS
    w += [0.08 / 10] * 10
    chars += b"_"
    w += [0.05]
    chars += _SPACE
    w += [0.10]
    chars += _PUNCT
    w += [0.07 / len(_PUNCT)] * len(_PUNCT)
    return bytes(chars), np.array(w)


def _lengths(rng: SplitMix64, n: int, lo: int, hi: int, decay: float) -> np.ndarray:
    ks = np.arange(lo, hi + 1)
    p = decay ** (ks - lo)
    return ks[rng.choice(n, p)]


@dataclasses.dataclass
class VocabSpec:
    V: int
    max_len: int            # longest multi-byte token
    substr_frac: float      # share drawn as substrings of `substr_src`
    run_frac: float         # share drawn as runs of [A-Z0-9]
    run_len: tuple[int, int]
    upper: bool
    mixed: bool
    decay: float = 0.78     # geometric length law: P(len) ~ decay**(len-2)


def byte_vocab(seed: int, spec: VocabSpec, substr_src: list[bytes] | None = None
               ) -> tuple[np.ndarray, np.ndarray]:
    """Vocabulary of V tokens: 256 single bytes, V-257 distinct multi-byte tokens, EOS.

    EOS is id V-1 and has no bytes. Multi-byte tokens are drawn from three
    sources: substrings (2..max_len) of the given strings, runs of [A-Z0-9],
    and a per-character frequency model; duplicates are redrawn.
    """
    V = spec.V
    if V < 257:
        raise ValueError("byte_vocab needs V >= 257 (256 single bytes + EOS)")
    rng = SplitMix64(seed * 1000003 + 71)
    toks: list[bytes] = [bytes([b]) for b in range(256)]
    seen: set[bytes] = set(toks)
    n_multi = V - 257
    chars, cw = _char_table(spec.upper, spec.mixed)
    src = substr_src or []
    n_sub = int(round(n_multi * spec.substr_frac)) if src else 0
    n_run = int(round(n_multi * spec.run_frac))
    want = [("sub", n_sub), ("run", n_run), ("model", n_multi - n_sub - n_run)]
    for kind, n in want:
        got = 0
        tries = 0
        while got < n:
            m = 2 * (n - got) + 64
            tries += 1
            if kind == "sub" and tries > 50:
                # the source strings ran out of distinct substrings
                want[-1] = ("model", want[-1][1] + (n - got))
                break
            if kind == "sub":
                si = rng.integers(0, len(src), m)
                lens = _lengths(rng, m, 2, spec.max_len, spec.decay)
                us = rng.random(m)
                for r in range(m):
                    s = src[si[r]]
                    L = min(int(lens[r]), len(s))
                    if L < 2:
                        continue
                    a = int(us[r] * (len(s) - L + 1))
                    t = s[a:a + L]
                    if t not in seen:
                        seen.add(t)
                        toks.append(t)
                        got += 1
                        if got == n:
                            break
            elif kind == "run":
                lens = rng.integers(spec.run_len[0], spec.run_len[1] + 1, m)
                ch = rng.integers(0, len(_ALNUM_UP), int(lens.sum()))
                pos = 0
                for r in range(m):
                    t = bytes(_ALNUM_UP[c] for c in ch[pos:pos + lens[r]])
                    pos += int(lens[r])
                    if t not in seen:
                        seen.add(t)
                        toks.append(t)
                        got += 1
                        if got == n:
                            break
            else:
                lens = _lengths(rng, m, 2, spec.max_len, spec.decay)
                ch = rng.choice(int(lens.sum()), cw)
                pos = 0
                for r in range(m):
                    t = bytes(chars[c] for c in ch[pos:pos + lens[r]])
                    pos += int(lens[r])
                    if t not in seen:
                        seen.add(t)
                        toks.append(t)
                        got += 1
                        if got == n:
                            break
    assert len(toks) == V - 1
    toks.append(b"")  # EOS
    return pack(toks)


# ------------------------------------------------------------------ configs

@dataclasses.dataclass
class Workload:
    name: str
    description: str
    set_bytes: np.ndarray
    set_offsets: np.ndarray
    vocab_bytes: np.ndarray
    vocab_offsets: np.ndarray
    V: int
    batch: int
    steps: int
    dtype: str              # "f32" or "bf16"
    logit_std: float
    logit_seed: int
    # forest workloads (per-request sets): set_offsets index strings, and
    # request r owns strings set_index[r]:set_index[r+1]
    set_index: np.ndarray | None = None

    @property
    def K(self) -> int:
        return len(self.set_offsets) - 1


CONFIG_NAMES = {
    1: "tools-K100-V32000-B1-f32",
    2: "tools-K1000-V128000-B64-bf16",
    3: "icd-K10000-V152064-B256-bf16",
    4: "icd-K74719-V262144-B256-f32",
    5: "dynamic-256x(K300-2000)-V128000-B256-bf16",
}


def _tools_vocab(seed: int, V: int, max_len: int, stems: list[bytes]):
    spec = VocabSpec(V=V, max_len=max_len, substr_frac=0.30, run_frac=0.0, run_len=(2, 4),
                     upper=False, mixed=False)
    return byte_vocab(seed, spec, substr_src=stems)


def config(idx: int) -> Workload:
    """The five workloads: tool-name and ICD-style code sets with V = 32K..262K."""
    if idx == 1:
        names = tool_names(0, 100, 40)
        vb, vo = _tools_vocab(0, 32000, 12, tool_stems(0, 40))
        sb, so = pack(names)
        return Workload(CONFIG_NAMES[1], "K=100 tool names, V=32,000, 64 steps at B=1, fp32 N(0,1)",
                        sb, so, vb, vo, 32000, 1, 64, "f32", 1.0, 100)
    if idx == 2:
        names = tool_names(1, 1000, 200)
        vb, vo = _tools_vocab(1, 128000, 16, tool_stems(1, 200))
        sb, so = pack(names)
        return Workload(CONFIG_NAMES[2], "K=1,000 tool names, V=128,000, 128 steps at B=64, bf16 N(0,2)",
                        sb, so, vb, vo, 128000, 64, 128, "bf16", 2.0, 200)
    if idx == 3:
        codes = icd_codes(3, 10000, 4)
        spec = VocabSpec(V=152064, max_len=16, substr_frac=0.0, run_frac=0.20, run_len=(2, 4),
                         upper=True, mixed=False)
        vb, vo = byte_vocab(3, spec)
        sb, so = pack(codes)
        return Workload(CONFIG_NAMES[3], "K=10,000 codes, V=152,064, 16 steps at B=256, bf16 N(0,2)",
                        sb, so, vb, vo, 152064, 256, 16, "bf16", 2.0, 300)
    if idx == 4:
        codes = icd_codes(4, 74719, 3)
        spec = VocabSpec(V=262144, max_len=24, substr_frac=0.0, run_frac=0.0, run_len=(2, 4),
                         upper=True, mixed=True, decay=0.85)
        vb, vo = byte_vocab(4, spec)
        sb, so = pack(codes)
        return Workload(CONFIG_NAMES[4], "K=74,719 codes, V=262,144, 16 steps at B=256, fp32 N(0,1)",
                        sb, so, vb, vo, 262144, 256, 16, "f32", 1.0, 400)
    if idx == 5:
        return dynamic_requests(256)
    raise ValueError(f"unknown config {idx}")


def dynamic_requests(n_requests: int, pool_size: int = 50000, k_lo: int = 300,
                     k_hi: int = 2000) -> Workload:
    """Per-query sets: request r draws K_r ~ U[k_lo, k_hi] names from one pool."""
    pool = tool_names(5, pool_size, 2000)
    sets: list[bytes] = []
    index = [0]
    for r in range(n_requests):
        rng = SplitMix64(5000 + r)
        k = int(rng.integers(k_lo, k_hi + 1, 1)[0])
        pick = np.argsort(rng.random(len(pool)), kind="stable")[:k]
        sets.extend(pool[i] for i in np.sort(pick))
        index.append(len(sets))
    vb, vo = _tools_vocab(1, 128000, 16, tool_stems(1, 200))
    sb, so = pack(sets)
    return Workload(CONFIG_NAMES[5], f"{n_requests} requests with K~U[{k_lo},{k_hi}] names "
                    "from a 50,000-name pool, V=128,000, 32 steps, bf16 N(0,2)",
                    sb, so, vb, vo, 128000, n_requests, 32, "bf16", 2.0, 500,
                    set_index=np.array(index, dtype=np.int32))


def logits(w: Workload, step: int, device: str = "cpu", batch: int | None = None):
    """[batch, V] logits ~ N(0, std) for one decode step, seeded per step."""
    import torch
    B = w.batch if batch is None else batch
    g = torch.Generator(device=device)
    g.manual_seed(w.logit_seed + step)
    x = torch.randn(B, w.V, generator=g, device=device, dtype=torch.float32) * w.logit_std
    return x.to(torch.bfloat16) if w.dtype == "bf16" else x


# ------------------------------------------------------------ fixed formats

# The fixed formats of App. K's comparison, as patterns: '#' a decimal digit,
# 'x' a lowercase hexadecimal digit, 'y' one of 8 9 a b (the UUID version 4
# variant nibble), any other character itself.
FORMATS = {
    "YYYY-MM-DD": "####-##-##",
    "datetime": "####-##-##T##:##:##",
    "datetime.ms": "####-##-##T##:##:##.###",
    "UUID v4": "xxxxxxxx-xxxx-4xxx-yxxx-xxxxxxxxxxxx",
}


def format_classes(pattern: str) -> np.ndarray:
    """uint8 [L, 32] class bitmaps of a pattern (byte c of position i: bit c % 8 of [i, c // 8])."""
    sets = {"#": b"0123456789", "x": b"0123456789abcdef", "y": b"89ab"}
    out = np.zeros((len(pattern), 32), np.uint8)
    for i, ch in enumerate(pattern):
        for c in sets.get(ch, ch.encode()):
            out[i, c // 8] |= 1 << (c % 8)
    return out

