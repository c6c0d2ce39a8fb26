// sm_103a kernels of libtriemask.
//
// Mask compile (bit[n][v] for every node n and token v; Sec. 4.1-4.2):
//  k_mask_probe        one thread per node m finds every token whose bytes
//                      spell the last k edges into m (k = 1..lmax), to be set
//                      in the row of the node k edges above m: the
//                      Aho-Corasick outputs of Sec. 4.2 step 2 (a token whose
//                      characters end at the current node is recorded at the
//                      node |token| characters earlier), found by hashing each
//                      suffix of the node's 16-label window instead of by
//                      failure links, so every node is independent. It records
//                      the hits, sets the segment summary and runs beside
//                      k_mask_fill_beside; k_mask_probe_pair is the same with
//                      2 or 4 threads per node for small tries.
//  k_mask_fill_beside  writes every mask word once (zero), 16-byte evict-first
//                      stores, 8 KB per CTA: HBM-write bound.
//  k_mask_scatter      ORs the recorded hits into the zeroed mask.
//  (small masks: k_mask_fill, then k_mask_probe_pair ORing its own hits;
//  the no-allocation entry point: k_mask_fill, then k_mask_patch; the
//  pair-by-pair form for the A/B: k_mask_pairwise.)
// Decode (Sec. 2, Eq. 1; Sec. 4.2; App. H.3):
//  k_advance           delta*(s, bytes(token)) per request.
//  k_apply_vec         -inf into the logits of disallowed tokens: one warp per
//                      1024-token segment; a segment the summary says is empty
//                      is one TMA bulk copy of a -inf tile and reads no mask
//                      word, the rest 16-byte stores, the logits read only in
//                      16-byte chunks that hold an allowed token.
//  k_advance_apply_vec the advance of one step and the apply of the next.
// Sparse lists (valid[n] as CSR; App. H.5): k_rt_insert (per vocabulary),
// k_list_walk (count, then write), k_scan_*, k_apply_lists.
// Lazy rows (App. H.5): k_lazy_resolve, k_lazy_rows, k_lazy_gather.
//
// Every kernel is launched with programmatic stream serialization (PDL): it
// lets the next kernel in the stream launch at once and waits for the
// previous kernel (griddepcontrol.wait) before it touches memory that kernel
// may write or read. That wait is the hardware grid dependency, which always
// resolves because the previous grid never waits on this one. A kernel that
// runs beside the one before it (the fill beside the probe, the search of the
// small-mask form beside its fill) reads only data that was complete before
// that kernel started, and waits before it writes what the other one writes.
#include <stdint.h>

#include <algorithm>

#include <cuda_runtime.h>

#include "tm_internal.h"

namespace tmk {

namespace {

constexpr int32_t kDead = -1;
constexpr int32_t kFinished = -2;
constexpr int kMaxClimb = 16;  // suffix lengths kept in registers by the patch kernel

// ------------------------------------------------------------------ fill

constexpr int kFillThreads = 128;
constexpr int kFillVecs = 4;  // 16-byte stores per thread: one CTA writes 8 KB

// One CTA per 8 KB of mask, each warp store 512 contiguous bytes. On GB300 a
// grid of short-lived CTAs streams writes faster than a persistent grid-stride
// loop (7.4 vs 6.2-6.4 TB/s measured on a 439 MB mask). CTA 0 also writes the
// unaligned head and tail words.
__global__ void __launch_bounds__(kFillThreads) k_mask_fill(uint32_t *__restrict__ mask, int64_t n_words,
                                                            int64_t head) {
    pdl_launch_dependents();
    pdl_wait();  // an earlier kernel may still read the old mask
    uint4 *v = reinterpret_cast<uint4 *>(mask + head);
    const int64_t n4 = (n_words - head) >> 2;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    const int64_t base = int64_t(blockIdx.x) * (kFillThreads * kFillVecs) + threadIdx.x;
#pragma unroll
    for (int j = 0; j < kFillVecs; j++) {
        const int64_t i = base + j * kFillThreads;
        if (i < n4) v[i] = z;
    }
    if (blockIdx.x == 0) {
        if (threadIdx.x < head) mask[threadIdx.x] = 0u;
        const int64_t tail0 = head + (n4 << 2);
        if (threadIdx.x < n_words - tail0) mask[tail0 + threadIdx.x] = 0u;
    }
}

// The fill of the probe-fill-scatter form: launched while k_mask_probe runs,
// with evict-first stores so that the 0.4-4 GB stream does not flush the
// tables the probe has prefetched into L2.
// It needs no wait at entry (the probe let it launch only after every earlier
// kernel had completed); CTA 0 waits for the probe at its end, so this grid
// never completes before the probe and the scatter's wait covers both.
__global__ void __launch_bounds__(kFillThreads) k_mask_fill_beside(uint32_t *__restrict__ mask, int64_t n_words,
                                                                   int64_t head) {
    pdl_launch_dependents();
    uint4 *v = reinterpret_cast<uint4 *>(mask + head);
    const int64_t n4 = (n_words - head) >> 2;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    const int64_t base = int64_t(blockIdx.x) * (kFillThreads * kFillVecs) + threadIdx.x;
#pragma unroll
    for (int j = 0; j < kFillVecs; j++) {
        const int64_t i = base + j * kFillThreads;
        if (i < n4) __stcs(v + i, z);  // evict-first: keep the probe's tables in L2
    }
    if (blockIdx.x == 0) {
        if (threadIdx.x < head) mask[threadIdx.x] = 0u;
        const int64_t tail0 = head + (n4 << 2);
        if (threadIdx.x < n_words - tail0) mask[tail0 + threadIdx.x] = 0u;
        if (threadIdx.x == 0) pdl_wait();
    }
}

// ------------------------------------------------------------------ patch

constexpr int kPatchThreads = 128;

struct PatchArgs {
    const int32_t *parent;
    const uint8_t *label;
    const uint8_t *terminal;
    int32_t n_nodes;
    const uint64_t *ht_key;
    const int32_t *ht_val;
    uint32_t pairs_mask;  // number of slot pairs - 1
    const uint32_t *tok_off;
    const uint16_t *tok_len;
    const uint8_t *blob;
    const uint4 *ht_pay;  // per slot {token, min(len, 31) << 27 | blob offset / 16, bytes 0-3, 4-7}, or null
    int32_t lmax;
    uint32_t *mask;
    int64_t W;
    int32_t eos;
    int2 *hits;          // [n_nodes * kHitSlots] (row, token), probe-scatter form only
    uint8_t *hit_count;  // [n_nodes]
    const ulonglong2 *window;  // probe-scatter form: last 16 labels per node
    const uint8_t *depth16;    // min(depth, 16)
    const int4 *anc;           // [n * 4]: ancestors 1..16 levels up
    int32_t dup_keys;          // two tokens share a hash key
    ulonglong2 *trans;         // transition table (row, token) -> end node, or null
    uint32_t trans_mask;       // slots - 1
    int32_t trans_fill;        // the probe inserts every transition it finds
    unsigned long long *seg_any;  // [n_nodes * seg_words] tagged summary words (see DevTrie), or null
    uint32_t *seg_epoch;          // the device's current epoch, set to seg_tag by the probe
    uint32_t seg_tag;             // this compile's epoch
    int32_t seg_words;            // words per row of seg_any (segments of 1,024 tokens)
};

// Transition table: open addressing over 16-byte slots {key, end node};
// key = (row << 32 | token) + 1, 0 = empty. For a fixed trie the entries
// depend only on the vocabulary, so it is cleared and filled (by the probe)
// only when a compile uses another vocabulary than the one it holds. An entry
// that finds no slot within kTransProbes is left out (the advance then walks).
constexpr int kTransProbes = 32;

__device__ __forceinline__ uint64_t trans_key(int32_t row, int32_t t) {
    return ((uint64_t(uint32_t(row)) << 32) | uint32_t(t)) + 1ull;
}

__device__ __forceinline__ uint32_t trans_slot(uint64_t key, uint32_t mask) {
    const uint64_t z = key * 0x9E3779B97F4A7C15ull;
    return uint32_t(z >> 32) & mask;
}

__device__ __forceinline__ void trans_insert(ulonglong2 *tab, uint32_t mask, int32_t row, int32_t t,
                                             int32_t dest) {
    const uint64_t key = trans_key(row, t);
    uint32_t s = trans_slot(key, mask);
    for (int i = 0; i < kTransProbes; i++) {
        unsigned long long *k = reinterpret_cast<unsigned long long *>(&tab[s].x);
        const unsigned long long old = atomicCAS(k, 0ull, key);
        if (old == 0ull || old == key) {
            tab[s].y = uint64_t(uint32_t(dest));
            return;
        }
        s = (s + 1u) & mask;
    }
}

constexpr int kHitOverflow = 255;

// Masks up to this size are compiled in two kernels (fill, then a search that
// ORs its hits itself): at K = 100 (5.5 MB) 10.4 us against 16.4 us for three
// kernels. Larger ones by the search beside the fill and a scatter of the
// recorded hits: there the search starts only once the fill's last wave is
// running and no longer hides under it (K = 1,000, 184 MB: 37.2 us against
// 33.4 us).
constexpr int64_t kSmallMaskBytes = int64_t(32) << 20;

// Read-only arrays the probe reads, for a bulk L2 prefetch.
struct Prefetch {
    const void *ptr[10];
    uint64_t bytes[10];
    int count;
};

// CTA `part` of `nparts` asks the TMA unit to pull its slice of every array
// into L2 (cp.async.bulk.prefetch: asynchronous, no completion to wait for).
__device__ __forceinline__ void l2_prefetch_slice(const Prefetch &pf, int part, int nparts) {
    for (int i = 0; i < pf.count; i++) {
        const uint64_t n = pf.bytes[i] & ~uint64_t(15);
        const uint64_t per = ((n / uint64_t(nparts)) + 15) & ~uint64_t(15);
        const uint64_t a0 = per * uint64_t(part);
        if (a0 >= n) continue;
        const uint64_t len = n - a0 < per ? n - a0 : per;
        const char *base = static_cast<const char *>(pf.ptr[i]) + a0;
        for (uint64_t o = 0; o < len; o += 65536) {
            const uint32_t l = uint32_t(len - o < 65536 ? len - o : 65536);
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" :: "l"(base + o), "r"(l) : "memory");
        }
    }
}

// Byte i of a 16-byte window packed little-endian into four words, without
// dynamic register indexing.
__device__ __forceinline__ uint32_t byte_at(const uint32_t (&w)[4], int32_t i) {
    const int32_t q = i >> 2;
    const uint32_t v = q == 0 ? w[0] : (q == 1 ? w[1] : (q == 2 ? w[2] : w[3]));
    return (v >> ((i & 3) * 8)) & 0xFFu;
}

// Calls hit(t) for every token id t stored under `key` whose bytes equal the
// k-edge path ending at node m. lab (if not null) holds the path's labels,
// byte i = label of the edge i levels above m; otherwise the path is walked
// again. Probing visits aligned slot pairs.
template <typename Hit>
__device__ __forceinline__ void probe(const PatchArgs &a, uint64_t key, int32_t k, const uint32_t (*lab)[4],
                                      int32_t m, Hit hit) {
    uint32_t pair = uint32_t(key >> 1) & a.pairs_mask;
    for (uint32_t it = 0; it <= a.pairs_mask; it++) {
        const ulonglong2 kk = __ldg(reinterpret_cast<const ulonglong2 *>(a.ht_key) + pair);
#pragma unroll
        for (int q = 0; q < 2; q++) {
            if ((q == 0 ? kk.x : kk.y) == key) {
                const int32_t t = __ldg(a.ht_val + 2 * pair + q);
                if (int32_t(__ldg(a.tok_len + t)) == k) {
                    const uint8_t *tb = a.blob + __ldg(a.tok_off + t);
                    bool eq = true;
                    if (lab) {
                        for (int32_t j = 0; j < k && eq; j++) eq = (uint32_t(tb[j]) == byte_at(*lab, k - 1 - j));
                    } else {
                        int32_t y = m;
                        for (int32_t j = k - 1; j >= 0 && eq; j--) {
                            eq = y >= 0 && a.label[y] == tb[j];
                            y = a.parent[y];
                        }
                    }
                    if (eq) hit(t);
                }
            }
        }
        if (kk.y == 0ull) return;  // the pair is not full: the probe chain ends here
        pair = (pair + 1u) & a.pairs_mask;
    }
}

// Every allowed (row, token) pair whose path ends at node m: EOS at m if m is
// terminal (App. G.5), and every token whose bytes spell the last k edges
// into m, for the row of the node k edges above m (Sec. 4.2 step 2). Calls
// emit(row, t) for each.
template <typename Emit>
__device__ __forceinline__ void node_hits(const PatchArgs &a, int32_t m, Emit emit) {
    const int32_t lim = a.lmax < kMaxClimb ? a.lmax : kMaxClimb;
    // climb: labels (packed) and start nodes of the suffixes of length 1..16
    uint32_t lab[4] = {0u, 0u, 0u, 0u};
    int32_t anc[kMaxClimb];
    int32_t depth = 0;
    int32_t x = m;
#pragma unroll
    for (int k = 0; k < kMaxClimb; k++) {
        anc[k] = -1;
        if (k < lim && x >= 0) {
            const int32_t p = __ldg(a.parent + x);
            if (p >= 0) {
                lab[k >> 2] |= uint32_t(__ldg(a.label + x)) << ((k & 3) * 8);
                anc[k] = p;
                depth = k + 1;
            }
            x = p;
        }
    }
    if (__ldg(a.terminal + m)) emit(m, a.eos);
    // suffix hashes (Horner over byte+1 from the suffix's first byte); the
    // first probe of 8 suffixes is issued before any result is used
    uint64_t h = 0, pw = 1;
#pragma unroll
    for (int k0 = 0; k0 < kMaxClimb; k0 += 8) {
        if (k0 < depth) {
            uint64_t key[8];
            ulonglong2 first[8];
#pragma unroll
            for (int i = 0; i < 8; i++) {
                const int k = k0 + i;
                key[i] = 0ull;
                first[i] = make_ulonglong2(0ull, 0ull);
                if (k < depth) {
                    h += (uint64_t(byte_at(lab, k)) + 1ull) * pw;
                    pw *= kHashBase;
                    key[i] = hash_finish(h, uint32_t(k + 1));
                    first[i] = __ldg(reinterpret_cast<const ulonglong2 *>(a.ht_key) +
                                     (uint32_t(key[i] >> 1) & a.pairs_mask));
                }
            }
#pragma unroll
            for (int i = 0; i < 8; i++) {
                const int k = k0 + i;
                // the full probe only when the first pair holds the key or continues
                if (k < depth && (first[i].x == key[i] || first[i].y == key[i] || first[i].y != 0ull)) {
                    const int32_t row = anc[k];
                    probe(a, key[i], k + 1, &lab, m, [&](int32_t t) { emit(row, t); });
                }
            }
        }
    }
    // suffixes longer than the register window (deep tries with long tokens)
    if (a.lmax > kMaxClimb && depth == kMaxClimb) {
        int32_t y = anc[kMaxClimb - 1];
        for (int32_t k = kMaxClimb + 1; k <= a.lmax; k++) {
            const int32_t p = a.parent[y];
            if (p < 0) break;
            h += (uint64_t(a.label[y]) + 1ull) * pw;
            pw *= kHashBase;
            const int32_t row = p;
            probe(a, hash_finish(h, uint32_t(k)), k, nullptr, m, [&](int32_t t) { emit(row, t); });
            y = p;
        }
    }
}

// Payload of every slot of the token table (thread per slot): the token, its
// length (saturated at 31) and blob offset / 16 in one word, and its first 8
// bytes (the blob is zero-padded to 16 bytes per token). Empty slots: zero.
__global__ void k_vocab_pay(const uint64_t *__restrict__ key, const int32_t *__restrict__ val,
                            const uint16_t *__restrict__ tok_len, const uint32_t *__restrict__ tok_off,
                            const uint8_t *__restrict__ blob, int64_t S, uint4 *__restrict__ pay) {
    for (int64_t s = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; s < S; s += int64_t(gridDim.x) * blockDim.x) {
        uint4 p = make_uint4(0u, 0u, 0u, 0u);
        if (key[s]) {
            const int32_t t = val[s];
            const uint32_t len = tok_len[t], off = tok_off[t];
            const uint2 b = *reinterpret_cast<const uint2 *>(blob + off);
            p = make_uint4(uint32_t(t), (min(len, 31u) << 27) | (off >> 4), b.x, b.y);
        }
        pay[s] = p;
    }
}

// Slot of each key of a batch in the paired-slot table, -1 if absent, for
// vocabularies in which no two tokens share a key (so a key is stored at
// most once). f holds each key's first pair, already loaded. The keys of the
// batch advance together: each round checks every pending key's current pair
// and loads the next pair of those still pending (a full pair without the
// key); a pair that is not full ends the chain. The table is at most a
// quarter full, so every chain ends.
template <int G>
__device__ __forceinline__ void find_slots(const PatchArgs &a, const uint64_t (&key)[G], uint32_t pending,
                                           ulonglong2 (&f)[G], int32_t (&slot)[G]) {
    const ulonglong2 *pairs = reinterpret_cast<const ulonglong2 *>(a.ht_key);
    uint32_t pr[G];
#pragma unroll
    for (int g = 0; g < G; g++) {
        pr[g] = uint32_t(key[g] >> 1) & a.pairs_mask;
        slot[g] = -1;
    }
    for (uint32_t it = 0; pending && it <= a.pairs_mask; it++) {
#pragma unroll
        for (int g = 0; g < G; g++) {
            if (!((pending >> g) & 1u)) continue;
            if (f[g].x == key[g]) {
                slot[g] = int32_t(2 * pr[g]);
                pending &= ~(1u << g);
            } else if (f[g].y == key[g]) {
                slot[g] = int32_t(2 * pr[g] + 1);
                pending &= ~(1u << g);
            } else if (f[g].y == 0ull) {
                pending &= ~(1u << g);
            } else {
                pr[g] = (pr[g] + 1u) & a.pairs_mask;
            }
        }
#pragma unroll
        for (int g = 0; g < G; g++)
            if ((pending >> g) & 1u) f[g] = __ldg(pairs + pr[g]);
    }
}

// Element k of a register copy of 16 ancestors, without dynamic indexing.
__device__ __forceinline__ int32_t anc_at(const int4 (&an)[4], int k) {
    const int4 q = k < 4 ? an[0] : (k < 8 ? an[1] : (k < 12 ? an[2] : an[3]));
    const int r = k & 3;
    return r == 0 ? q.x : (r == 1 ? q.y : (r == 2 ? q.z : q.w));
}

// node_hits from the precomputed label window and ancestor table: one round
// of loads gives every suffix of length <= 16 and every start row. The 8
// suffixes of a batch are resolved as a wavefront: the first slot pair of all
// 8 keys, then the token ids of the matches, their lengths and offsets, then
// their bytes, each round issued for all candidates before any is used; keys
// not in their first pair follow their chains together (find_slots). In a
// vocabulary where some tokens share a key, a key whose first pair is full
// takes the sequential probe, which finds every token under it.
// One wavefront of node_hits_window: the suffixes of lengths k0 + 1 ..
// k0 + N (those within depth) of node m (N = 8, or 4 for the quad probe). h and pw hold the hash of the
// first k0 labels and B^k0 and are advanced over the batch; hit(i, row, t)
// is called for every token t that is the suffix of length k0 + i + 1
// (starting at row).
template <int N, typename Hit>
__device__ __forceinline__ void wavefront(const PatchArgs &a, int32_t m, int k0, int32_t depth,
                                          const uint32_t (&lab)[4], const int4 (&an)[4], uint64_t &h,
                                          uint64_t &pw, Hit hit) {
    const ulonglong2 *pairs = reinterpret_cast<const ulonglong2 *>(a.ht_key);
    uint64_t key[N];
    ulonglong2 first[N];
#pragma unroll
    for (int i = 0; i < N; i++) {
        key[i] = 0ull;
        first[i] = make_ulonglong2(0ull, 0ull);
        if (k0 + i < depth) {
            h += (uint64_t(byte_at(lab, k0 + i)) + 1ull) * pw;
            pw *= kHashBase;
            key[i] = hash_finish(h, uint32_t(k0 + i + 1));
            first[i] = __ldg(pairs + (uint32_t(key[i] >> 1) & a.pairs_mask));
        }
    }
    int32_t slot[N];  // slot of the key, -1 none
    uint32_t slow = 0;  // bit i: candidate i needs the sequential probe
    if (!a.dup_keys) {
        uint32_t pending = 0;
#pragma unroll
        for (int i = 0; i < N; i++)
            if (k0 + i < depth) pending |= 1u << i;
        find_slots<N>(a, key, pending, first, slot);
    } else {
#pragma unroll
        for (int i = 0; i < N; i++) {
            const bool m0 = first[i].x == key[i], m1 = first[i].y == key[i];
            const uint32_t pr = uint32_t(key[i] >> 1) & a.pairs_mask;
            slot[i] = (k0 + i < depth && (m0 || m1)) ? int32_t(2 * pr + (m0 ? 0 : 1)) : -1;
            if (k0 + i < depth && first[i].y != 0ull) {
                slow |= 1u << i;
                slot[i] = -1;
            }
        }
    }
    int32_t tid[N];
    int32_t tlen[N];
    uint32_t toff[N];
    uint4 tb[N];
    if (a.ht_pay) {
        // one load per match gives the token, its length, its offset
        // and its first 8 bytes; suffixes of 9-16 bytes then read the
        // rest from the blob
#pragma unroll
        for (int i = 0; i < N; i++) {
            const uint4 p = slot[i] >= 0 ? __ldg(a.ht_pay + slot[i]) : make_uint4(0u, 0u, 0u, 0u);
            tid[i] = slot[i] >= 0 ? int32_t(p.x) : -1;
            tlen[i] = slot[i] >= 0 ? int32_t(p.y >> 27) : -1;
            toff[i] = (p.y & 0x07FFFFFFu) << 4;
            tb[i] = make_uint4(p.z, p.w, 0u, 0u);
        }
#pragma unroll
        for (int i = 0; i < N; i++)
            if (k0 + i + 1 > 8 && tlen[i] == k0 + i + 1)
                tb[i] = __ldg(reinterpret_cast<const uint4 *>(a.blob + toff[i]));
    } else {
#pragma unroll
        for (int i = 0; i < N; i++) tid[i] = slot[i] >= 0 ? __ldg(a.ht_val + slot[i]) : -1;
#pragma unroll
        for (int i = 0; i < N; i++) {
            tlen[i] = tid[i] >= 0 ? int32_t(__ldg(a.tok_len + tid[i])) : -1;
            toff[i] = tid[i] >= 0 ? __ldg(a.tok_off + tid[i]) : 0u;
        }
        // token bytes: 16-byte aligned in the blob, which has 16 bytes of tail room
#pragma unroll
        for (int i = 0; i < N; i++)
            tb[i] = tlen[i] == k0 + i + 1 ? __ldg(reinterpret_cast<const uint4 *>(a.blob + toff[i]))
                                          : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int i = 0; i < N; i++) {
        const int k = k0 + i + 1;  // suffix length
        if (slow & (1u << i)) {
            probe(a, key[i], k, &lab, m, [&](int32_t t) { hit(i, anc_at(an, k - 1), t); });
        } else if (tlen[i] == k) {
            // token byte j must equal the label k-1-j levels above m
            const uint32_t tw[4] = {tb[i].x, tb[i].y, tb[i].z, tb[i].w};
            bool eq = true;
#pragma unroll
            for (int j = 0; j < kMaxClimb; j++)
                if (j < k) eq = eq && byte_at(tw, j) == byte_at(lab, k - 1 - j);
            if (eq) hit(i, anc_at(an, k - 1), tid[i]);
        }
    }
}

template <typename Hit>
__device__ __forceinline__ void wavefront8(const PatchArgs &a, int32_t m, int k0, int32_t depth,
                                           const uint32_t (&lab)[4], const int4 (&an)[4], uint64_t &h,
                                           uint64_t &pw, Hit hit) {
    wavefront<8>(a, m, k0, depth, lab, an, h, pw, hit);
}

template <typename Emit>
__device__ __forceinline__ void node_hits_window(const PatchArgs &a, int32_t m, Emit emit) {
    const ulonglong2 win = __ldg(a.window + m);
    int4 an[4];
#pragma unroll
    for (int q = 0; q < 4; q++) an[q] = __ldg(a.anc + int64_t(m) * 4 + q);
    const int32_t d16 = __ldg(a.depth16 + m);
    const int32_t depth = a.lmax < d16 ? a.lmax : d16;
    const uint32_t lab[4] = {uint32_t(win.x), uint32_t(win.x >> 32), uint32_t(win.y), uint32_t(win.y >> 32)};
    if (__ldg(a.terminal + m)) emit(m, a.eos);
    uint64_t h = 0, pw = 1;
#pragma unroll
    for (int k0 = 0; k0 < kMaxClimb; k0 += 8) {
        if (k0 < depth)
            wavefront8(a, m, k0, depth, lab, an, h, pw, [&](int, int32_t row, int32_t t) { emit(row, t); });
    }
    // suffixes longer than the window (deep tries with long tokens)
    if (a.lmax > kMaxClimb && depth == kMaxClimb) {
        int32_t y = anc_at(an, kMaxClimb - 1);  // start of the 16-byte suffix
        for (int32_t k = kMaxClimb + 1; k <= a.lmax; k++) {
            const int32_t p = a.parent[y];
            if (p < 0) break;
            h += (uint64_t(a.label[y]) + 1ull) * pw;
            pw *= kHashBase;
            const int32_t row = p;
            probe(a, hash_finish(h, uint32_t(k)), k, nullptr, m, [&](int32_t t) { emit(row, t); });
            y = p;
        }
    }
}

__device__ __forceinline__ void set_mask_bit(const PatchArgs &a, int32_t row, int32_t t) {
    atomicOr(a.mask + int64_t(row) * a.W + (t >> 5), 1u << (t & 31));
}

// The row's segment bit in the summary the apply reads first (a 1,024-token
// segment whose bit is clear holds no allowed token), set by the probe while
// the fill runs. A word that still carries an earlier compile's epoch is
// claimed with this compile's epoch and the bit in one compare-and-swap (a
// failed swap means another thread of this compile claimed it, so the loop
// runs at most twice); a word of this compile gets the bit unless it has it
// already (the rows near the root get thousands of hits in a few words).
__device__ __forceinline__ void set_seg_bit(const PatchArgs &a, int32_t row, int32_t t) {
    if (!a.seg_any) return;
    const int32_t g = t >> 10;
    unsigned long long *p = a.seg_any + int64_t(row) * a.seg_words + (g >> 5);
    const unsigned long long bit = 1ull << (g & 31);
    const unsigned long long tag = static_cast<unsigned long long>(a.seg_tag) << 32;
    unsigned long long old = *reinterpret_cast<volatile unsigned long long *>(p);
    while ((old & 0xFFFFFFFF00000000ull) != tag) {
        const unsigned long long prev = atomicCAS(p, old, tag | bit);
        if (prev == old) return;
        old = prev;
    }
    if (!(old & bit)) atomicOr(p, bit);
}

// set_seg_bit for up to G hits at once (tok < 0: none), in two rounds of
// memory operations for all of them instead of two per hit: the words are
// read, then claimed with compare-and-swaps or ORed; a swap that fails (a word
// another hit of the batch or another thread claimed first) retries alone.
template <int G>
__device__ __forceinline__ void set_seg_bits(const PatchArgs &a, const int32_t (&row)[G], const int32_t (&tok)[G]) {
    if (!a.seg_any) return;
    const unsigned long long tag = static_cast<unsigned long long>(a.seg_tag) << 32;
    unsigned long long *p[G];
    unsigned long long bit[G], old[G];
#pragma unroll
    for (int i = 0; i < G; i++) {
        const int32_t g = tok[i] >> 10;
        p[i] = tok[i] >= 0 ? a.seg_any + int64_t(row[i]) * a.seg_words + (g >> 5) : nullptr;
        bit[i] = 1ull << (g & 31);
    }
#pragma unroll
    for (int i = 0; i < G; i++) old[i] = p[i] ? *reinterpret_cast<volatile unsigned long long *>(p[i]) : 0ull;
    unsigned long long prev[G];
#pragma unroll
    for (int i = 0; i < G; i++) {
        prev[i] = old[i];
        if (!p[i]) continue;
        if ((old[i] & 0xFFFFFFFF00000000ull) != tag) prev[i] = atomicCAS(p[i], old[i], tag | bit[i]);
        else if (!(old[i] & bit[i])) atomicOr(p[i], bit[i]);
    }
#pragma unroll
    for (int i = 0; i < G; i++)
        if (p[i] && prev[i] != old[i]) set_seg_bit(a, row[i], tok[i]);
}

// Makes this compile's epoch the current one (the probe, before any apply of
// this compile can read the summary).
__device__ __forceinline__ void publish_seg_epoch(const PatchArgs &a) {
    if (a.seg_any && blockIdx.x == 0 && threadIdx.x == 0) *a.seg_epoch = a.seg_tag;
}

// Fill-then-patch form (two kernels): climbs and probes overlap the fill,
// the bits are set once the fill has completed.
__global__ void __launch_bounds__(kPatchThreads) k_mask_patch(PatchArgs a) {
    pdl_launch_dependents();
    bool waited = false;
    const int32_t stride = gridDim.x * blockDim.x;
    for (int32_t m = blockIdx.x * blockDim.x + threadIdx.x; m < a.n_nodes; m += stride) {
        node_hits(a, m, [&](int32_t row, int32_t t) {
            if (!waited) {
                pdl_wait();  // the fill of this mask must be complete
                waited = true;
            }
            set_mask_bit(a, row, t);
        });
    }
    if (!waited) pdl_wait();
}

// Probe-fill-scatter form (three kernels). k_mask_probe records up to
// kHitSlots hits per node in a buffer (count kHitOverflow: more hits, found
// again by the scatter). It waits for all earlier work at entry, prefetches
// its tables into L2 (its dependent loads then hit L2 while the fill
// saturates HBM) and only then lets the fill launch, which runs beside it.
__global__ void __launch_bounds__(kPatchThreads, 4) k_mask_probe(PatchArgs a, Prefetch pf) {
    pdl_wait();  // an earlier scatter may still read the hit buffer (an apply, the summary)
    if (threadIdx.x == 0) l2_prefetch_slice(pf, blockIdx.x, gridDim.x);
    pdl_launch_dependents();
    publish_seg_epoch(a);
    const int32_t stride = gridDim.x * blockDim.x;
    for (int32_t m = blockIdx.x * blockDim.x + threadIdx.x; m < a.n_nodes; m += stride) {
        int32_t c = 0;
        int2 *slot = a.hits + int64_t(m) * kHitSlots;
        node_hits_window(a, m, [&](int32_t row, int32_t t) {
            if (c < kHitSlots) slot[c] = make_int2(row, t);
            c++;
            set_seg_bit(a, row, t);
            if (a.trans_fill && t != a.eos) trans_insert(a.trans, a.trans_mask, row, t, m);
        });
        a.hit_count[m] = uint8_t(c > kHitSlots ? kHitOverflow : c);
    }
}

// k_mask_probe with L = 2 or 4 threads per node, for tries so small that one
// thread per node leaves most SMs idle and the probe's chain of dependent
// loads sets the compile time: lanes Lj .. Lj + L - 1 of a warp take node j
// of the warp's 32 / L, lane q the suffixes of lengths 16q/L + 1 .. 16(q+1)/L
// (lane 0 also EOS), each as one wavefront (the same instructions on every
// lane). The lanes then write their hits in node_hits_window's order (EOS,
// lengths 1..16) into the node's slots, so the hit buffer is that of
// k_mask_probe. Only for vocabularies with the per-slot payload (at most one
// token per suffix) and tokens of at most 16 bytes.
//
// kOr: the two-kernel form for small masks. The zero fill runs first; this
// kernel searches (read-only tables) while the fill runs, waits for it, and
// ORs its hits into the mask itself: no hit buffer, no scatter launch.
template <int L, bool kOr>
__global__ void __launch_bounds__(kPatchThreads, 3) k_mask_probe_pair(PatchArgs a, Prefetch pf) {
    constexpr int N = 16 / L;  // suffix lengths per lane
    if (!kOr) {
        pdl_wait();  // an earlier scatter may still read the hit buffer (an apply, the summary)
        if (threadIdx.x == 0) l2_prefetch_slice(pf, blockIdx.x, gridDim.x);
        publish_seg_epoch(a);
    }
    pdl_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int q = lane & (L - 1);  // this lane's share of the node: lengths k0 + 1 .. k0 + N
    const int k0 = N * q;
    const int64_t stride = int64_t(gridDim.x) * blockDim.x;
    const int64_t nl = L * int64_t(a.n_nodes);
    // every lane of a warp runs the same iterations (the shuffles below)
    for (int64_t w0 = int64_t(blockIdx.x) * blockDim.x + (threadIdx.x & ~31); w0 < nl; w0 += stride) {
        const int64_t t = w0 + lane;
        const bool valid = t < nl;
        const int32_t m = valid ? int32_t(t / L) : 0;
        int32_t found[N];
#pragma unroll
        for (int i = 0; i < N; i++) found[i] = -1;
        int4 an[4] = {};
        bool eos = false;
        if (valid) {
            const ulonglong2 win = __ldg(a.window + m);
#pragma unroll
            for (int g = 0; g < 4; g++) an[g] = __ldg(a.anc + int64_t(m) * 4 + g);
            const int32_t d16 = __ldg(a.depth16 + m);
            const int32_t depth = a.lmax < d16 ? a.lmax : d16;
            const uint32_t lab[4] = {uint32_t(win.x), uint32_t(win.x >> 32), uint32_t(win.y),
                                     uint32_t(win.y >> 32)};
            eos = q == 0 && __ldg(a.terminal + m);
            uint64_t h = 0, pw = 1;
#pragma unroll
            for (int j = 0; j < 16 - N; j++)  // the hash of the labels before this lane's first
                if (j < k0 && j < depth) {
                    h += (uint64_t(byte_at(lab, j)) + 1ull) * pw;
                    pw *= kHashBase;
                }
            if (k0 < depth)
                wavefront<N>(a, m, k0, depth, lab, an, h, pw, [&](int i, int32_t, int32_t tok) { found[i] = tok; });
        }
        int32_t c = eos ? 1 : 0;
#pragma unroll
        for (int i = 0; i < N; i++) c += found[i] >= 0 ? 1 : 0;
        // hits before this lane's within the node (lanes of a node are consecutive)
        int32_t before = 0, total = 0;
#pragma unroll
        for (int r = 0; r < L; r++) {
            const int32_t cr = __shfl_sync(0xffffffffu, c, (lane & ~(L - 1)) + r);
            before += r < q ? cr : 0;
            total += cr;
        }
        if (!valid) continue;
        if (kOr) pdl_wait();  // the fill of this mask (and of the transition table) is complete
        int2 *slot = a.hits + int64_t(m) * kHitSlots;
        int32_t s = before;
        auto rec = [&](int32_t row, int32_t tok) {
            if (kOr) {
                set_mask_bit(a, row, tok);
            } else {
                if (s < kHitSlots) slot[s] = make_int2(row, tok);
                s++;
            }
            if (a.trans_fill && tok != a.eos) trans_insert(a.trans, a.trans_mask, row, tok, m);
        };
        if (eos) rec(m, a.eos);
#pragma unroll
        for (int i = 0; i < N; i++)
            if (found[i] >= 0) rec(anc_at(an, k0 + i), found[i]);
        if (!kOr) {  // the summary bits of the lane's hits, together
            int32_t hr[N + 1], ht[N + 1];
#pragma unroll
            for (int i = 0; i < N; i++) {
                hr[i] = anc_at(an, k0 + i);
                ht[i] = found[i];
            }
            hr[N] = m;
            ht[N] = eos ? a.eos : -1;
            set_seg_bits<N + 1>(a, hr, ht);
        }
        if (!kOr && q == 0) a.hit_count[m] = uint8_t(total > kHitSlots ? kHitOverflow : total);
    }
}

// Sets the recorded bits after the fill (which completes after the probe).
__global__ void __launch_bounds__(kPatchThreads, 4) k_mask_scatter(PatchArgs a) {
    pdl_launch_dependents();
    pdl_wait();  // fill complete, and through it the probe
    const int32_t stride = gridDim.x * blockDim.x;
    for (int32_t m = blockIdx.x * blockDim.x + threadIdx.x; m < a.n_nodes; m += stride) {
        auto emit = [&](int32_t row, int32_t t) { set_mask_bit(a, row, t); };
        const int32_t c = a.hit_count[m];
        if (c == kHitOverflow) {
            node_hits_window(a, m, emit);
            continue;
        }
        const int2 *slot = a.hits + int64_t(m) * kHitSlots;
        for (int32_t i = 0; i < c; i++) {
            const int2 hv = slot[i];
            emit(hv.x, hv.y);
        }
    }
}

// ------------------------------------------------------------------ advance

constexpr int kAdvanceThreads = 128;

// End node of (row, token) from the transition table; false if absent.
__device__ __forceinline__ bool trans_lookup(const ulonglong2 *__restrict__ tab, uint32_t mask, int32_t row,
                                             int32_t t, int32_t *dest) {
    const uint64_t key = trans_key(row, t);
    uint32_t s = trans_slot(key, mask);
    for (int i = 0; i < kTransProbes; i++) {
        const ulonglong2 e = __ldg(tab + s);
        if (e.x == key) {
            *dest = int32_t(uint32_t(e.y));
            return true;
        }
        if (e.x == 0ull) return false;
        s = (s + 1u) & mask;
    }
    return false;
}

struct AdvanceArgs {
    const int32_t *first_child;
    const uint32_t *child_bits;
    const uint8_t *terminal;
    int32_t n_nodes;
    const uint32_t *tok_off;
    const uint16_t *tok_len;
    const uint8_t *blob;
    int32_t V;
    const ulonglong2 *trans;  // transition table of this vocabulary, or null
    uint32_t trans_mask;
};

// delta*(s, bytes(v)) (Sec. 2, Eq. 1) with the FINISHED / DEAD rules.
__device__ __forceinline__ int32_t advance_one(const AdvanceArgs &a, int32_t s, int32_t v) {
    const int32_t eos = a.V - 1;
    if (s == kDead) return kDead;
    if (v < 0 || v >= a.V) return kDead;
    if (s == kFinished) return (v == eos) ? kFinished : kDead;
    if (s < 0 || s >= a.n_nodes) return kDead;
    if (v == eos) return a.terminal[s] ? kFinished : kDead;
    int32_t nxt;
    if (a.trans && trans_lookup(a.trans, a.trans_mask, s, v, &nxt)) return nxt;  // recorded by the compile
    const int32_t L = a.tok_len[v];
    if (L <= 0) return kDead;
    const uint8_t *p = a.blob + a.tok_off[v];
    int32_t x = s;
    for (int32_t j = 0; j < L; j++) {
        const uint32_t c = p[j];
        const uint4 *cb = reinterpret_cast<const uint4 *>(a.child_bits + int64_t(x) * 8);
        const uint4 lo = cb[0], hi = cb[1];
        const int32_t fc = a.first_child[x];
        const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
        const uint32_t wi = c >> 5, bit = c & 31u;
        uint32_t below = 0, cur = 0;
#pragma unroll
        for (uint32_t i = 0; i < 8; i++) {
            below += (i < wi) ? __popc(w[i]) : 0u;
            cur = (i == wi) ? w[i] : cur;
        }
        if (!((cur >> bit) & 1u)) return kDead;
        x = fc + int32_t(below + __popc(cur & ((1u << bit) - 1u)));
    }
    return x;
}

// states_out[b] = delta*(states_in[b], tokens[b]); states_out may equal
// states_in (in place). Every move into DEAD from a non-DEAD state counts.
__global__ void __launch_bounds__(kAdvanceThreads) k_advance(AdvanceArgs a, const int32_t *states_in,
                                                             int32_t *states_out, const int32_t *__restrict__ tokens,
                                                             int32_t B, int32_t *__restrict__ err) {
    pdl_launch_dependents();
    pdl_wait();  // states / tokens come from earlier kernels
    const int32_t b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    const int32_t s = states_in[b];
    const int32_t nxt = advance_one(a, s, tokens[b]);
    if (nxt == kDead && s != kDead && err) atomicAdd(err, 1);
    states_out[b] = nxt;
}

// ------------------------------------------------------------ pairwise form
// The compile as the pair-by-pair evaluation of the definition (Sec. 4.1,
// App. G.5): bit[n][v] = 1 iff v is not EOS, has bytes, and every byte of v
// finds a child walking down from n; bit[n][EOS] = terminal(n). One warp per
// (node, 32 mask words): lane l tests token 32 i + l of word i by walking its
// bytes (child-label set + first child, as the advance does), a warp ballot
// assembles the word, and lane i keeps word i for one coalesced 128-byte
// store. Kept as the measured alternative to the suffix search: its cost is
// one walk per (node, token) pair, N * V walks, instead of a few probes per
// node.
constexpr int kPairwiseThreads = 256;

__device__ __forceinline__ bool token_walks(const AdvanceArgs &a, int32_t n, int32_t t) {
    const int32_t L = __ldg(a.tok_len + t);
    if (L <= 0) return false;
    const uint8_t *p = a.blob + __ldg(a.tok_off + t);
    int32_t x = n;
    for (int32_t j = 0; j < L; j++) {
        const uint32_t c = __ldg(p + j);
        const uint32_t wv = __ldg(a.child_bits + int64_t(x) * 8 + (c >> 5));
        const uint32_t bit = c & 31u;
        if (!((wv >> bit) & 1u)) return false;
        uint32_t below = __popc(wv & ((1u << bit) - 1u));
        for (uint32_t i = 0; i < (c >> 5); i++) below += __popc(__ldg(a.child_bits + int64_t(x) * 8 + i));
        x = __ldg(a.first_child + x) + int32_t(below);
    }
    return true;
}

__global__ void __launch_bounds__(kPairwiseThreads) k_mask_pairwise(AdvanceArgs a, uint32_t *__restrict__ mask,
                                                                    int64_t W, int64_t chunks) {
    pdl_launch_dependents();
    pdl_wait();  // an earlier kernel may still read the old mask
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = (int64_t(gridDim.x) * blockDim.x) >> 5;
    const int64_t tasks = int64_t(a.n_nodes) * chunks;
    const int32_t eos = a.V - 1;
    for (int64_t task = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; task < tasks; task += nwarps) {
        const int32_t n = int32_t(task / chunks);
        const int64_t w0 = (task - int64_t(n) * chunks) * 32;
        const bool term = __ldg(a.terminal + n) != 0;
        uint32_t out = 0u;
        for (int i = 0; i < 32 && w0 + i < W; i++) {  // uniform across the warp
            const int64_t t = (w0 + i) * 32 + lane;
            bool ok = false;
            if (t < eos) ok = token_walks(a, n, int32_t(t));
            else if (t == eos) ok = term;
            const uint32_t word = __ballot_sync(0xffffffffu, ok);
            if (lane == i) out = word;
        }
        if (w0 + lane < W) mask[int64_t(n) * W + w0 + lane] = out;
    }
}

// ------------------------------------------------------------------ apply

constexpr int kApplyThreads = 256;

// Mask word of (state, word index w): the node's row, or {EOS} for FINISHED,
// DEAD and ids that are not nodes.
__device__ __forceinline__ uint32_t row_word(const uint32_t *__restrict__ mask, int32_t s,
                                             int32_t n_nodes, int64_t W, int64_t w, int32_t eos) {
    if (w >= W) return 0u;
    if (s >= 0 && s < n_nodes) return __ldg(mask + int64_t(s) * W + w);
    return (w == (eos >> 5)) ? (1u << (eos & 31)) : 0u;
}

// The current summary epoch (read once a kernel's wait for earlier work is done).
__device__ __forceinline__ uint32_t seg_epoch_now(const SegRef &sg) { return sg.words ? __ldg(sg.epoch) : 0u; }

// Mask word w of state s's row, reading the row only when the segment
// summary (if any) says segment seg holds an allowed token: a summary word
// that does not carry the current epoch ep says no segment of it does.
__device__ __forceinline__ uint32_t seg_row_word(const uint32_t *__restrict__ mask, const SegRef &sg, uint32_t ep,
                                                 int32_t s, int32_t n_nodes, int64_t W, int32_t seg, int64_t w,
                                                 int32_t eos) {
    if (sg.words && s >= 0 && s < n_nodes) {
        const unsigned long long v = __ldg(sg.words + int64_t(s) * sg.per_row + (seg >> 5));
        const uint32_t bits = uint32_t(v >> 32) == ep ? uint32_t(v) : 0u;
        if (!((bits >> (seg & 31)) & 1u)) return 0u;
    }
    return row_word(mask, s, n_nodes, W, w, eos);
}

// -inf pattern of 16 bytes of logits.
template <int kElt>
__device__ __forceinline__ uint4 ninf16() {
    return (kElt == 2) ? make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u)
                       : make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
}

// Fills the CTA's -inf tile (one segment of logits) and makes it visible to
// the bulk copies. Must be called by every thread of the CTA.
template <int kElt>
__device__ __forceinline__ void init_ninf_tile(uint4 *tile) {
    constexpr int kSegChunks = 1024 / (16 / kElt);
    for (int i = threadIdx.x; i < kSegChunks; i += blockDim.x) tile[i] = ninf16<kElt>();
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // tile visible to the bulk copies
    __syncthreads();
}

// Writes one 1024-token segment of a logits row (by one warp; lane l holds
// mask word l of the segment). A segment without an allowed token is one TMA
// bulk copy of the -inf tile; otherwise the lanes write 16-byte chunks,
// reading the logits only in chunks that hold an allowed token. Stores use an
// L2 evict-first policy: the logits stream must not flush the trie tables.
template <int kElt>
__device__ __forceinline__ void write_segment(uint4 *__restrict__ row, int64_t c0, int64_t row_chunks,
                                              uint32_t word, int lane, const uint4 *tile) {
    constexpr int kPer = 16 / kElt;            // tokens per 16-byte chunk
    constexpr int kChunks = 1024 / kPer / 32;  // chunks per lane per segment
    constexpr int kSegChunks = 1024 / kPer;
    if (!__any_sync(0xffffffffu, word != 0u)) {
        if (lane == 0) {
            const int64_t nch = (row_chunks - c0 < kSegChunks) ? row_chunks - c0 : kSegChunks;
            const uint32_t ts = static_cast<uint32_t>(__cvta_generic_to_shared(tile));
            uint64_t policy;
            asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;"
                         :: "l"(row + c0), "r"(ts), "r"(uint32_t(nch * 16)), "l"(policy) : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");  // tile read before exit
        }
        return;
    }
    const uint4 ninf = ninf16<kElt>();
#pragma unroll
    for (int j = 0; j < kChunks; j++) {
        const int q = j * 32 + lane;  // chunk within the segment
        const uint32_t wv = __shfl_sync(0xffffffffu, word, (q * kPer) >> 5);
        const uint32_t bits = (wv >> ((q * kPer) & 31)) & ((1u << kPer) - 1u);
        const int64_t chunk = c0 + q;
        if (chunk >= row_chunks) continue;
        if (bits == 0u) {
            __stcs(row + chunk, ninf);
        } else {
            const uint4 x = row[chunk];
            uint32_t e[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int i = 0; i < 4; i++) {
                if (kElt == 4) {
                    if (!((bits >> i) & 1u)) e[i] = 0xFF800000u;
                } else {
                    if (!((bits >> (2 * i)) & 1u)) e[i] = (e[i] & 0xFFFF0000u) | 0xFF80u;
                    if (!((bits >> (2 * i + 1)) & 1u)) e[i] = (e[i] & 0x0000FFFFu) | 0xFF800000u;
                }
            }
            __stcs(row + chunk, make_uint4(e[0], e[1], e[2], e[3]));
        }
    }
}

// kElt = 2 (bf16) or 4 (fp32). Requires V % (16 / kElt) == 0 and a 16-byte
// aligned logits base, so that every row starts on a 16-byte boundary.
// One warp per 1024-token segment of a row (one mask word per lane).
template <int kElt>
__global__ void __launch_bounds__(kApplyThreads) k_apply_vec(uint4 *__restrict__ logits,
                                                             const uint32_t *__restrict__ mask,
                                                             const int32_t *__restrict__ states, int32_t B,
                                                             int32_t V, int64_t W, int32_t n_nodes,
                                                             int32_t segs, SegRef sg) {
    constexpr int kSegChunks = 1024 / (16 / kElt);
    __shared__ __align__(128) uint4 tile[kSegChunks];
    init_ninf_tile<kElt>(tile);
    pdl_launch_dependents();
    pdl_wait();  // logits and states come from earlier kernels
    const int lane = threadIdx.x & 31;
    const int32_t item = int32_t(blockIdx.x) * (kApplyThreads / 32) + (threadIdx.x >> 5);
    if (item >= B * segs) return;  // uniform per warp
    const int32_t b = item / segs, seg = item - b * segs;
    const uint32_t word = seg_row_word(mask, sg, seg_epoch_now(sg), __ldg(states + b), n_nodes, W, seg,
                                       int64_t(seg) * 32 + lane, V - 1);
    const int64_t row_chunks = int64_t(V) / (16 / kElt);
    write_segment<kElt>(logits + int64_t(b) * row_chunks, int64_t(seg) * kSegChunks, row_chunks, word, lane,
                        tile);
}

// Advance, then apply, in one launch (one decode step once the sampler has
// picked tokens[b] for the previous logits): states_out[b] = delta*(states_in[b],
// tokens[b]), and logits[b] (the next step's) are masked by the row of
// states_out[b]. CTA (row b, part p) covers segments 8p .. 8p + 7 of row b,
// one warp each; its thread 0 computes the row's new state once for the CTA
// (shared memory), and the CTA of part 0 stores it and counts a move into
// DEAD.
template <int kElt>
__global__ void __launch_bounds__(kApplyThreads) k_advance_apply_vec(AdvanceArgs aa, uint4 *__restrict__ logits,
                                                                     const uint32_t *__restrict__ mask,
                                                                     const int32_t *__restrict__ states_in,
                                                                     const int32_t *__restrict__ tokens,
                                                                     int32_t *__restrict__ states_out,
                                                                     int32_t *__restrict__ err, int32_t B,
                                                                     int64_t W, int32_t segs, int32_t parts,
                                                                     SegRef sg) {
    constexpr int kSegChunks = 1024 / (16 / kElt);
    __shared__ __align__(128) uint4 tile[kSegChunks];
    __shared__ int32_t next_state;
    __shared__ uint32_t epoch;
    pdl_launch_dependents();
    const int32_t b = int32_t(blockIdx.x) / parts, part = int32_t(blockIdx.x) - b * parts;
    for (int i = threadIdx.x; i < kSegChunks; i += blockDim.x) tile[i] = ninf16<kElt>();
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // tile visible to the bulk copies
    if (threadIdx.x == 0) {
        pdl_wait();  // states and tokens come from earlier kernels
        epoch = seg_epoch_now(sg);  // loaded beside the advance's chain
        const int32_t s = __ldg(states_in + b);
        const int32_t nxt = advance_one(aa, s, __ldg(tokens + b));
        next_state = nxt;
        if (part == 0) {
            states_out[b] = nxt;
            if (nxt == kDead && s != kDead && err) atomicAdd(err, 1);
        }
    }
    __syncthreads();
    pdl_wait();  // logits come from earlier kernels
    const int lane = threadIdx.x & 31;
    const int32_t seg = part * (kApplyThreads / 32) + int32_t(threadIdx.x >> 5);
    if (seg >= segs) return;  // uniform per warp
    const uint32_t word = seg_row_word(mask, sg, epoch, next_state, aa.n_nodes, W, seg,
                                       int64_t(seg) * 32 + lane, aa.V - 1);
    const int64_t row_chunks = int64_t(aa.V) / (16 / kElt);
    write_segment<kElt>(logits + int64_t(b) * row_chunks, int64_t(seg) * kSegChunks, row_chunks, word, lane,
                        tile);
}

// ---------------------------------------------------------------- valid lists
// Sparse form of the masks (the valid[n] lists the paper stores, Sec. 4.2 and
// App. H.5): for every node, the ids of its allowed tokens (EOS included at
// terminal nodes) in no particular order, as CSR offsets[N+1] + tokens.

// Exclusive scan of the row counts into int64 offsets, in three passes over
// tiles of kScanTile counts: tile sums, a scan of the tile sums by one CTA,
// and the offsets of every row.
constexpr int kScanThreads = 1024;
constexpr int kScanPer = 4;
constexpr int kScanTile = kScanThreads * kScanPer;

__device__ __forceinline__ int64_t block_exclusive_scan(int64_t v, int64_t *smem_warp, int64_t *total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int64_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) smem_warp[wid] = x;
    __syncthreads();
    if (wid == 0) {
        int64_t w = lane < int(blockDim.x >> 5) ? smem_warp[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        smem_warp[lane] = w;  // inclusive scan of the warp totals
    }
    __syncthreads();
    const int64_t warp_base = wid ? smem_warp[wid - 1] : 0;
    *total = smem_warp[(blockDim.x >> 5) - 1];
    __syncthreads();
    return warp_base + x - v;
}

__global__ void __launch_bounds__(kScanThreads) k_scan_tiles(const int32_t *__restrict__ cnt, int32_t n,
                                                             int64_t *__restrict__ tile_sum) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ int64_t sw[32];
    const int64_t base = int64_t(blockIdx.x) * kScanTile + int64_t(threadIdx.x) * kScanPer;
    int64_t v = 0;
    if (base + kScanPer <= n) {
        const int4 q = *reinterpret_cast<const int4 *>(cnt + base);
        v = int64_t(q.x) + q.y + q.z + q.w;
    } else {
#pragma unroll
        for (int j = 0; j < kScanPer; j++)
            if (base + j < n) v += cnt[base + j];
    }
    int64_t total;
    block_exclusive_scan(v, sw, &total);
    if (threadIdx.x == 0) tile_sum[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kScanThreads) k_scan_tile_sums(int64_t *__restrict__ tile_sum, int32_t n_tiles,
                                                                 int64_t *__restrict__ grand_total) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ int64_t sw[32];
    int64_t carry = 0;
    for (int32_t t0 = 0; t0 < n_tiles; t0 += kScanThreads) {
        const int32_t i = t0 + threadIdx.x;
        const int64_t v = i < n_tiles ? tile_sum[i] : 0;
        int64_t total;
        const int64_t ex = block_exclusive_scan(v, sw, &total);
        if (i < n_tiles) tile_sum[i] = carry + ex;
        carry += total;
    }
    if (threadIdx.x == 0) *grand_total = carry;
}

// Exclusive sums of the row counts, written one place up: off[0] = 0 and
// off[i + 1] = cnt[0] + .. + cnt[i - 1], the first position of row i. The
// writing walk then claims row i's positions from off[i + 1], which ends at
// cnt[0] + .. + cnt[i]: the offsets array is complete when the walk is.
__global__ void __launch_bounds__(kScanThreads) k_scan_rows(const int32_t *__restrict__ cnt, int32_t n,
                                                            const int64_t *__restrict__ tile_off,
                                                            int64_t *__restrict__ off) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ int64_t sw[32];
    const int64_t base = int64_t(blockIdx.x) * kScanTile + int64_t(threadIdx.x) * kScanPer;
    int64_t c[kScanPer];
    int64_t v = 0;
    if (base + kScanPer <= n) {
        const int4 q = *reinterpret_cast<const int4 *>(cnt + base);
        c[0] = q.x, c[1] = q.y, c[2] = q.z, c[3] = q.w;
    } else {
#pragma unroll
        for (int j = 0; j < kScanPer; j++) c[j] = base + j < n ? cnt[base + j] : 0;
    }
#pragma unroll
    for (int j = 0; j < kScanPer; j++) v += c[j];
    int64_t total;
    int64_t run = tile_off[blockIdx.x] + block_exclusive_scan(v, sw, &total);
#pragma unroll
    for (int j = 0; j < kScanPer; j++) {
        if (base + j < n) off[base + j + 1] = run;
        run += c[j];
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) off[0] = 0;
}

// ------------------------------------------------------------ list walk
// The valid lists from the reversed-token trie (the vocabulary's tokens read
// backwards, as an edge table): from every node m the walk follows the labels
// above m, the label into m first. After j + 1 steps it stands on the
// reversed prefix of every token that ends with the last j + 1 edges into m;
// a token ending there is allowed at the node j + 1 levels above m (Sec. 4.2
// step 2: an output found at the current node belongs to the node |token|
// characters up). The walk stops at the first label no token continues with,
// so it costs one exact edge lookup per step and no hashing of whole
// suffixes. Two walks: the first counts the entries of every row, the second
// writes them at positions claimed from the rows' offsets (order within a row
// unspecified).

struct WalkArgs {
    const uint8_t *terminal;
    const ulonglong2 *window;  // last 16 labels into each node (byte i = i levels up)
    const uint8_t *depth16;    // min(depth, 16)
    const int32_t *anc;        // [n * 16]: ancestors 1..16 levels up
    const int32_t *parent;
    const uint8_t *label;
    int32_t n_nodes;
    int32_t lmax;              // min(longest token, trie depth)
    int32_t eos;
    const uint4 *edge;         // {(parent << 8 | byte) + 1, child, token or -1, 0}; key 0 = empty
    uint32_t edge_mask;        // slots - 1
    uint32_t edge_shift;       // 32 - log2(slots)
    const int32_t *tok_next;   // tokens with the same bytes, or null
    int32_t *count;            // [n] entries per row (counting walk)
    unsigned long long *off;   // [n + 1]: off[i + 1] = next position of row i (writing walk)
    int32_t *toks;
    int32_t *ends;             // [tok_cap]: the node each entry's token leads to (FINISHED for EOS)
    unsigned long long tok_cap;  // entries toks holds (a write past it is dropped)
};

constexpr int kWalkThreads = 256;  // also the 256 root edges each CTA stages

__device__ __forceinline__ uint32_t edge_slot(uint32_t key, uint32_t shift) { return (key * 0x9E3779B1u) >> shift; }

// The edge of reversed-trie node x for byte c (e.y = child, e.z = token
// ending at the child or -1); false if there is none. The table is at most
// half full, so an empty slot ends every probe sequence.
__device__ __forceinline__ bool rt_step(const uint4 *__restrict__ edge, uint32_t mask, uint32_t shift, int32_t x,
                                        uint32_t c, uint4 *out) {
    const uint32_t key = ((uint32_t(x) << 8) | c) + 1u;
    uint32_t s = edge_slot(key, shift);
    for (uint32_t i = 0; i <= mask; i++) {
        const uint4 e = __ldg(edge + s);
        if (e.x == key) {
            *out = e;
            return true;
        }
        if (e.x == 0u) return false;
        s = (s + 1u) & mask;
    }
    return false;
}

// Inserts the edge into every node c > 0 of a reversed-token trie.
__global__ void k_rt_insert(const int32_t *__restrict__ parent, const uint8_t *__restrict__ label,
                            const int32_t *__restrict__ token, int32_t n, uint4 *__restrict__ edge, uint32_t mask,
                            uint32_t shift) {
    for (int32_t c = 1 + blockIdx.x * blockDim.x + threadIdx.x; c < n; c += gridDim.x * blockDim.x) {
        const uint32_t key = ((uint32_t(parent[c]) << 8) | label[c]) + 1u;
        uint32_t s = edge_slot(key, shift);
        for (uint32_t i = 0; i <= mask; i++) {  // keys are distinct: the first empty slot takes it
            if (atomicCAS(&edge[s].x, 0u, key) == 0u) {
                edge[s].y = uint32_t(c);
                edge[s].z = uint32_t(token[c]);
                break;
            }
            s = (s + 1u) & mask;
        }
    }
}

// Every (row, token) entry whose path ends at node m: EOS at m if m is
// terminal (App. G.5), then the tokens met by the walk (row = the node as
// many levels above m as the token has bytes). root[c] = {child, token} of
// the reversed trie's root for byte c.
template <typename Tok>
__device__ __forceinline__ void walk_node(const WalkArgs &a, const int2 *root, int32_t m, Tok tok) {
    if (__ldg(a.terminal + m)) tok(m, a.eos, kFinished);
    const int32_t d16 = __ldg(a.depth16 + m);
    const int32_t lim = a.lmax < d16 ? a.lmax : d16;
    if (lim <= 0) return;
    const ulonglong2 win = __ldg(a.window + m);
    const int32_t *up = a.anc + int64_t(m) * 16;
    const int2 r0 = root[uint32_t(win.x) & 0xFFu];
    int32_t x = r0.x;
    if (x < 0) return;
    if (r0.y >= 0) tok(__ldg(up), r0.y, m);
    for (int32_t j = 1; j < lim; j++) {
        const uint32_t c = uint32_t((j < 8 ? win.x >> (8 * j) : win.y >> (8 * (j - 8))) & 0xFFu);
        uint4 e;
        if (!rt_step(a.edge, a.edge_mask, a.edge_shift, x, c, &e)) return;
        x = int32_t(e.y);
        if (int32_t(e.z) >= 0) tok(__ldg(up + j), int32_t(e.z), m);
    }
    // tokens longer than the 16-label window, in a trie deeper than 16
    if (lim == 16 && a.lmax > 16) {
        int32_t y = __ldg(up + 15);  // 16 levels above m: its label is the 17th
        for (int32_t j = 16; j < a.lmax; j++) {
            const int32_t p = __ldg(a.parent + y);
            if (p < 0) return;
            uint4 e;
            if (!rt_step(a.edge, a.edge_mask, a.edge_shift, x, __ldg(a.label + y), &e)) return;
            x = int32_t(e.y);
            if (int32_t(e.z) >= 0) tok(p, int32_t(e.z), m);
            y = p;
        }
    }
}

// kWrite = false: count[row] += 1 for every entry; true: the entry's token
// at the position claimed from off[row + 1]. Persistent grid (each CTA first
// stages the reversed trie's 256 root edges in shared memory), a node per
// thread in a grid-stride loop.
template <bool kWrite>
__global__ void __launch_bounds__(kWalkThreads) k_list_walk(WalkArgs a) {
    __shared__ int2 root[256];
    {
        uint4 e;
        root[threadIdx.x] = rt_step(a.edge, a.edge_mask, a.edge_shift, 0, threadIdx.x, &e)
                                ? make_int2(int32_t(e.y), int32_t(e.z))
                                : make_int2(-1, -1);
    }
    __syncthreads();
    pdl_launch_dependents();
    pdl_wait();  // counts zeroed, or offsets scanned, by the previous kernels
    auto emit = [&](int32_t row, int32_t t, int32_t end) {
        if (kWrite) {
            const unsigned long long p = atomicAdd(a.off + row + 1, 1ull);
            if (p < a.tok_cap) {
                a.toks[p] = t;
                a.ends[p] = end;
            }
        } else {
            atomicAdd(a.count + row, 1);
        }
    };
    auto tok = [&](int32_t row, int32_t t, int32_t end) {
        emit(row, t, end);
        if (a.tok_next)
            for (int32_t u = __ldg(a.tok_next + t); u >= 0; u = __ldg(a.tok_next + u)) emit(row, u, end);
    };
    const int32_t stride = gridDim.x * blockDim.x;
    for (int32_t m = blockIdx.x * blockDim.x + threadIdx.x; m < a.n_nodes; m += stride) walk_node(a, root, m, tok);
}
// Apply from the lists: CTA (row b, part p) covers 8 segments (8,192 tokens).
// It rebuilds their 256 mask words in shared memory from the row's list and
// writes them like k_apply_vec (kVec) or one logit per thread (any V and
// alignment). With kAdvance the row's state is first moved by its token
// (thread 0; the CTA of part 0 stores it and counts a move into DEAD): the
// advance of one decode step and the apply of the next in one launch.
template <int kElt, bool kVec, bool kAdvance>
__global__ void __launch_bounds__(kApplyThreads) k_apply_lists(void *__restrict__ logits,
                                                               const int64_t *__restrict__ off,
                                                               const int32_t *__restrict__ toks, AdvanceArgs aa,
                                                               const int32_t *__restrict__ states,
                                                               const int32_t *__restrict__ tokens,
                                                               int32_t *__restrict__ states_out,
                                                               int32_t *__restrict__ err, int32_t B, int32_t V,
                                                               int32_t n_nodes, int32_t parts,
                                                               const int32_t *__restrict__ ends) {
    constexpr int kSegChunks = 1024 / (16 / kElt);
    constexpr int kWords = 8 * 32;
    __shared__ __align__(128) uint4 tile[kVec ? kSegChunks : 1];
    __shared__ uint32_t words[kWords];
    __shared__ int32_t state, moved;
    for (int i = threadIdx.x; i < kWords; i += kApplyThreads) words[i] = 0u;
    if (threadIdx.x == 0) moved = kDead;
    if (kVec) init_ninf_tile<kElt>(tile);
    else __syncthreads();
    pdl_launch_dependents();
    pdl_wait();  // logits, states and tokens come from earlier kernels
    const int32_t b = int32_t(blockIdx.x) / parts, part = int32_t(blockIdx.x) - b * parts;
    const int32_t s0 = __ldg(states + b);
    if (kAdvance) {
        // from a node, the move is the entry of the token in the node's list
        // (its end node, FINISHED for EOS), DEAD if the token is not there:
        // the advance's rules, in two dependent loads instead of a byte walk
        // (each entry's token and end are loaded together)
        const int32_t t = __ldg(tokens + b);
        const bool listed = ends && s0 >= 0 && s0 < n_nodes && t >= 0 && t < V;
        if (listed) {
            const int64_t lo = __ldg(off + s0), hi = __ldg(off + s0 + 1);
            for (int64_t i = lo + threadIdx.x; i < hi; i += kApplyThreads) {
                const int32_t tk = __ldg(toks + i), en = __ldg(ends + i);
                if (tk == t) moved = en;
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            const int32_t s1 = listed ? moved : advance_one(aa, s0, t);
            if (part == 0) {
                states_out[b] = s1;
                if (s1 == kDead && s0 != kDead && err) atomicAdd(err, 1);
            }
            state = s1;
        }
    } else if (threadIdx.x == 0) {
        state = s0;
    }
    __syncthreads();
    const int32_t s = state;
    const int32_t t0 = part * 8192, eos = V - 1;
    if (s >= 0 && s < n_nodes) {
        const int64_t lo = __ldg(off + s), hi = __ldg(off + s + 1);
        for (int64_t i = lo + threadIdx.x; i < hi; i += kApplyThreads) {
            const int32_t t = __ldg(toks + i) - t0;
            if (t >= 0 && t < 8192) atomicOr(words + (t >> 5), 1u << (t & 31));
        }
    } else if (threadIdx.x == 0 && eos - t0 >= 0 && eos - t0 < 8192) {
        words[(eos - t0) >> 5] = 1u << ((eos - t0) & 31);  // FINISHED, DEAD, not a node: {EOS}
    }
    __syncthreads();
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (kVec) {
        const int64_t row_chunks = int64_t(V) / (16 / kElt);
        const int64_t c0 = (int64_t(part) * 8 + wid) * kSegChunks;
        if (c0 >= row_chunks) return;
        write_segment<kElt>(static_cast<uint4 *>(logits) + int64_t(b) * row_chunks, c0, row_chunks,
                            words[wid * 32 + lane], lane, tile);
    } else {
        for (int32_t j = threadIdx.x; j < 8192; j += kApplyThreads) {
            const int32_t v = t0 + j;
            if (v >= V) break;
            if ((words[j >> 5] >> (j & 31)) & 1u) continue;
            const int64_t idx = int64_t(b) * V + v;
            if (kElt == 4) static_cast<uint32_t *>(logits)[idx] = 0xFF800000u;
            else static_cast<uint16_t *>(logits)[idx] = 0xFF80u;
        }
    }
}

// Any V and alignment: one thread per logit.
template <int kElt>
__global__ void __launch_bounds__(kApplyThreads) k_apply_scalar(void *__restrict__ logits,
                                                                const uint32_t *__restrict__ mask,
                                                                const int32_t *__restrict__ states,
                                                                int32_t B, int32_t V, int64_t W,
                                                                int32_t n_nodes) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t total = int64_t(B) * V;
    const int32_t eos = V - 1;
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += int64_t(gridDim.x) * blockDim.x) {
        const int32_t b = int32_t(i / V), v = int32_t(i % V);
        const uint32_t word = row_word(mask, __ldg(states + b), n_nodes, W, v >> 5, eos);
        if ((word >> (v & 31)) & 1u) continue;
        if (kElt == 4) static_cast<uint32_t *>(logits)[i] = 0xFF800000u;
        else static_cast<uint16_t *>(logits)[i] = 0xFF80u;
    }
}

// ------------------------------------------------------------ lazy rows
// valid[n] computed when a state first reaches n and kept in a row cache
// (App. H.5), instead of all rows up front. A call is three kernels:
//   k_lazy_resolve  one CTA: (advance,) then map every batch row's state to a
//                   cache row: a hit refreshes the row's stamp; the distinct
//                   missing nodes get the least recently used row of their
//                   set (or a per-call row when every row of the set is in use
//                   by this call);
//   k_lazy_rows     one CTA per task: valid[s] of a missing node s from s's
//                   subtree, or one part of it for a large subtree;
//   apply (k_apply_vec on the cache rows) or k_lazy_gather.

struct LazyArgs {
    uint32_t *rows;
    int32_t *tag;
    uint32_t *stamp;
    LazyCtrl *ctrl;
    int32_t *slot_of;
    int32_t *miss_node;
    int32_t *miss_slot;
    int32_t *row_u;
    int4 *task;
    const int32_t *pre_node;
    const int32_t *pre_depth;
    const int32_t *pre_size;
    const int32_t *pos_of;
    const LazyNode *pre;
    int32_t C;        // cache rows
    int32_t n_sets;   // C / kLazyWays
    int32_t n_nodes;
    int64_t W;
    int32_t uniq;     // slots of the resolve's table of distinct missing nodes (a power of two)
};

constexpr int kResolveThreads = 1024;
constexpr int kLazyRowThreads = 256;
constexpr int32_t kPending = -3;

__device__ __forceinline__ uint32_t mix32(uint32_t x) {
    x ^= x >> 16;
    x *= 0x7FEB352Du;
    x ^= x >> 15;
    x *= 0x846CA68Bu;
    x ^= x >> 16;
    return x;
}

__device__ __forceinline__ int32_t lazy_set(int32_t s, int32_t n_sets) {
    return int32_t((uint64_t(mix32(uint32_t(s))) * uint64_t(uint32_t(n_sets))) >> 32);
}

// Cache tags and stamps are read through L2 (ld.global.cg): other threads of
// the CTA change them with atomics during the kernel.
template <bool kAdvance>
__global__ void __launch_bounds__(kResolveThreads) k_lazy_resolve(LazyArgs L, AdvanceArgs aa,
                                                                  const int32_t *states_in,
                                                                  const int32_t *__restrict__ tokens,
                                                                  int32_t *states_out, int32_t *__restrict__ err,
                                                                  int32_t B) {
    extern __shared__ int32_t sh[];  // [uniq] node keys, [uniq] their miss index
    int32_t *keys = sh;
    int32_t *vals = sh + L.uniq;
    __shared__ int32_t n_u, n_tasks, n_split;
    __shared__ int32_t split_slot[kLazySplitRows];
    __shared__ unsigned long long n_hit, n_miss_rows;
    for (int32_t i = threadIdx.x; i < L.uniq; i += blockDim.x) keys[i] = -1;
    if (threadIdx.x == 0) {
        n_u = 0;
        n_tasks = 0;
        n_split = 0;
        n_hit = 0ull;
        n_miss_rows = 0ull;
    }
    __syncthreads();
    pdl_launch_dependents();
    pdl_wait();  // states, tokens, cache and scratch of earlier kernels
    const uint32_t now = __ldcg(&L.ctrl->now);
    const uint32_t umask = uint32_t(L.uniq - 1);
    // 1. states; cache lookups; distinct missing nodes into the table
    for (int32_t b = threadIdx.x; b < B; b += blockDim.x) {
        int32_t s;
        if (kAdvance) {
            const int32_t s0 = states_in[b];
            s = advance_one(aa, s0, tokens[b]);
            if (s == kDead && s0 != kDead && err) atomicAdd(err, 1);
            states_out[b] = s;
        } else {
            s = states_in[b];
        }
        int32_t slot = -1;  // the {EOS} row
        if (s >= 0 && s < L.n_nodes) {
            const int32_t base = (L.n_sets > 0 ? lazy_set(s, L.n_sets) : 0) * kLazyWays;
            int32_t hit = -1;
            if (L.n_sets > 0) {
#pragma unroll
                for (int w = 0; w < kLazyWays; w++)
                    if (__ldcg(L.tag + base + w) == s) hit = base + w;
            }
            if (hit >= 0) {
                L.stamp[hit] = now;
                slot = hit;
                atomicAdd(&n_hit, 1ull);
            } else {
                uint32_t h = mix32(uint32_t(s)) & umask;
                for (uint32_t it = 0; it <= umask; it++) {  // the table holds >= 2 B slots
                    const int32_t k = atomicCAS(keys + h, -1, s);
                    if (k == -1 || k == s) break;
                    h = (h + 1u) & umask;
                }
                L.row_u[b] = int32_t(h);
                slot = kPending;
                atomicAdd(&n_miss_rows, 1ull);
            }
        }
        L.slot_of[b] = slot;
    }
    __syncthreads();
    // 2. number the distinct missing nodes
    for (int32_t i = threadIdx.x; i < L.uniq; i += blockDim.x) {
        const int32_t k = keys[i];
        if (k >= 0) {
            const int32_t u = atomicAdd(&n_u, 1);
            vals[i] = u;
            L.miss_node[u] = k;
        }
    }
    __syncthreads();
    // 3. a row for each: the least recently used row of its set that this call
    // does not use, claimed by a compare-and-swap of its stamp
    for (int32_t u = threadIdx.x; u < n_u; u += blockDim.x) {
        const int32_t s = L.miss_node[u];
        int32_t slot = L.C + u;  // per-call row
        if (L.n_sets > 0) {
            const int32_t base = lazy_set(s, L.n_sets) * kLazyWays;
            for (int att = 0; att < 4 * kLazyWays; att++) {
                int32_t best = -1;
                uint32_t best_st = 0xFFFFFFFFu;
#pragma unroll
                for (int w = 0; w < kLazyWays; w++) {
                    const uint32_t st = __ldcg(L.stamp + base + w);
                    if (st != now && st < best_st) {
                        best_st = st;
                        best = w;
                    }
                }
                if (best < 0) break;
                if (atomicCAS(L.stamp + base + best, best_st, now) == best_st) {
                    slot = base + best;
                    L.tag[slot] = s;
                    break;
                }
            }
        }
        L.miss_slot[u] = slot;
        // CTA tasks: one, or up to kLazyMaxParts for a large subtree (for the
        // first kLazySplitRows such rows of the call)
        const int32_t desc = __ldg(L.pre_size + __ldg(L.pos_of + s)) - 1;
        int32_t parts = 1;
        if (desc > kLazyPartNodes) {
            const int32_t i = atomicAdd(&n_split, 1);
            if (i < kLazySplitRows) {
                parts = (desc + kLazyPartNodes - 1) / kLazyPartNodes;
                parts = parts < kLazyMaxParts ? parts : kLazyMaxParts;
                split_slot[i] = slot;
            }
        }
        const int32_t t0 = atomicAdd(&n_tasks, parts);
        for (int32_t p = 0; p < parts; p++) L.task[t0 + p] = make_int4(u, p, parts, 0);
    }
    __syncthreads();
    // rows built in parts are ORed together by atomics: zero them first
    const int32_t n_zero = n_split < kLazySplitRows ? n_split : kLazySplitRows;
    for (int32_t r = 0; r < n_zero; r++) {
        uint32_t *row = L.rows + int64_t(split_slot[r]) * L.W;
        for (int64_t i = threadIdx.x; i < L.W; i += blockDim.x) row[i] = 0u;
    }
    // 4. batch rows of missing nodes
    for (int32_t b = threadIdx.x; b < B; b += blockDim.x)
        if (L.slot_of[b] == kPending) L.slot_of[b] = L.miss_slot[vals[L.row_u[b]]];
    if (threadIdx.x == 0) {
        L.ctrl->n_miss = n_u;
        L.ctrl->n_tasks = n_tasks;
        L.ctrl->now = now + 1u;
        L.ctrl->hits += n_hit;
        L.ctrl->misses += n_miss_rows;
    }
}

// valid[s] for a missing node s (App. H.5), written to its cache row. The
// allowed tokens are the strings of the paths from s down into its subtree
// (App. G.5 condition (i): the token's bytes walk from s inside the trie),
// and EOS if s is terminal. The subtree is one interval of the pre-order
// tables; a descendant d at depth j below s (1 <= j <= the longest token)
// contributes the token, if any, whose bytes are the last j edge labels into
// d. A CTA builds the row (or, for a subtree split into parts, the part of it
// from its share of the interval) in shared memory, then stores it (a part
// ORs its non-zero words into the row, which the resolve has zeroed).
// B^j mod 2^64 by squaring.
__device__ __forceinline__ uint64_t hash_pow(uint32_t j) {
    uint64_t r = 1, b = kHashBase;
    while (j) {
        if (j & 1u) r *= b;
        b *= b;
        j >>= 1;
    }
    return r;
}

constexpr int kLazyNodesPerThread = 4;  // descendants resolved together by one thread

__global__ void __launch_bounds__(kLazyRowThreads, 2) k_lazy_rows(LazyArgs L, PatchArgs a) {
    extern __shared__ uint32_t bits[];
    pdl_launch_dependents();
    pdl_wait();  // the resolve's task list
    const int32_t n_tasks = __ldcg(&L.ctrl->n_tasks);
    const ulonglong2 *pairs = reinterpret_cast<const ulonglong2 *>(a.ht_key);
    for (int32_t ti = blockIdx.x; ti < n_tasks; ti += gridDim.x) {
        const int4 tk = __ldcg(L.task + ti);  // {miss, part, parts, -}
        const int32_t s = L.miss_node[tk.x];
        for (int64_t i = threadIdx.x; i < L.W; i += blockDim.x) bits[i] = 0u;
        __syncthreads();
        if (threadIdx.x == 0 && tk.y == 0 && __ldg(a.terminal + s)) atomicOr(bits + (a.eos >> 5), 1u << (a.eos & 31));
        const int32_t pos = __ldg(L.pos_of + s);
        const int32_t desc = __ldg(L.pre_size + pos) - 1;
        const int32_t k0 = pos + 1 + int32_t(int64_t(desc) * tk.y / tk.z);
        const int32_t k1 = pos + 1 + int32_t(int64_t(desc) * (tk.y + 1) / tk.z);
        const ulonglong2 *rec = reinterpret_cast<const ulonglong2 *>(L.pre);  // 2 per record
        const ulonglong2 sh0 = __ldg(rec + 2 * int64_t(pos));
        const uint64_t ps = sh0.x;
        const int32_t d0 = int32_t(uint32_t(sh0.y));
        for (int32_t kb = k0 + int32_t(threadIdx.x); kb < k1; kb += kLazyNodesPerThread * blockDim.x) {
            int32_t d[kLazyNodesPerThread], j[kLazyNodesPerThread];
            uint64_t pd[kLazyNodesPerThread];
            uint32_t lab[kLazyNodesPerThread][4];
#pragma unroll
            for (int g = 0; g < kLazyNodesPerThread; g++) {
                const int32_t k = kb + g * int32_t(blockDim.x);
                ulonglong2 r0 = make_ulonglong2(0ull, 0ull), r1 = make_ulonglong2(0ull, 0ull);
                if (k < k1) {
                    r0 = __ldg(rec + 2 * int64_t(k));
                    r1 = __ldg(rec + 2 * int64_t(k) + 1);
                }
                pd[g] = r0.x;
                j[g] = k < k1 ? int32_t(uint32_t(r0.y)) - d0 : 0;
                d[g] = int32_t(uint32_t(r0.y >> 32));
                if (j[g] > a.lmax) j[g] = 0;  // no token is this long
                lab[g][0] = uint32_t(r1.x);
                lab[g][1] = uint32_t(r1.x >> 32);
                lab[g][2] = uint32_t(r1.y);
                lab[g][3] = uint32_t(r1.y >> 32);
            }
            uint64_t key[kLazyNodesPerThread];
            ulonglong2 f[kLazyNodesPerThread];
#pragma unroll
            for (int g = 0; g < kLazyNodesPerThread; g++) {
                key[g] = hash_finish(pd[g] - ps * hash_pow(uint32_t(j[g])), uint32_t(j[g]));
                f[g] = j[g] > 0 ? __ldg(pairs + (uint32_t(key[g] >> 1) & a.pairs_mask)) : make_ulonglong2(0ull, 0ull);
            }
            // keys are resolved together (find_slots); paths longer than the
            // label window, and full first pairs in a vocabulary where tokens
            // share keys, take the sequential probe
            int32_t slot[kLazyNodesPerThread];
            uint32_t slow = 0;
            if (!a.dup_keys) {
                uint32_t pending = 0;
#pragma unroll
                for (int g = 0; g < kLazyNodesPerThread; g++) {
                    if (j[g] > kMaxClimb) slow |= 1u << g;
                    else if (j[g] > 0) pending |= 1u << g;
                }
                find_slots<kLazyNodesPerThread>(a, key, pending, f, slot);
            } else {
#pragma unroll
                for (int g = 0; g < kLazyNodesPerThread; g++) {
                    const bool m0 = f[g].x == key[g], m1 = f[g].y == key[g];
                    const uint32_t pr = uint32_t(key[g] >> 1) & a.pairs_mask;
                    slot[g] = -1;
                    if (j[g] > 0) {
                        if (j[g] > kMaxClimb || f[g].y != 0ull) slow |= 1u << g;
                        else if (m0 || m1) slot[g] = int32_t(2 * pr + (m0 ? 0 : 1));
                    }
                }
            }
            int32_t tid[kLazyNodesPerThread];
#pragma unroll
            for (int g = 0; g < kLazyNodesPerThread; g++) tid[g] = slot[g] >= 0 ? __ldg(a.ht_val + slot[g]) : -1;
            int32_t tlen[kLazyNodesPerThread];
            uint32_t toff[kLazyNodesPerThread];
#pragma unroll
            for (int g = 0; g < kLazyNodesPerThread; g++) {
                tlen[g] = tid[g] >= 0 ? int32_t(__ldg(a.tok_len + tid[g])) : -1;
                toff[g] = tid[g] >= 0 ? __ldg(a.tok_off + tid[g]) : 0u;
            }
            uint4 tb[kLazyNodesPerThread];
#pragma unroll
            for (int g = 0; g < kLazyNodesPerThread; g++)
                tb[g] = tlen[g] == j[g] ? __ldg(reinterpret_cast<const uint4 *>(a.blob + toff[g]))
                                        : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int g = 0; g < kLazyNodesPerThread; g++) {
                // token t moves s to d: its bit, and the move for later advances
                auto hit = [&](int32_t t) {
                    atomicOr(bits + (t >> 5), 1u << (t & 31));
                    if (a.trans_fill) trans_insert(a.trans, a.trans_mask, s, t, d[g]);
                };
                if (slow & (1u << g)) {
                    if (j[g] > kMaxClimb) probe(a, key[g], j[g], nullptr, d[g], hit);
                    else probe(a, key[g], j[g], &lab[g], d[g], hit);
                } else if (tid[g] >= 0 && tlen[g] == j[g]) {
                    // token byte i must equal the label j-1-i levels above d
                    const uint32_t tw[4] = {tb[g].x, tb[g].y, tb[g].z, tb[g].w};
                    bool eq = true;
#pragma unroll
                    for (int i = 0; i < kMaxClimb; i++)
                        if (i < j[g]) eq = eq && byte_at(tw, i) == byte_at(lab[g], j[g] - 1 - i);
                    if (eq) hit(tid[g]);
                }
            }
        }
        __syncthreads();
        uint32_t *row = L.rows + int64_t(L.miss_slot[tk.x]) * L.W;
        if (tk.z == 1) {
            for (int64_t i = threadIdx.x; i < L.W; i += blockDim.x) row[i] = bits[i];
        } else {
            for (int64_t i = threadIdx.x; i < L.W; i += blockDim.x)
                if (bits[i]) atomicOr(row + i, bits[i]);
        }
        __syncthreads();  // bits are reused by the next task
    }
}

// Copies the rows of a call out: out[b] = row of slot_of[b] ({EOS} if < 0).
__global__ void __launch_bounds__(kApplyThreads) k_lazy_gather(const uint32_t *__restrict__ rows,
                                                               const int32_t *__restrict__ slot_of, int32_t B,
                                                               int64_t W, int32_t n_rows, int32_t eos,
                                                               uint32_t *__restrict__ out) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t total = int64_t(B) * W;
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += int64_t(gridDim.x) * blockDim.x) {
        const int32_t b = int32_t(i / W);
        out[i] = row_word(rows, slot_of[b], n_rows, W, i - int64_t(b) * W, eos);
    }
}

// The pre-order records of the lazy rows: for position k, node d =
// pre_node[k], pos_of[d] = k, d's depth and label window, and the path hash
// of d: the Horner polynomial of the token table's hash over (label + 1) of
// the edges from the root to d, P(d) = P(parent) * B + label(d) + 1
// (mod 2^64), summed here by climbing to the root. The path from s down to a
// descendant d, j edges long, then hashes to P(d) - P(s) * B^j.
__global__ void k_lazy_tables(const int32_t *__restrict__ pre_node, const int32_t *__restrict__ pre_depth,
                              const int32_t *__restrict__ parent, const uint8_t *__restrict__ label,
                              const ulonglong2 *__restrict__ window, int32_t n, int32_t *__restrict__ pos_of,
                              LazyNode *__restrict__ pre) {
    for (int32_t k = blockIdx.x * blockDim.x + threadIdx.x; k < n; k += gridDim.x * blockDim.x) {
        const int32_t d = pre_node[k];
        pos_of[d] = k;
        uint64_t h = 0, pw = 1;
        for (int32_t y = d; __ldg(parent + y) >= 0; y = __ldg(parent + y)) {
            h += (uint64_t(__ldg(label + y)) + 1ull) * pw;
            pw *= kHashBase;
        }
        LazyNode r;
        r.phash = h;
        r.depth = pre_depth[k];
        r.node = d;
        r.window = window[d];
        pre[k] = r;
    }
}


PatchArgs patch_args(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax, uint32_t *mask,
                     int64_t W) {
    PatchArgs a;
    a.parent = t.parent;
    a.label = t.label;
    a.terminal = t.terminal;
    a.n_nodes = n_nodes;
    a.ht_key = v.ht_key;
    a.ht_val = v.ht_val;
    a.pairs_mask = v.ht_mask >> 1;
    a.tok_off = v.tok_off;
    a.tok_len = v.tok_len;
    a.blob = v.blob;
    a.ht_pay = v.ht_pay;
    a.lmax = lmax;
    a.mask = mask;
    a.W = W;
    a.eos = v.V - 1;
    a.hits = t.hits;
    a.hit_count = t.hit_count;
    a.window = t.window;
    a.depth16 = t.depth16;
    a.anc = t.anc;
    a.dup_keys = v.dup_keys;
    a.trans = t.trans;
    a.trans_mask = t.trans_mask;
    a.trans_fill = 0;
    a.seg_any = nullptr;
    a.seg_epoch = nullptr;
    a.seg_tag = 0;
    a.seg_words = 0;
    return a;
}

inline int grid_for(int64_t work, int64_t per_block, int64_t cap) {
    int64_t g = (work + per_block - 1) / per_block;
    if (g < 1) g = 1;
    if (g > cap) g = cap;
    return int(g);
}

// The probe: two threads per node while even those fill at most half of the
// resident slots (4 CTAs of kPatchThreads per SM) and the vocabulary allows
// it (per-slot payload, tokens of at most 16 bytes), else one per node. Its
// grid is resident at once (so that every CTA passes its entry wait and lets
// the fill launch right away); nodes in a grid-stride loop.
bool pair_probe(const PatchArgs &a, int num_sms) {
    const int64_t resident = int64_t(num_sms) * 4 * kPatchThreads;
    return a.ht_pay && a.lmax <= kMaxClimb && 2 * int64_t(a.n_nodes) * 2 <= resident;
}

// Lanes per node of the small-trie probe: 4 beside the fill (K = 1,000:
// 32.9 us per compile against 35.0 us with 2: the search under the fill's
// write stream is the long pole there, and 4 lanes shorten each lane's
// chain), 2 in the small-mask form (K = 100: 10.3 us against 12.3 us with 4).
constexpr int kProbeLanesBeside = 4;
constexpr int kProbeLanesSmall = 2;

cudaError_t launch_probe(const PatchArgs &a, const Prefetch &pf, int num_sms, cudaStream_t st) {
    if (pair_probe(a, num_sms))
        return launch_pdl(k_mask_probe_pair<kProbeLanesBeside, false>,
                          grid_for(kProbeLanesBeside * int64_t(a.n_nodes), kPatchThreads, int64_t(num_sms) * 4),
                          kPatchThreads, st, a, pf);
    return launch_pdl(k_mask_probe, grid_for(a.n_nodes, kPatchThreads, int64_t(num_sms) * 4), kPatchThreads, st, a,
                      pf);
}

}  // namespace

cudaError_t launch_mask_fill(uint32_t *mask, int64_t n_words, int num_sms, cudaStream_t st) {
    const uintptr_t a = reinterpret_cast<uintptr_t>(mask);
    int64_t head = int64_t(((16u - (a & 15u)) & 15u) >> 2);
    if (head > n_words) head = n_words;
    const int64_t n4 = (n_words - head) >> 2;
    (void)num_sms;
    const int grid = grid_for(n4, kFillThreads * kFillVecs, INT32_MAX);
    return launch_pdl(k_mask_fill, grid, kFillThreads, st, mask, n_words, head);
}

cudaError_t launch_mask_patch(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                              uint32_t *mask, int64_t W, int num_sms, cudaStream_t st) {
    PatchArgs a = patch_args(t, n_nodes, v, lmax, mask, W);
    const int grid = grid_for(n_nodes, kPatchThreads, int64_t(num_sms) * 32);
    return launch_pdl(k_mask_patch, grid, kPatchThreads, st, a);
}

cudaError_t launch_trans_clear(const DevTrie &t, int num_sms, cudaStream_t st) {
    return launch_mask_fill(reinterpret_cast<uint32_t *>(t.trans), 4 * (int64_t(t.trans_mask) + 1), num_sms, st);
}

cudaError_t launch_vocab_pay(const DevVocab &v, uint4 *pay, int num_sms, cudaStream_t st) {
    const int64_t S = int64_t(v.ht_mask) + 1;
    const int grid = grid_for(S, 256, int64_t(num_sms) * 8);
    k_vocab_pay<<<grid, 256, 0, st>>>(v.ht_key, v.ht_val, v.tok_len, v.tok_off, v.blob, S, pay);
    return cudaGetLastError();
}

cudaError_t launch_mask_compile3(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                                 uint32_t *mask, int64_t W, int num_sms, bool fill_trans, cudaStream_t st,
                                 unsigned long long *seg_any, uint32_t *seg_epoch, uint32_t epoch,
                                 int32_t seg_words, bool *seg_written) {
    PatchArgs a = patch_args(t, n_nodes, v, lmax, mask, W);
    a.trans_fill = fill_trans && t.trans;
    *seg_written = false;
    Prefetch pf;
    pf.count = 0;
    auto add = [&](const void *p, uint64_t n) {
        pf.ptr[pf.count] = p;
        pf.bytes[pf.count] = n;
        pf.count++;
    };
    const int64_t n_words = int64_t(n_nodes) * W;
    if (pair_probe(a, num_sms) && n_words * 4 <= kSmallMaskBytes) {
        // small masks: the zero fill, then the search ORing its hits itself
        cudaError_t e = launch_mask_fill(mask, n_words, num_sms, st);
        if (e != cudaSuccess) return e;
        return launch_pdl(k_mask_probe_pair<kProbeLanesSmall, true>,
                          grid_for(kProbeLanesSmall * int64_t(n_nodes), kPatchThreads, int64_t(num_sms) * 4),
                          kPatchThreads, st, a, pf);
    }
    a.seg_any = seg_any;  // the probe sets it (with this compile's epoch)
    a.seg_epoch = seg_epoch;
    a.seg_tag = epoch;
    a.seg_words = seg_words;
    *seg_written = seg_any != nullptr;
    const uint64_t S = uint64_t(v.ht_mask) + 1, nn = uint64_t(n_nodes), nv = uint64_t(v.V);
    add(v.ht_key, 8 * S);  // every suffix probe reads a slot pair
    if (!v.ht_pay) {       // only matches read the payload: it is not prefetched (measured slower
                           // with it: K = 1,000 35.8 against 35.2 us, K = 10,000 66.3 against 65.0 us)
        add(v.ht_val, 4 * S);
        add(v.tok_len, 2 * nv);
        add(v.tok_off, 4 * nv);
    }
    add(v.blob, v.blob_bytes);
    add(t.window, 16 * nn);
    add(t.anc, 64 * nn);
    add(t.depth16, nn);
    add(t.terminal, nn);
    cudaError_t e = launch_probe(a, pf, num_sms, st);
    if (e != cudaSuccess) return e;
    const uintptr_t addr = reinterpret_cast<uintptr_t>(mask);
    int64_t head = int64_t(((16u - (addr & 15u)) & 15u) >> 2);
    if (head > n_words) head = n_words;
    const int fill_grid = grid_for((n_words - head) >> 2, kFillThreads * kFillVecs, INT32_MAX);
    e = launch_pdl(k_mask_fill_beside, fill_grid, kFillThreads, st, mask, n_words, head);
    if (e != cudaSuccess) return e;
    const int scatter_grid = grid_for(n_nodes, kPatchThreads, int64_t(num_sms) * 16);
    return launch_pdl(k_mask_scatter, scatter_grid, kPatchThreads, st, a);
}

AdvanceArgs advance_args(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans) {
    AdvanceArgs a;
    a.first_child = t.first_child;
    a.child_bits = t.child_bits;
    a.terminal = t.terminal;
    a.n_nodes = n_nodes;
    a.tok_off = v.tok_off;
    a.tok_len = v.tok_len;
    a.blob = v.blob;
    a.V = v.V;
    a.trans = use_trans ? t.trans : nullptr;
    a.trans_mask = t.trans_mask;
    return a;
}

cudaError_t launch_mask_pairwise(const DevTrie &t, int32_t n_nodes, const DevVocab &v, uint32_t *mask, int num_sms,
                                 cudaStream_t st) {
    const AdvanceArgs a = advance_args(t, n_nodes, v, false);
    const int64_t W = (int64_t(v.V) + 31) / 32, chunks = (W + 31) / 32;
    const int grid = grid_for(int64_t(n_nodes) * chunks, kPairwiseThreads / 32, int64_t(num_sms) * 8);
    return launch_pdl(k_mask_pairwise, grid, kPairwiseThreads, st, a, mask, W, chunks);
}

cudaError_t launch_advance(const DevTrie &t, int32_t n_nodes, const DevVocab &v, const int32_t *states_in,
                           int32_t *states_out, const int32_t *tokens, int32_t B, int32_t *err, bool use_trans,
                           cudaStream_t st) {
    const int grid = (B + kAdvanceThreads - 1) / kAdvanceThreads;
    return launch_pdl(k_advance, grid, kAdvanceThreads, st, advance_args(t, n_nodes, v, use_trans), states_in,
                      states_out, tokens, B, err);
}

cudaError_t launch_advance_apply(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans,
                                 const int32_t *states_in, const int32_t *tokens, int32_t *states_out,
                                 int32_t *err, void *logits, int dtype, const uint32_t *mask, int32_t B,
                                 int num_sms, cudaStream_t st, const SegRef &seg) {
    const int32_t V = v.V;
    const int64_t W = (int64_t(V) + 31) / 32;
    const int elt = dtype == 0 ? 4 : 2;
    const int32_t segs = int32_t((W + 31) / 32);
    const bool vec = (reinterpret_cast<uintptr_t>(logits) & 15u) == 0 && (int64_t(V) * elt) % 16 == 0 &&
                     int64_t(B) * segs < int64_t(INT32_MAX);
    if (!vec) {  // any V and alignment: the two kernels one after the other
        cudaError_t e = launch_advance(t, n_nodes, v, states_in, states_out, tokens, B, err, use_trans, st);
        if (e != cudaSuccess) return e;
        return launch_apply(logits, dtype, mask, states_out, B, V, n_nodes, num_sms, st, seg);
    }
    const AdvanceArgs aa = advance_args(t, n_nodes, v, use_trans);
    const int32_t parts = (segs + kApplyThreads / 32 - 1) / (kApplyThreads / 32);
    const int64_t grid = int64_t(B) * parts;
    if (grid > INT32_MAX) return cudaErrorInvalidValue;
    if (elt == 2)
        return launch_pdl(k_advance_apply_vec<2>, grid, kApplyThreads, st, aa, static_cast<uint4 *>(logits), mask,
                          states_in, tokens, states_out, err, B, W, segs, parts, seg);
    return launch_pdl(k_advance_apply_vec<4>, grid, kApplyThreads, st, aa, static_cast<uint4 *>(logits), mask,
                      states_in, tokens, states_out, err, B, W, segs, parts, seg);
}

cudaError_t launch_apply(void *logits, int dtype, const uint32_t *mask, const int32_t *states,
                         int32_t B, int32_t V, int32_t n_nodes, int num_sms, cudaStream_t st,
                         const SegRef &seg) {
    const int64_t W = (int64_t(V) + 31) / 32;
    const int elt = dtype == 0 ? 4 : 2;
    const int32_t segs = int32_t((W + 31) / 32);
    const bool vec = (reinterpret_cast<uintptr_t>(logits) & 15u) == 0 && (int64_t(V) * elt) % 16 == 0 &&
                     int64_t(B) * segs < int64_t(INT32_MAX);
    if (vec) {
        const int64_t items = int64_t(B) * segs;
        const int grid = grid_for(items, kApplyThreads / 32, INT32_MAX);
        if (elt == 2)
            return launch_pdl(k_apply_vec<2>, grid, kApplyThreads, st, static_cast<uint4 *>(logits), mask,
                              states, B, V, W, n_nodes, segs, seg);
        return launch_pdl(k_apply_vec<4>, grid, kApplyThreads, st, static_cast<uint4 *>(logits), mask, states,
                          B, V, W, n_nodes, segs, seg);
    }
    const int grid = grid_for(int64_t(B) * V, kApplyThreads, int64_t(num_sms) * 16);
    if (elt == 2)
        return launch_pdl(k_apply_scalar<2>, grid, kApplyThreads, st, logits, mask, states, B, V, W, n_nodes);
    return launch_pdl(k_apply_scalar<4>, grid, kApplyThreads, st, logits, mask, states, B, V, W, n_nodes);
}

namespace {

// Up to three copies in one launch, reading the sources directly (host memory
// that the device reads coherently, or device memory): 16-byte blocks where
// both ends are 16-byte aligned, else bytes.
struct CopySeg {
    uint8_t *dst;
    const uint8_t *src;
    int64_t bytes;
};

__global__ void k_copy_segments(CopySeg s0, CopySeg s1, CopySeg s2) {
    pdl_launch_dependents();
    pdl_wait();  // the destination may still be read by an earlier kernel
    const int64_t stride = int64_t(gridDim.x) * blockDim.x;
    const int64_t i0 = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    const CopySeg seg[3] = {s0, s1, s2};
#pragma unroll
    for (int k = 0; k < 3; k++) {
        const CopySeg c = seg[k];
        int64_t done = 0;
        if (((reinterpret_cast<uintptr_t>(c.dst) | reinterpret_cast<uintptr_t>(c.src)) & 15u) == 0) {
            const int64_t nv = c.bytes >> 4;
            for (int64_t i = i0; i < nv; i += stride)
                reinterpret_cast<uint4 *>(c.dst)[i] = reinterpret_cast<const uint4 *>(c.src)[i];
            done = nv << 4;
        }
        for (int64_t i = done + i0; i < c.bytes; i += stride) c.dst[i] = c.src[i];
    }
}

}  // namespace

cudaError_t launch_copy3(void *d0, const void *s0, int64_t b0, void *d1, const void *s1, int64_t b1, void *d2,
                         const void *s2, int64_t b2, int num_sms, cudaStream_t st) {
    const int64_t most = std::max(b0, std::max(b1, b2));
    if (most <= 0) return cudaSuccess;
    const int grid = grid_for((most + 15) / 16, 256, int64_t(num_sms) * 4);
    return launch_pdl(k_copy_segments, grid, 256, st,
                      CopySeg{static_cast<uint8_t *>(d0), static_cast<const uint8_t *>(s0), b0},
                      CopySeg{static_cast<uint8_t *>(d1), static_cast<const uint8_t *>(s1), b1},
                      CopySeg{static_cast<uint8_t *>(d2), static_cast<const uint8_t *>(s2), b2});
}

cudaError_t launch_rt_build(const int32_t *parent, const uint8_t *label, const int32_t *token, int32_t n,
                            uint4 *edge, uint32_t mask, int num_sms, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(edge, 0, sizeof(uint4) * (size_t(mask) + 1), st);
    if (e != cudaSuccess || n <= 1) return e;
    const uint32_t shift = 32u - uint32_t(__builtin_popcount(mask));
    const int grid = grid_for(n, 256, int64_t(num_sms) * 8);
    k_rt_insert<<<grid, 256, 0, st>>>(parent, label, token, n, edge, mask, shift);
    return cudaGetLastError();
}

namespace {

WalkArgs walk_args(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax, const DevLists &L) {
    WalkArgs a;
    a.terminal = t.terminal;
    a.window = t.window;
    a.depth16 = t.depth16;
    a.anc = reinterpret_cast<const int32_t *>(t.anc);
    a.parent = t.parent;
    a.label = t.label;
    a.n_nodes = n_nodes;
    a.lmax = lmax;
    a.eos = v.V - 1;
    a.edge = v.rt_edge;
    a.edge_mask = v.rt_mask;
    a.edge_shift = 32u - uint32_t(__builtin_popcount(v.rt_mask));
    a.tok_next = v.tok_next;
    a.count = L.count;
    a.off = reinterpret_cast<unsigned long long *>(L.off);
    a.toks = L.toks;
    a.ends = L.ends;
    a.tok_cap = static_cast<unsigned long long>(L.tok_cap);
    return a;
}

}  // namespace

cudaError_t launch_lists_count(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                               const DevLists &L, int num_sms, cudaStream_t st) {
    const WalkArgs a = walk_args(t, n_nodes, v, lmax, L);
    cudaError_t e = launch_mask_fill(reinterpret_cast<uint32_t *>(L.count), int64_t(n_nodes), num_sms, st);
    if (e != cudaSuccess) return e;
    const int grid = grid_for(n_nodes, kWalkThreads, int64_t(num_sms) * 8);
    if ((e = launch_pdl(k_list_walk<false>, grid, kWalkThreads, st, a)) != cudaSuccess) return e;
    const int32_t n_tiles = int32_t((int64_t(n_nodes) + kScanTile - 1) / kScanTile);
    if ((e = launch_pdl(k_scan_tiles, n_tiles, kScanThreads, st, static_cast<const int32_t *>(L.count), n_nodes,
                        L.tile_sum)) != cudaSuccess)
        return e;
    if ((e = launch_pdl(k_scan_tile_sums, 1, kScanThreads, st, L.tile_sum, n_tiles, L.total)) != cudaSuccess)
        return e;
    if ((e = launch_pdl(k_scan_rows, n_tiles, kScanThreads, st, static_cast<const int32_t *>(L.count), n_nodes,
                        static_cast<const int64_t *>(L.tile_sum), L.off)) != cudaSuccess)
        return e;
    return cudaSuccess;
}

cudaError_t launch_lists_write(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                               const DevLists &L, int num_sms, cudaStream_t st) {
    const WalkArgs a = walk_args(t, n_nodes, v, lmax, L);
    const int grid = grid_for(n_nodes, kWalkThreads, int64_t(num_sms) * 8);
    return launch_pdl(k_list_walk<true>, grid, kWalkThreads, st, a);
}

namespace {

cudaError_t launch_lists(void *logits, int dtype, const DevLists &L, const AdvanceArgs *aa,
                         const int32_t *states, const int32_t *tokens, int32_t *states_out, int32_t *err,
                         int32_t B, int32_t V, int32_t n_nodes, cudaStream_t st) {
    const int elt = dtype == 0 ? 4 : 2;
    const int32_t parts = int32_t((int64_t(V) + 8191) / 8192);
    const bool vec = (reinterpret_cast<uintptr_t>(logits) & 15u) == 0 && (int64_t(V) * elt) % 16 == 0;
    const int64_t grid = int64_t(B) * parts;
    if (grid > INT32_MAX) return cudaErrorInvalidValue;
    const int32_t *tk = L.toks;
    const int64_t *of = L.off;
    const AdvanceArgs a = aa ? *aa : AdvanceArgs{};
    if (aa) {
        if (vec)
            return elt == 2 ? launch_pdl(k_apply_lists<2, true, true>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                         states, tokens, states_out, err, B, V, n_nodes, parts, L.ends)
                            : launch_pdl(k_apply_lists<4, true, true>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                         states, tokens, states_out, err, B, V, n_nodes, parts, L.ends);
        return elt == 2 ? launch_pdl(k_apply_lists<2, false, true>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                     states, tokens, states_out, err, B, V, n_nodes, parts, L.ends)
                        : launch_pdl(k_apply_lists<4, false, true>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                     states, tokens, states_out, err, B, V, n_nodes, parts, L.ends);
    }
    if (vec)
        return elt == 2 ? launch_pdl(k_apply_lists<2, true, false>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                     states, tokens, states_out, err, B, V, n_nodes, parts, L.ends)
                        : launch_pdl(k_apply_lists<4, true, false>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                     states, tokens, states_out, err, B, V, n_nodes, parts, L.ends);
    return elt == 2 ? launch_pdl(k_apply_lists<2, false, false>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                 states, tokens, states_out, err, B, V, n_nodes, parts, L.ends)
                    : launch_pdl(k_apply_lists<4, false, false>, int(grid), kApplyThreads, st, logits, of, tk, a,
                                 states, tokens, states_out, err, B, V, n_nodes, parts, L.ends);
}

}  // namespace

cudaError_t launch_apply_lists(void *logits, int dtype, const DevLists &L, const int32_t *states, int32_t B,
                               int32_t V, int32_t n_nodes, cudaStream_t st) {
    return launch_lists(logits, dtype, L, nullptr, states, nullptr, nullptr, nullptr, B, V, n_nodes, st);
}

cudaError_t launch_advance_apply_lists(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans,
                                       const int32_t *states_in, const int32_t *tokens, int32_t *states_out,
                                       int32_t *err, void *logits, int dtype, const DevLists &L, int32_t B,
                                       cudaStream_t st) {
    const AdvanceArgs aa = advance_args(t, n_nodes, v, use_trans);
    return launch_lists(logits, dtype, L, &aa, states_in, tokens, states_out, err, B, v.V, n_nodes, st);
}

cudaError_t launch_lazy_tables(const DevTrie &t, const DevLazy &L, int32_t n_nodes, cudaStream_t st) {
    // shared memory above the default 48 KB: the resolve's table of distinct
    // nodes (<= 2 * 2 * kLazyMaxBatch int32) and the row kernel's row
    const int uniq_max = int(2 * 2 * kLazyMaxBatch * sizeof(int32_t));
    const int row_max = int(kLazyMaxWords * sizeof(uint32_t));
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(k_lazy_resolve<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, uniq_max)) !=
        cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_lazy_resolve<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, uniq_max)) !=
        cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_lazy_rows, cudaFuncAttributeMaxDynamicSharedMemorySize, row_max)) !=
        cudaSuccess)
        return e;
    if (n_nodes <= 0) return cudaSuccess;
    const int grid = grid_for(n_nodes, 256, 4096);
    k_lazy_tables<<<grid, 256, 0, st>>>(L.pre_node, L.pre_depth, t.parent, t.label, t.window, n_nodes, L.pos_of,
                                        L.pre);
    return cudaGetLastError();
}

cudaError_t launch_lazy(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans, bool fill_trans,
                        int32_t lmax,
                        const DevLazy &L, const int32_t *states_in, const int32_t *tokens, int32_t *states_out,
                        int32_t *err, int32_t B, void *logits, int dtype, uint32_t *rows_out, int num_sms,
                        cudaStream_t st) {
    LazyArgs la;
    la.rows = L.rows;
    la.tag = L.tag;
    la.stamp = L.stamp;
    la.ctrl = L.ctrl;
    la.slot_of = L.slot_of;
    la.miss_node = L.miss_node;
    la.miss_slot = L.miss_slot;
    la.row_u = L.row_u;
    la.task = L.task;
    la.pre_node = L.pre_node;
    la.pre_depth = L.pre_depth;
    la.pre_size = L.pre_size;
    la.pos_of = L.pos_of;
    la.pre = L.pre;
    la.C = L.C;
    la.n_sets = L.C / kLazyWays;
    la.n_nodes = n_nodes;
    la.W = L.W;
    int32_t uniq = 16;
    while (uniq < 2 * B) uniq <<= 1;
    la.uniq = uniq;
    const AdvanceArgs aa = advance_args(t, n_nodes, v, use_trans);
    const size_t rsmem = size_t(2) * size_t(uniq) * sizeof(int32_t);
    cudaError_t e = tokens ? launch_pdl_smem(k_lazy_resolve<true>, 1, kResolveThreads, rsmem, st, la, aa, states_in,
                                             tokens, states_out, err, B)
                           : launch_pdl_smem(k_lazy_resolve<false>, 1, kResolveThreads, rsmem, st, la, aa,
                                             states_in, tokens, states_out, err, B);
    if (e != cudaSuccess) return e;
    PatchArgs pa = patch_args(t, n_nodes, v, lmax, nullptr, L.W);
    pa.trans_fill = fill_trans && t.trans;
    // tasks in a grid-stride loop over two CTAs per SM
    const int rows_grid = grid_for(int64_t(B) + int64_t(kLazySplitRows) * kLazyMaxParts, 1, int64_t(num_sms) * 2);
    e = launch_pdl_smem(k_lazy_rows, rows_grid, kLazyRowThreads, size_t(L.W) * sizeof(uint32_t), st, la, pa);
    if (e != cudaSuccess) return e;
    const int32_t n_rows = L.C + L.max_batch;
    if (logits) return launch_apply(logits, dtype, L.rows, L.slot_of, B, L.V, n_rows, num_sms, st);
    const int grid = grid_for(int64_t(B) * L.W, kApplyThreads, int64_t(num_sms) * 8);
    return launch_pdl(k_lazy_gather, grid, kApplyThreads, st, static_cast<const uint32_t *>(L.rows),
                      static_cast<const int32_t *>(L.slot_of), B, L.W, n_rows, L.V - 1, rows_out);
}

}  // namespace tmk
