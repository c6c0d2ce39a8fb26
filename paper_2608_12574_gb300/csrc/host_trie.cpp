// Host side of libtriemask: the byte-trie builder (Sec. 4.1; App. G.1 Step 1)
// and the per-tokenizer vocabulary packing (App. H.4 Phase 2).
//
// The trie is built from the sorted, de-duplicated strings: in sorted order
// the longest prefix of a string already in the trie is its longest common
// prefix with the previous string, so nodes are created in pre-order without
// any child lookup. Breadth-first ids with siblings by ascending byte are
// then the nodes sorted by (depth, pre-order index): at one depth, pre-order
// is lexicographic order of the prefixes, which is exactly sibling-sorted
// BFS order.
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <numeric>
#include <string>
#include <thread>
#include <vector>

#include "tm_internal.h"

namespace tmk {

namespace {

struct Str {
    const uint8_t *p;
    int64_t n;
    uint64_t key;  // first 8 bytes, big-endian, zero padded
};

inline int cmp_str(const Str &a, const Str &b) {
    if (a.key != b.key) return a.key < b.key ? -1 : 1;
    int64_t m = std::min(a.n, b.n);
    if (m > 8) {
        int c = memcmp(a.p + 8, b.p + 8, size_t(m - 8));
        if (c) return c;
    }
    return a.n < b.n ? -1 : (a.n > b.n ? 1 : 0);
}

}  // namespace

std::string build_trie(const uint8_t *bytes, const int64_t *offsets, int32_t first, int32_t last,
                       HostTrie *out) {
    const int64_t K = int64_t(last) - first;
    std::vector<Str> s(size_t(std::max<int64_t>(K, 0)));
    int64_t total = 0;
    for (int64_t i = 0; i < K; i++) {
        int64_t a = offsets[first + i], e = offsets[first + i + 1];
        if (a < 0 || e < a) return "offsets must be non-negative and non-decreasing";
        Str &x = s[size_t(i)];
        x.p = bytes + a;
        x.n = e - a;
        uint64_t k = 0;
        for (int j = 0; j < 8; j++) k = (k << 8) | (j < x.n ? x.p[j] : 0);
        x.key = k;
        total += x.n;
    }
    if (total > int64_t(INT32_MAX) - 2) return "trie would exceed 2^31-1 nodes";
    std::sort(s.begin(), s.end(), [](const Str &a, const Str &b) { return cmp_str(a, b) < 0; });

    // pre-order creation (at most 1 + total nodes)
    hvec<int32_t> pparent(size_t(total) + 1), pdepth(size_t(total) + 1);
    hvec<uint8_t> plabel(size_t(total) + 1), pterm(size_t(total) + 1);
    pparent[0] = -1;
    pdepth[0] = 0;
    plabel[0] = 0;
    pterm[0] = 0;
    int32_t n = 1;
    std::vector<int32_t> path(1, 0);
    const Str *prev = nullptr;
    int64_t n_chars = 0;
    int32_t max_depth = 0;
    for (const Str &x : s) {
        int64_t lcp = 0;
        if (prev) {
            if (cmp_str(*prev, x) == 0) continue;  // duplicate value
            int64_t m = std::min(prev->n, x.n);
            while (lcp < m && prev->p[lcp] == x.p[lcp]) lcp++;
        }
        if (int64_t(path.size()) < x.n + 1) path.resize(size_t(x.n + 1));
        for (int64_t d = lcp + 1; d <= x.n; d++) {
            const size_t id = size_t(n++);
            pparent[id] = path[size_t(d - 1)];
            plabel[id] = x.p[d - 1];
            pterm[id] = 0;
            pdepth[id] = int32_t(d);
            path[size_t(d)] = int32_t(id);
        }
        pterm[size_t(path[size_t(x.n)])] = 1;
        n_chars += x.n;
        max_depth = std::max<int32_t>(max_depth, int32_t(x.n));
        prev = &x;
    }
    pdepth.resize(size_t(n));

    // breadth-first ids: stable bucket by depth
    std::vector<int32_t> level(size_t(max_depth) + 2, 0);
    for (int32_t i = 0; i < n; i++) level[size_t(pdepth[i]) + 1]++;
    for (size_t d = 1; d < level.size(); d++) level[d] += level[d - 1];
    hvec<int32_t> bfs(static_cast<size_t>(n));
    for (int32_t i = 0; i < n; i++) bfs[size_t(i)] = level[size_t(pdepth[i])]++;
    // subtree sizes in pre-order (a parent precedes its descendants)
    hvec<int32_t> psize(static_cast<size_t>(n));
    for (int32_t i = 0; i < n; i++) psize[size_t(i)] = 1;
    for (int32_t i = n - 1; i > 0; i--) psize[size_t(pparent[size_t(i)])] += psize[size_t(i)];

    out->n = n;
    out->parent.resize(size_t(n));
    out->label.resize(size_t(n));
    out->terminal.resize(size_t(n));
    for (int32_t i = 0; i < n; i++) {  // every BFS id is written once
        int32_t b = bfs[size_t(i)];
        out->label[size_t(b)] = plabel[size_t(i)];
        out->terminal[size_t(b)] = pterm[size_t(i)];
        out->parent[size_t(b)] = pparent[size_t(i)] < 0 ? -1 : bfs[size_t(pparent[size_t(i)])];
    }
    out->pre_node = std::move(bfs);
    out->pre_depth = std::move(pdepth);
    out->pre_size = std::move(psize);
    out->roots.assign(1, 0);
    out->n_chars = n_chars;
    out->max_depth = max_depth;
    return "";
}

std::string build_forest(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets,
                         int32_t M, HostTrie *out) {
    std::vector<HostTrie> parts(static_cast<size_t>(M));
    std::vector<std::string> errs(static_cast<size_t>(M));
    unsigned hw = std::max(1u, std::thread::hardware_concurrency());
    unsigned nth = std::min<unsigned>(hw, unsigned(M));
    // phase 1: every set's trie on its own, in parallel
    std::atomic<int32_t> next(0);
    auto build = [&]() {
        for (;;) {
            int32_t i = next.fetch_add(1);
            if (i >= M) return;
            errs[size_t(i)] = build_trie(bytes, offsets, set_offsets[i], set_offsets[i + 1], &parts[size_t(i)]);
        }
    };
    std::vector<std::thread> th;
    for (unsigned t = 1; t < nth; t++) th.emplace_back(build);
    build();
    for (auto &t : th) t.join();
    th.clear();
    int64_t total = 0, n_chars = 0;
    int32_t max_depth = 0;
    std::vector<int32_t> base(static_cast<size_t>(M));
    for (int32_t i = 0; i < M; i++) {
        if (!errs[size_t(i)].empty()) return "set " + std::to_string(i) + ": " + errs[size_t(i)];
        base[size_t(i)] = int32_t(std::min<int64_t>(total, INT32_MAX));
        total += parts[size_t(i)].n;
        n_chars += parts[size_t(i)].n_chars;
        max_depth = std::max(max_depth, parts[size_t(i)].max_depth);
    }
    if (total > int64_t(INT32_MAX) - 2) return "forest would exceed 2^31-1 nodes";
    const size_t n = size_t(total);
    // phase 2: concatenate, each worker copying (and first touching) its sets
    out->n = int32_t(n);
    out->parent.resize(n);
    out->label.resize(n);
    out->terminal.resize(n);
    out->pre_node.resize(n);
    out->pre_depth.resize(n);
    out->pre_size.resize(n);
    out->roots.assign(base.begin(), base.end());
    next = 0;
    auto concat = [&]() {
        for (;;) {
            int32_t i = next.fetch_add(1);
            if (i >= M) return;
            HostTrie &p = parts[size_t(i)];
            const int32_t b = base[size_t(i)];
            const size_t g = size_t(b), pn = size_t(p.n);
            for (size_t j = 0; j < pn; j++) out->parent[g + j] = p.parent[j] < 0 ? -1 : p.parent[j] + b;
            for (size_t j = 0; j < pn; j++) out->pre_node[g + j] = p.pre_node[j] + b;
            memcpy(&out->pre_depth[g], p.pre_depth.data(), sizeof(int32_t) * pn);
            memcpy(&out->pre_size[g], p.pre_size.data(), sizeof(int32_t) * pn);
            memcpy(&out->label[g], p.label.data(), pn);
            memcpy(&out->terminal[g], p.terminal.data(), pn);
            p = HostTrie();  // release the part's memory early
        }
    };
    for (unsigned t = 1; t < nth; t++) th.emplace_back(concat);
    concat();
    for (auto &t : th) t.join();
    out->n_chars = n_chars;
    out->max_depth = max_depth;
    return "";
}

std::string pack_vocab(const uint8_t *bytes, const int64_t *offsets, int32_t V, HostVocab *out) {
    if (V < 2) return "V must be >= 2 (token V-1 is EOS)";
    if (offsets[0] < 0) return "vocab offsets must be non-negative";
    out->V = V;
    out->tok_off.assign(size_t(V), 0);
    out->tok_len.assign(size_t(V), 0);
    uint64_t pos = 0;
    int64_t n_ins = 0;
    int32_t max_len = 0;
    for (int32_t v = 0; v < V; v++) {
        int64_t a = offsets[v], e = offsets[v + 1];
        if (e < a) return "vocab offsets must be non-decreasing";
        int64_t L = (v == V - 1) ? 0 : e - a;  // EOS bytes are ignored
        if (L > 65535) return "token " + std::to_string(v) + " is longer than 65535 bytes";
        out->tok_off[size_t(v)] = uint32_t(pos);
        out->tok_len[size_t(v)] = uint16_t(L);
        pos += uint64_t((L + 15) / 16 * 16);
        if (pos > 0xFFFFFFF0ull) return "packed vocabulary exceeds 4 GiB";
        if (L > 0) {
            n_ins++;
            max_len = std::max<int32_t>(max_len, int32_t(L));
        }
    }
    out->max_len = max_len;
    out->blob.assign(size_t(pos) + 16, 0);
    for (int32_t v = 0; v < V; v++)
        if (out->tok_len[size_t(v)])
            memcpy(&out->blob[out->tok_off[size_t(v)]], bytes + offsets[v], out->tok_len[size_t(v)]);
    // load factor <= 1/4; slots are probed in aligned pairs (one 16-byte load
    // holds two keys), pair after pair, the even slot of a pair filled first
    uint64_t S = 16;
    while (S < uint64_t(4 * n_ins)) S <<= 1;
    if (S > (uint64_t(1) << 31)) return "vocabulary too large for the token hash table";
    out->ht_key.assign(size_t(S), 0ull);
    out->ht_val.assign(size_t(S), -1);
    out->ht_mask = uint32_t(S - 1);
    const uint64_t pairs_mask = S / 2 - 1;
    for (int32_t v = 0; v < V; v++) {
        uint32_t L = out->tok_len[size_t(v)];
        if (!L) continue;
        const uint8_t *p = bytes + offsets[v];
        uint64_t h = 0;
        for (uint32_t j = 0; j < L; j++) h = h * kHashBase + uint64_t(p[j]) + 1;
        const uint64_t key = hash_finish(h, L);
        uint64_t pair = (key >> 1) & pairs_mask;
        for (;;) {
            size_t s0 = size_t(2 * pair);
            // an equal key: a repeated token string, or two strings whose hashes collide
            if (out->ht_key[s0] == key || out->ht_key[s0 + 1] == key) out->dup_keys = 1;
            if (!out->ht_key[s0]) { out->ht_key[s0] = key; out->ht_val[s0] = v; break; }
            if (!out->ht_key[s0 + 1]) { out->ht_key[s0 + 1] = key; out->ht_val[s0 + 1] = v; break; }
            pair = (pair + 1) & pairs_mask;
        }
    }
    return "";
}

}  // namespace tmk
