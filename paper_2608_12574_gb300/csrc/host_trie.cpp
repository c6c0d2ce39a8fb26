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
#include <cstdlib>
#include <mutex>
#include <numeric>
#include <string>
#include <thread>
#include <vector>

#include "tm_internal.h"

namespace tmk {

namespace {

struct BlockCache {
    std::mutex mu;
    std::vector<std::pair<size_t, void *>> free;  // (size class in bytes, block)
    size_t held = 0;
};
constexpr size_t kBlockCacheMax = size_t(1) << 30;

BlockCache &block_cache() {
    static BlockCache *c = new BlockCache();  // never destroyed: blocks may be freed during exit
    return *c;
}

size_t block_class(size_t bytes) { return (bytes + kBigBlock - 1) / kBigBlock * kBigBlock; }

}  // namespace

void *big_block_alloc(size_t bytes) {
    const size_t cls = block_class(bytes);
    BlockCache &c = block_cache();
    {
        std::lock_guard<std::mutex> lk(c.mu);
        for (size_t i = 0; i < c.free.size(); i++)
            if (c.free[i].first == cls) {
                void *p = c.free[i].second;
                c.free[i] = c.free.back();
                c.free.pop_back();
                c.held -= cls;
                return p;
            }
    }
    return std::malloc(cls);
}

void big_block_free(void *p, size_t bytes) {
    if (!p) return;
    const size_t cls = block_class(bytes);
    BlockCache &c = block_cache();
    {
        std::lock_guard<std::mutex> lk(c.mu);
        if (c.held + cls <= kBlockCacheMax) {
            c.free.emplace_back(cls, p);
            c.held += cls;
            return;
        }
    }
    std::free(p);
}

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

namespace {

// A set's nodes in pre-order (the order the sorted strings create them).
struct PreTrie {
    int32_t n = 0;
    hvec<int32_t> pparent, pdepth;
    hvec<uint8_t> plabel, pterm;
    int64_t n_chars = 0;
    int32_t max_depth = 0;
};

// Sorts strings first..last-1 and creates their nodes in pre-order.
std::string prepare_trie(const uint8_t *bytes, const int64_t *offsets, int32_t first, int32_t last, PreTrie *out) {
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
    out->pparent = std::move(pparent);
    out->plabel = std::move(plabel);
    out->pterm = std::move(pterm);
    out->pdepth = std::move(pdepth);
    out->n = n;
    out->n_chars = n_chars;
    out->max_depth = max_depth;
    return "";
}

// Writes a prepared set into out's arrays at node ids base .. base + n - 1:
// breadth-first ids (the pre-order nodes stably bucketed by depth), parent /
// label / terminal, and the pre-order tables (node, depth, subtree size).
void emit_trie(const PreTrie &p, int32_t base, HostTrie *out) {
    const int32_t n = p.n;
    const size_t g = size_t(base);
    std::vector<int32_t> level(size_t(p.max_depth) + 2, 0);
    for (int32_t i = 0; i < n; i++) level[size_t(p.pdepth[size_t(i)]) + 1]++;
    for (size_t d = 1; d < level.size(); d++) level[d] += level[d - 1];
    int32_t *bfs = &out->pre_node[g];  // local BFS ids first, offset below
    for (int32_t i = 0; i < n; i++) bfs[i] = level[size_t(p.pdepth[size_t(i)])]++;
    int32_t *psize = &out->pre_size[g];  // subtree sizes (a parent precedes its descendants)
    for (int32_t i = 0; i < n; i++) psize[i] = 1;
    for (int32_t i = n - 1; i > 0; i--) psize[p.pparent[size_t(i)]] += psize[i];
    for (int32_t i = 0; i < n; i++) {  // every BFS id is written once
        const size_t b = g + size_t(bfs[i]);
        out->label[b] = p.plabel[size_t(i)];
        out->terminal[b] = p.pterm[size_t(i)];
        out->parent[b] = p.pparent[size_t(i)] < 0 ? -1 : bfs[p.pparent[size_t(i)]] + base;
    }
    memcpy(&out->pre_depth[g], p.pdepth.data(), sizeof(int32_t) * size_t(n));
    for (int32_t i = 0; i < n; i++) bfs[i] += base;
}

void alloc_out(HostTrie *out, size_t n) {
    out->n = int32_t(n);
    out->parent.resize(n);
    out->label.resize(n);
    out->terminal.resize(n);
    out->pre_node.resize(n);
    out->pre_depth.resize(n);
    out->pre_size.resize(n);
}

}  // namespace

std::string build_trie(const uint8_t *bytes, const int64_t *offsets, int32_t first, int32_t last,
                       HostTrie *out) {
    PreTrie p;
    std::string err = prepare_trie(bytes, offsets, first, last, &p);
    if (!err.empty()) return err;
    alloc_out(out, size_t(p.n));
    emit_trie(p, 0, out);
    out->roots.assign(1, 0);
    out->n_chars = p.n_chars;
    out->max_depth = p.max_depth;
    return "";
}

std::string build_forest(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets,
                         int32_t M, HostTrie *out) {
    std::vector<PreTrie> parts(static_cast<size_t>(M));
    std::vector<std::string> errs(static_cast<size_t>(M));
    unsigned hw = std::max(1u, std::thread::hardware_concurrency());
    unsigned nth = std::min<unsigned>(hw, unsigned(M));
    auto run = [&](auto &&work) {  // work(i) for every set, on nth threads
        std::atomic<int32_t> next(0);
        auto loop = [&]() {
            for (int32_t i; (i = next.fetch_add(1)) < M;) work(i);
        };
        std::vector<std::thread> th;
        for (unsigned t = 1; t < nth; t++) th.emplace_back(loop);
        loop();
        for (auto &t : th) t.join();
    };
    // phase 1: every set sorted and laid out in pre-order, in parallel
    run([&](int32_t i) {
        errs[size_t(i)] = prepare_trie(bytes, offsets, set_offsets[i], set_offsets[i + 1], &parts[size_t(i)]);
    });
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
    // phase 2: every set written at its offset of the forest's arrays
    alloc_out(out, size_t(total));
    run([&](int32_t i) {
        emit_trie(parts[size_t(i)], base[size_t(i)], out);
        parts[size_t(i)] = PreTrie();  // release the set's memory early
    });
    out->roots.assign(base.begin(), base.end());
    out->n_chars = n_chars;
    out->max_depth = max_depth;
    return "";
}

// In breadth-first order with ascending sibling bytes, the children of a node
// are consecutive ids after it, so a depth-first walk that visits them in id
// order is the builder's pre-order (sorted strings); set i's walk fills
// positions roots[i] .. roots[i + 1] - 1.
void pre_order_from_parents(HostTrie *t) {
    const int32_t n = t->n;
    t->pre_node.resize(size_t(n));
    t->pre_depth.resize(size_t(n));
    t->pre_size.resize(size_t(n));
    std::vector<int32_t> first(size_t(n), -1), cnt(size_t(n), 0), size(size_t(n), 1);
    for (int32_t c = 0; c < n; c++) {
        const int32_t p = t->parent[size_t(c)];
        if (p < 0) continue;
        if (first[size_t(p)] < 0) first[size_t(p)] = c;
        cnt[size_t(p)]++;
    }
    for (int32_t c = n - 1; c > 0; c--)  // a child's id is above its parent's
        if (t->parent[size_t(c)] >= 0) size[size_t(t->parent[size_t(c)])] += size[size_t(c)];
    std::vector<std::pair<int32_t, int32_t>> stack;  // (node, depth)
    int32_t pos = 0;
    for (const int32_t r : t->roots) {
        stack.emplace_back(r, 0);
        while (!stack.empty()) {
            const auto [x, d] = stack.back();
            stack.pop_back();
            t->pre_node[size_t(pos)] = x;
            t->pre_depth[size_t(pos)] = d;
            t->pre_size[size_t(pos)] = size[size_t(x)];
            pos++;
            for (int32_t k = cnt[size_t(x)] - 1; k >= 0; k--) stack.emplace_back(first[size_t(x)] + k, d + 1);
        }
    }
}

void pack_token_bytes(const uint8_t *bytes, const int64_t *offsets, int32_t V, uint32_t *tok_off,
                      uint16_t *tok_len, uint8_t *blob) {
    uint32_t pos = 0;
    for (int32_t v = 0; v < V; v++) {
        const int64_t L = (v == V - 1) ? 0 : offsets[v + 1] - offsets[v];  // EOS bytes are ignored
        tok_off[v] = pos;
        tok_len[v] = uint16_t(L);
        if (L > 0) memcpy(blob + pos, bytes + offsets[v], size_t(L));
        pos += uint32_t((L + 15) / 16 * 16);
    }
}

bool fill_token_table(const uint8_t *bytes, const int64_t *offsets, const uint16_t *tok_len, int32_t V,
                      uint64_t S, uint64_t *key, int32_t *val) {
    // load factor <= 1/4; slots are probed in aligned pairs (one 16-byte load
    // holds two keys), pair after pair, the even slot of a pair filled first
    std::fill(key, key + S, 0ull);
    std::fill(val, val + S, -1);
    const uint64_t pairs_mask = S / 2 - 1;
    bool dup = false;
    for (int32_t v = 0; v < V; v++) {
        const uint32_t L = tok_len[v];
        if (!L) continue;
        const uint8_t *p = bytes + offsets[v];
        uint64_t h = 0;
        for (uint32_t j = 0; j < L; j++) h = h * kHashBase + uint64_t(p[j]) + 1;
        const uint64_t k = hash_finish(h, L);
        uint64_t pair = (k >> 1) & pairs_mask;
        for (;;) {
            const size_t s0 = size_t(2 * pair);
            // an equal key: a repeated token string, or two strings whose hashes collide
            if (key[s0] == k || key[s0 + 1] == k) dup = true;
            if (!key[s0]) { key[s0] = k; val[s0] = v; break; }
            if (!key[s0 + 1]) { key[s0 + 1] = k; val[s0 + 1] = v; break; }
            pair = (pair + 1) & pairs_mask;
        }
    }
    return dup;
}

uint64_t token_table_slots(int64_t n_tokens_with_bytes) {
    uint64_t S = 16;
    while (S < uint64_t(4 * n_tokens_with_bytes)) S <<= 1;
    return S;
}

namespace {

// One subtree of the reversed-token trie: the tokens whose last byte is b,
// sorted by their reversed bytes, laid out in pre-order (local node 0 is the
// root's child for b).
struct RevPart {
    hvec<int32_t> parent;  // local ids; -1 for local node 0
    hvec<uint8_t> label;
    hvec<int32_t> token;
    std::vector<std::pair<int32_t, int32_t>> dup;  // (earlier id, later id) with equal bytes
};

void build_rev_part(const uint8_t *bytes, const int64_t *offsets, std::vector<int32_t> &ids, RevPart *out) {
    // reversed byte i of token v
    auto rb = [&](int32_t v, int64_t i) { return bytes[offsets[v + 1] - 1 - i]; };
    auto len = [&](int32_t v) { return offsets[v + 1] - offsets[v]; };
    std::vector<std::pair<uint64_t, int32_t>> keyed(ids.size());
    for (size_t i = 0; i < ids.size(); i++) {
        const int32_t v = ids[i];
        uint64_t k = 0;
        for (int j = 0; j < 8; j++) k = (k << 8) | (j < len(v) ? rb(v, j) : 0);
        keyed[i] = {k, v};
    }
    auto less = [&](const std::pair<uint64_t, int32_t> &a, const std::pair<uint64_t, int32_t> &b) {
        if (a.first != b.first) return a.first < b.first;
        const int64_t la = len(a.second), lb = len(b.second), m = std::min(la, lb);
        for (int64_t i = 8; i < m; i++) {
            const uint8_t x = rb(a.second, i), y = rb(b.second, i);
            if (x != y) return x < y;
        }
        if (la != lb) return la < lb;
        return a.second < b.second;  // equal bytes: ascending id
    };
    std::sort(keyed.begin(), keyed.end(), less);
    int64_t total = 0;
    for (const auto &kv : keyed) total += len(kv.second);
    out->parent.resize(size_t(total));
    out->label.resize(size_t(total));
    out->token.resize(size_t(total));
    int32_t n = 0;
    std::vector<int32_t> path;  // path[d] = local node at depth d + 1
    int32_t prev = -1;
    for (const auto &kv : keyed) {
        const int32_t v = kv.second;
        const int64_t L = len(v);
        int64_t lcp = 0;
        if (prev >= 0) {
            const int64_t m = std::min(len(prev), L);
            while (lcp < m && rb(prev, lcp) == rb(v, lcp)) lcp++;
            if (lcp == L && len(prev) == L) {  // the same bytes as the previous token
                out->dup.emplace_back(prev, v);
                prev = v;
                continue;
            }
        }
        if (int64_t(path.size()) < L) path.resize(size_t(L));
        for (int64_t d = lcp; d < L; d++) {
            const int32_t id = n++;
            out->parent[size_t(id)] = d == 0 ? -1 : path[size_t(d - 1)];
            out->label[size_t(id)] = rb(v, d);
            out->token[size_t(id)] = -1;
            path[size_t(d)] = id;
        }
        out->token[size_t(path[size_t(L - 1)])] = v;
        prev = v;
    }
    out->parent.resize(size_t(n));
    out->label.resize(size_t(n));
    out->token.resize(size_t(n));
}

}  // namespace

std::string build_reversed_token_trie(const uint8_t *bytes, const int64_t *offsets, int32_t V,
                                      RevTokenTrie *out) {
    // tokens with bytes (EOS = V-1 excluded), bucketed by their last byte
    std::vector<std::vector<int32_t>> bucket(256);
    for (int32_t v = 0; v + 1 < V; v++)
        if (offsets[v + 1] > offsets[v]) bucket[bytes[offsets[v + 1] - 1]].push_back(v);
    std::vector<RevPart> part(256);
    const unsigned hw = std::max(1u, std::thread::hardware_concurrency());
    const unsigned nth = std::min<unsigned>(hw, 16u);
    std::atomic<int> next(0);
    auto loop = [&]() {
        for (int b; (b = next.fetch_add(1)) < 256;)
            if (!bucket[size_t(b)].empty()) build_rev_part(bytes, offsets, bucket[size_t(b)], &part[size_t(b)]);
    };
    std::vector<std::thread> th;
    for (unsigned t = 1; t < nth; t++) th.emplace_back(loop);
    loop();
    for (auto &t : th) t.join();
    int64_t n = 1;
    std::vector<int64_t> base(256);
    for (int b = 0; b < 256; b++) {
        base[size_t(b)] = n;
        n += int64_t(part[size_t(b)].parent.size());
    }
    if (n > kRevTrieMaxNodes) return "reversed-token trie would exceed 2^24 - 2 nodes";
    out->n = int32_t(n);
    out->parent.resize(size_t(n));
    out->label.resize(size_t(n));
    out->token.resize(size_t(n));
    out->parent[0] = -1;
    out->label[0] = 0;
    out->token[0] = -1;
    bool dups = false;
    for (int b = 0; b < 256; b++) {
        const RevPart &p = part[size_t(b)];
        const int64_t g = base[size_t(b)];
        for (size_t i = 0; i < p.parent.size(); i++) {
            out->parent[size_t(g) + i] = p.parent[i] < 0 ? 0 : int32_t(g + p.parent[i]);
            out->label[size_t(g) + i] = p.label[i];
            out->token[size_t(g) + i] = p.token[i];
        }
        dups = dups || !p.dup.empty();
    }
    out->next.clear();
    out->max_mult = 1;
    if (dups) {
        out->next.assign(size_t(V), -1);
        std::vector<int32_t> is_later(size_t(V), 0);
        for (const RevPart &p : part)
            for (const auto &d : p.dup) {
                out->next[size_t(d.first)] = d.second;
                is_later[size_t(d.second)] = 1;
            }
        for (int32_t v = 0; v < V; v++) {  // chain heads: the longest chain
            if (is_later[size_t(v)] || out->next[size_t(v)] < 0) continue;
            int32_t len = 1;
            for (int32_t u = out->next[size_t(v)]; u >= 0; u = out->next[size_t(u)]) len++;
            out->max_mult = std::max(out->max_mult, len);
        }
    }
    return "";
}

std::string pack_vocab(const uint8_t *bytes, const int64_t *offsets, int32_t V, HostVocab *out) {
    if (V < 2) return "V must be >= 2 (token V-1 is EOS)";
    if (offsets[0] < 0) return "vocab offsets must be non-negative";
    out->V = V;
    uint64_t pos = 0;
    int64_t n_ins = 0;
    int32_t max_len = 0;
    for (int32_t v = 0; v < V; v++) {
        int64_t a = offsets[v], e = offsets[v + 1];
        if (e < a) return "vocab offsets must be non-decreasing";
        int64_t L = (v == V - 1) ? 0 : e - a;  // EOS bytes are ignored
        if (L > 65535) return "token " + std::to_string(v) + " is longer than 65535 bytes";
        pos += uint64_t((L + 15) / 16 * 16);
        if (pos > 0xFFFFFFF0ull) return "packed vocabulary exceeds 4 GiB";
        if (L > 0) {
            n_ins++;
            max_len = std::max<int32_t>(max_len, int32_t(L));
        }
    }
    out->max_len = max_len;
    out->tok_off.assign(size_t(V), 0);
    out->tok_len.assign(size_t(V), 0);
    out->blob.assign(size_t(pos) + 16, 0);
    pack_token_bytes(bytes, offsets, V, out->tok_off.data(), out->tok_len.data(), out->blob.data());
    const uint64_t S = token_table_slots(n_ins);
    if (S > (uint64_t(1) << 31)) return "vocabulary too large for the token hash table";
    out->ht_key.resize(size_t(S));
    out->ht_val.resize(size_t(S));
    out->ht_mask = uint32_t(S - 1);
    out->dup_keys = fill_token_table(bytes, offsets, out->tok_len.data(), V, S, out->ht_key.data(),
                                     out->ht_val.data()) ? 1 : 0;
    return "";
}

}  // namespace tmk
