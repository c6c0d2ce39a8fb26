/*
 * ac.c -- the paper's own mask precomputation on the CPU: an Aho-Corasick
 * automaton over the vocabulary and a pass over the enum trie that carries
 * the automaton state (Sec. 4.2 steps 1-2; App. G.1 Steps 2-3; App. H.4
 * Phases 3-4).
 *
 * TEST AND BENCH INFRASTRUCTURE ONLY, like the rest of oracle/: it is the
 * stronger timed CPU baseline and a third, independent check of the masks
 * (tests compare it with the brute-force oracle). It shares no code with the
 * CUDA path and takes the trie as plain arrays (parent, label, depth; node
 * ids breadth-first, so a parent always precedes its children).
 *
 * Automaton (Aho & Corasick 1975): the goto trie of every token's bytes (EOS,
 * id V-1, and byte-less tokens are left out), failure links computed breadth
 * first (the longest proper suffix of a state that is also a state), output
 * sets (the token ids ending at a state) and dictionary links (the nearest
 * state on the failure chain with a non-empty output set).
 *
 * Traversal: the automaton state of trie node m is the state after reading
 * the path string root -> m, i.e. delta(state(parent), label(m)); the
 * outputs found there are exactly the tokens that are suffixes of that path,
 * and a token of length L found at m is allowed at the node L levels above m
 * (App. G.1 Step 3). States are computed level by level (all parents first),
 * the nodes of a level in parallel.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int32_t n_states;
    int64_t edge_cap;       /* hash slots (power of two) */
    uint64_t *edge_key;     /* (state << 8 | byte) + 1, 0 = empty */
    int32_t *edge_val;      /* child state */
    int32_t *fail;
    int32_t *dict;          /* nearest failure-chain state with output, -1 if none */
    int32_t *out_head;      /* first token ending here, -1 if none */
    int32_t *out_next;      /* [V] next token with the same bytes, -1 */
    int32_t *tok_len;       /* [V] */
    int32_t V;
} ac_t;

static uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static int32_t goto_get(const ac_t *a, int32_t s, uint8_t c) {
    uint64_t key = (((uint64_t)s << 8) | c) + 1;
    uint64_t mask = (uint64_t)a->edge_cap - 1, i = mix64(key) & mask;
    while (a->edge_key[i]) {
        if (a->edge_key[i] == key) return a->edge_val[i];
        i = (i + 1) & mask;
    }
    return -1;
}

static void goto_put(ac_t *a, int32_t s, uint8_t c, int32_t v) {
    uint64_t key = (((uint64_t)s << 8) | c) + 1;
    uint64_t mask = (uint64_t)a->edge_cap - 1, i = mix64(key) & mask;
    while (a->edge_key[i]) i = (i + 1) & mask;
    a->edge_key[i] = key;
    a->edge_val[i] = v;
}

/* delta(s, c): follow failure links until a goto edge for c exists. */
static int32_t ac_step(const ac_t *a, int32_t s, uint8_t c) {
    for (;;) {
        int32_t v = goto_get(a, s, c);
        if (v >= 0) return v;
        if (s == 0) return 0;
        s = a->fail[s];
    }
}

void ac_free(ac_t *a) {
    if (!a) return;
    free(a->edge_key);
    free(a->edge_val);
    free(a->fail);
    free(a->dict);
    free(a->out_head);
    free(a->out_next);
    free(a->tok_len);
    free(a);
}

/* Automaton over tokens 0..V-2 that have bytes. NULL on allocation failure. */
ac_t *ac_build(const uint8_t *vb, const int64_t *vo, int32_t V) {
    ac_t *a = calloc(1, sizeof(ac_t));
    if (!a) return NULL;
    int64_t total = 0;
    for (int32_t v = 0; v + 1 < V; v++) total += vo[v + 1] - vo[v];
    int64_t max_states = total + 1;
    a->V = V;
    a->edge_cap = 16;
    while (a->edge_cap < 2 * max_states) a->edge_cap <<= 1;
    a->edge_key = calloc((size_t)a->edge_cap, sizeof(uint64_t));
    a->edge_val = malloc(sizeof(int32_t) * (size_t)a->edge_cap);
    a->fail = calloc((size_t)max_states, sizeof(int32_t));
    a->dict = malloc(sizeof(int32_t) * (size_t)max_states);
    a->out_head = malloc(sizeof(int32_t) * (size_t)max_states);
    a->out_next = malloc(sizeof(int32_t) * (size_t)V);
    a->tok_len = malloc(sizeof(int32_t) * (size_t)V);
    int32_t *bfs = malloc(sizeof(int32_t) * (size_t)max_states);
    int32_t *first = malloc(sizeof(int32_t) * (size_t)max_states); /* child lists for the BFS */
    int32_t *sib = malloc(sizeof(int32_t) * (size_t)max_states);
    uint8_t *lab = malloc((size_t)max_states);
    if (!a->edge_key || !a->edge_val || !a->fail || !a->dict || !a->out_head || !a->out_next ||
        !a->tok_len || !bfs || !first || !sib || !lab) {
        free(bfs); free(first); free(sib); free(lab); ac_free(a);
        return NULL;
    }
    memset(a->out_head, 0xff, sizeof(int32_t) * (size_t)max_states);
    memset(first, 0xff, sizeof(int32_t) * (size_t)max_states);
    int32_t n = 1;
    /* goto trie */
    for (int32_t v = 0; v < V; v++) {
        a->out_next[v] = -1;
        a->tok_len[v] = (v + 1 < V) ? (int32_t)(vo[v + 1] - vo[v]) : 0;
        if (v + 1 == V || a->tok_len[v] == 0) continue;
        int32_t s = 0;
        for (int64_t p = vo[v]; p < vo[v + 1]; p++) {
            int32_t c = goto_get(a, s, vb[p]);
            if (c < 0) {
                c = n++;
                goto_put(a, s, vb[p], c);
                lab[c] = vb[p];
                sib[c] = first[s];
                first[s] = c;
            }
            s = c;
        }
        a->out_next[v] = a->out_head[s];
        a->out_head[s] = v;
    }
    a->n_states = n;
    /* failure and dictionary links, breadth first */
    int32_t head = 0, tail = 0;
    a->fail[0] = 0;
    a->dict[0] = -1;
    for (int32_t c = first[0]; c >= 0; c = sib[c]) {
        a->fail[c] = 0;
        a->dict[c] = -1;
        bfs[tail++] = c;
    }
    while (head < tail) {
        int32_t u = bfs[head++];
        for (int32_t c = first[u]; c >= 0; c = sib[c]) {
            int32_t f = a->fail[u];
            int32_t g;
            for (;;) {
                g = goto_get(a, f, lab[c]);
                if (g >= 0 || f == 0) break;
                f = a->fail[f];
            }
            a->fail[c] = (g >= 0 && g != c) ? g : 0;
            int32_t fc = a->fail[c];
            a->dict[c] = (a->out_head[fc] >= 0) ? fc : a->dict[fc];
            bfs[tail++] = c;
        }
    }
    free(bfs); free(first); free(sib); free(lab);
    return a;
}

int32_t ac_num_states(const ac_t *a) { return a->n_states; }

/* Automaton state of every trie node (parent before child; depth[] gives the
 * levels, which are contiguous in breadth-first order). */
static void ac_states(const ac_t *a, int32_t n, const int32_t *parent, const uint8_t *label,
                      const int32_t *depth, int32_t *q, int32_t nthreads) {
    int32_t lo = 0;
    while (lo < n) {
        int32_t hi = lo;
        while (hi < n && depth[hi] == depth[lo]) hi++;
#ifdef _OPENMP
#pragma omp parallel for schedule(static) num_threads(nthreads > 0 ? nthreads : 1)
#endif
        for (int32_t m = lo; m < hi; m++)
            q[m] = parent[m] < 0 ? 0 : ac_step(a, q[parent[m]], label[m]);
        lo = hi;
    }
    (void)nthreads;
}

static int32_t ancestor(const int32_t *parent, int32_t m, int32_t L) {
    while (L-- > 0 && m >= 0) m = parent[m];
    return m;
}

/* Every allowed (start node, token) pair, EOS excluded: pass 1 counts the
 * outputs per node, pass 2 writes them. Returns the number of pairs; writes
 * them to rows[] / toks[] only if it is <= cap. */
int64_t ac_valid_pairs(const ac_t *a, int32_t n, const int32_t *parent, const uint8_t *label,
                       const int32_t *depth, int32_t *rows, int32_t *toks, int64_t cap,
                       int32_t nthreads) {
    int32_t *q = malloc(sizeof(int32_t) * (size_t)(n > 0 ? n : 1));
    int64_t *off = malloc(sizeof(int64_t) * (size_t)(n + 1));
    if (!q || !off) { free(q); free(off); return -1; }
    ac_states(a, n, parent, label, depth, q, nthreads);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 256) num_threads(nthreads > 0 ? nthreads : 1)
#endif
    for (int32_t m = 0; m < n; m++) {
        int64_t c = 0;
        for (int32_t x = a->out_head[q[m]] >= 0 ? q[m] : a->dict[q[m]]; x > 0; x = a->dict[x])
            for (int32_t t = a->out_head[x]; t >= 0; t = a->out_next[t]) c++;
        off[m + 1] = c;
    }
    off[0] = 0;
    for (int32_t m = 0; m < n; m++) off[m + 1] += off[m];
    int64_t total = off[n];
    if (total <= cap) {
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 256) num_threads(nthreads > 0 ? nthreads : 1)
#endif
        for (int32_t m = 0; m < n; m++) {
            int64_t o = off[m];
            for (int32_t x = a->out_head[q[m]] >= 0 ? q[m] : a->dict[q[m]]; x > 0; x = a->dict[x])
                for (int32_t t = a->out_head[x]; t >= 0; t = a->out_next[t]) {
                    rows[o] = ancestor(parent, m, a->tok_len[t]);
                    toks[o] = t;
                    o++;
                }
        }
    }
    free(q);
    free(off);
    (void)nthreads;
    return total;
}
