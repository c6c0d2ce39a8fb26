/*
 * oracle.c -- plain, slow, brute-force CPU oracle for the trie automaton.
 *
 * TEST INFRASTRUCTURE ONLY. Only tests/, the smoke check and the bench's
 * CPU-baseline leg may load this file's library. The CUDA path shares no
 * code, header, table or helper with it.
 *
 * What it computes (Xu & Bouyarmane, "Trie Automata for Constrained Decoding
 * over Large Finite Sets"):
 *
 *  - The character (byte) trie of the enum set E = {e_1..e_K} (Sec. 4.1,
 *    App. G.1 Step 1): every string inserted byte by byte, shared prefixes
 *    merged, a node marked terminal where some e_i ends. Duplicate strings
 *    collapse (E is a set); the empty string makes the root terminal.
 *    Node ids follow one canonical order: breadth first from the root,
 *    siblings by ascending byte; root = 0.
 *
 *  - valid[n] by its definition, not by Aho-Corasick (Sec. 4.1; Sec. 4.2
 *    step 2; App. G.5 proof, conditions (i)+(ii)): token v is valid at node n
 *    iff every byte of v, walked from n, finds a child edge. Landing on a
 *    leaf is allowed, overshooting it is not. Because every trie node is a
 *    prefix of some e_i, condition (ii) then holds automatically. A token
 *    with no bytes is never valid. The AC traversal of Sec. 4.2 reaches
 *    exactly this set; the oracle is the naive O(N * V * l) walk the paper
 *    names as the definition (Sec. 4.1, last paragraph).
 *
 *  - EOS (id V-1, its bytes ignored): allowed at n iff n is terminal
 *    (App. G.5 "EOS token handling"; Sec. 4.2 step 2 for terminal nodes that
 *    are also internal).
 *
 *  - The state transition delta*(s, bytes(token)) (Sec. 2, Eq. 1 context):
 *    a byte walk. Our reading where the paper is silent: EOS at a terminal
 *    node -> FINISHED (-2); FINISHED + EOS -> FINISHED; every other move
 *    that the walk cannot make -> DEAD (-1); DEAD stays DEAD. Every move
 *    into DEAD from a state other than DEAD counts one error.
 *
 *  - Mask application (Sec. 4.2 last paragraph; App. H.3): logits of tokens
 *    whose bit is clear become -inf, the rest keep their bits. FINISHED and
 *    DEAD rows allow only EOS.
 *
 * Bit layout of a mask row: W = ceil(V/32) uint32 words, token v is bit
 * (v % 32) of word v / 32, bits >= V are zero.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_DEAD (-1)
#define ORACLE_FINISHED (-2)

typedef struct {
    int32_t n;         /* nodes */
    int32_t *child;    /* [n * 256] child id per byte, -1 if none */
    uint8_t *terminal; /* [n] */
    int32_t *parent;   /* [n], -1 for the root */
    uint8_t *label;    /* [n] byte on the edge into the node (0 for root) */
    int32_t *depth;    /* [n] */
    int64_t n_chars;   /* sum of |e| over the distinct strings */
} otrie;

void oracle_trie_free(otrie *t) {
    if (!t) return;
    free(t->child);
    free(t->terminal);
    free(t->parent);
    free(t->label);
    free(t->depth);
    free(t);
}

/* Build the byte trie of the K strings bytes[offsets[i]:offsets[i+1]].
 * Returns NULL on allocation failure or bad offsets. */
otrie *oracle_trie_build(const uint8_t *bytes, const int64_t *offsets, int32_t K) {
    /* 1. insertion-order trie with a dense 256-way child table */
    int64_t cap = 1024, n = 1;
    int32_t *ch = malloc(sizeof(int32_t) * 256 * cap);
    uint8_t *term = calloc(cap, 1);
    uint8_t *lab = calloc(cap, 1);
    if (!ch || !term || !lab) { free(ch); free(term); free(lab); return NULL; }
    memset(ch, 0xff, sizeof(int32_t) * 256);
    for (int32_t i = 0; i < K; i++) {
        if (offsets[i + 1] < offsets[i]) { free(ch); free(term); free(lab); return NULL; }
        int64_t x = 0;
        for (int64_t p = offsets[i]; p < offsets[i + 1]; p++) {
            uint8_t b = bytes[p];
            if (ch[x * 256 + b] < 0) {
                if (n == cap) {
                    int64_t nc = cap * 2;
                    int32_t *c2 = realloc(ch, sizeof(int32_t) * 256 * nc);
                    uint8_t *t2 = realloc(term, nc);
                    uint8_t *l2 = realloc(lab, nc);
                    if (c2) ch = c2;
                    if (t2) term = t2;
                    if (l2) lab = l2;
                    if (!c2 || !t2 || !l2) { free(ch); free(term); free(lab); return NULL; }
                    memset(term + cap, 0, nc - cap);
                    cap = nc;
                }
                memset(ch + n * 256, 0xff, sizeof(int32_t) * 256);
                lab[n] = b;
                ch[x * 256 + b] = (int32_t)n;
                n++;
            }
            x = ch[x * 256 + b];
        }
        term[x] = 1;
    }
    /* 2. breadth-first renumbering, siblings by ascending byte */
    int32_t *order = malloc(sizeof(int32_t) * n); /* new id -> old id */
    int32_t *newid = malloc(sizeof(int32_t) * n); /* old id -> new id */
    otrie *t = calloc(1, sizeof(otrie));
    if (!order || !newid || !t) { free(order); free(newid); free(t); free(ch); free(term); free(lab); return NULL; }
    int64_t head = 0, tail = 0;
    order[tail++] = 0;
    while (head < tail) {
        int32_t x = order[head++];
        for (int b = 0; b < 256; b++)
            if (ch[(int64_t)x * 256 + b] >= 0) order[tail++] = ch[(int64_t)x * 256 + b];
    }
    for (int64_t i = 0; i < n; i++) newid[order[i]] = (int32_t)i;
    t->n = (int32_t)n;
    t->child = malloc(sizeof(int32_t) * 256 * n);
    t->terminal = malloc(n);
    t->parent = malloc(sizeof(int32_t) * n);
    t->label = malloc(n);
    t->depth = malloc(sizeof(int32_t) * n);
    if (!t->child || !t->terminal || !t->parent || !t->label || !t->depth) {
        free(order); free(newid); free(ch); free(term); free(lab); oracle_trie_free(t); return NULL;
    }
    t->parent[0] = -1;
    t->depth[0] = 0;
    t->n_chars = 0;
    for (int64_t i = 0; i < n; i++) {
        int32_t o = order[i];
        t->terminal[i] = term[o];
        t->label[i] = lab[o];
        for (int b = 0; b < 256; b++) {
            int32_t c = ch[(int64_t)o * 256 + b];
            t->child[i * 256 + b] = c < 0 ? -1 : newid[c];
        }
    }
    /* parents and depths follow from the child table (BFS: parent before child) */
    for (int64_t i = 0; i < n; i++)
        for (int b = 0; b < 256; b++) {
            int32_t c = t->child[i * 256 + b];
            if (c >= 0) { t->parent[c] = (int32_t)i; t->depth[c] = t->depth[i] + 1; }
        }
    for (int64_t i = 0; i < n; i++)
        if (t->terminal[i]) t->n_chars += t->depth[i];
    free(order); free(newid); free(ch); free(term); free(lab);
    return t;
}

int32_t oracle_trie_num_nodes(const otrie *t) { return t->n; }
int64_t oracle_trie_num_chars(const otrie *t) { return t->n_chars; }
int32_t oracle_trie_child(const otrie *t, int32_t node, int32_t byte) {
    return t->child[(int64_t)node * 256 + byte];
}

void oracle_trie_info(const otrie *t, int32_t *parent, uint8_t *label, uint8_t *terminal,
                      int32_t *depth) {
    memcpy(parent, t->parent, sizeof(int32_t) * t->n);
    memcpy(label, t->label, t->n);
    memcpy(terminal, t->terminal, t->n);
    memcpy(depth, t->depth, sizeof(int32_t) * t->n);
}

/* End node of the byte walk of token v from node n, or -1 if it leaves the trie
 * (or if v has no bytes). */
static int32_t walk(const otrie *t, int32_t n, const uint8_t *vb, const int64_t *vo, int32_t v) {
    int64_t a = vo[v], e = vo[v + 1];
    if (e <= a) return -1;
    int32_t x = n;
    for (int64_t p = a; p < e; p++) {
        x = t->child[(int64_t)x * 256 + vb[p]];
        if (x < 0) return -1;
    }
    return x;
}

/* One mask row for node n (or for FINISHED / DEAD: only EOS) into row[W]. */
static void mask_row(const otrie *t, const uint8_t *vb, const int64_t *vo, int32_t V,
                     int32_t n, uint32_t *row) {
    int32_t W = (V + 31) / 32;
    int32_t eos = V - 1;
    memset(row, 0, sizeof(uint32_t) * W);
    int node = (n >= 0 && n < t->n);
    if (node) {
        for (int32_t v = 0; v < eos; v++)
            if (walk(t, n, vb, vo, v) >= 0) row[v / 32] |= 1u << (v % 32);
    }
    if (!node || t->terminal[n]) row[eos / 32] |= 1u << (eos % 32);
}

/* Mask rows for the node ids rows[0..nrows), into out[nrows * W].
 * An id that is not a node (FINISHED, DEAD, out of range) gives the row {EOS}.
 * Rows are independent; nthreads > 1 splits them over OpenMP threads. */
void oracle_mask_rows(const otrie *t, const uint8_t *vb, const int64_t *vo, int32_t V,
                      const int32_t *rows, int64_t nrows, uint32_t *out, int32_t nthreads) {
    int64_t W = (V + 31) / 32;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 4) num_threads(nthreads > 0 ? nthreads : 1)
#endif
    for (int64_t i = 0; i < nrows; i++) mask_row(t, vb, vo, V, rows[i], out + i * W);
    (void)nthreads;
}

/* delta* for a batch: states[b] <- next state after tokens[b]. Returns the
 * number of moves into DEAD from a state other than DEAD. */
int64_t oracle_advance(const otrie *t, const uint8_t *vb, const int64_t *vo, int32_t V,
                       int32_t *states, const int32_t *tokens, int64_t B) {
    int64_t errors = 0;
    int32_t eos = V - 1;
    for (int64_t b = 0; b < B; b++) {
        int32_t s = states[b], v = tokens[b], nxt;
        if (s == ORACLE_DEAD) continue;
        if (v < 0 || v >= V) nxt = ORACLE_DEAD;
        else if (s == ORACLE_FINISHED) nxt = (v == eos) ? ORACLE_FINISHED : ORACLE_DEAD;
        else if (s < 0 || s >= t->n) nxt = ORACLE_DEAD;
        else if (v == eos) nxt = t->terminal[s] ? ORACLE_FINISHED : ORACLE_DEAD;
        else {
            int32_t e = walk(t, s, vb, vo, v);
            nxt = e >= 0 ? e : ORACLE_DEAD;
        }
        if (nxt == ORACLE_DEAD) errors++;
        states[b] = nxt;
    }
    return errors;
}

/* logits[b][v] <- -inf where v is not allowed at states[b]; other entries keep
 * their bits. dtype 0: fp32 words (-inf = 0xFF800000); dtype 1: bf16 halves
 * (-inf = 0xFF80). Logits are handled as raw bit patterns. */
void oracle_apply(const otrie *t, const uint8_t *vb, const int64_t *vo, int32_t V,
                  void *logits, int32_t dtype, const int32_t *states, int64_t B) {
    int64_t W = (V + 31) / 32;
    uint32_t *row = malloc(sizeof(uint32_t) * W);
    if (!row) return;
    for (int64_t b = 0; b < B; b++) {
        mask_row(t, vb, vo, V, states[b], row);
        for (int64_t v = 0; v < V; v++) {
            if ((row[v / 32] >> (v % 32)) & 1u) continue;
            if (dtype == 0) ((uint32_t *)logits)[b * V + v] = 0xFF800000u;
            else ((uint16_t *)logits)[b * V + v] = 0xFF80u;
        }
    }
    free(row);
}

/* Greedy choice per row: the largest logit, the lowest id among equals.
 * bf16 values widen exactly to fp32 (the 16 bits become the high half). */
void oracle_argmax(const void *logits, int32_t dtype, int64_t B, int32_t V, int32_t *out) {
    for (int64_t b = 0; b < B; b++) {
        int32_t best = 0;
        float bv = 0.0f;
        for (int32_t v = 0; v < V; v++) {
            float x;
            if (dtype == 0) {
                memcpy(&x, (const uint32_t *)logits + b * V + v, 4);
            } else {
                uint32_t w = (uint32_t)((const uint16_t *)logits)[b * V + v] << 16;
                memcpy(&x, &w, 4);
            }
            if (v == 0 || x > bv) { bv = x; best = v; }
        }
        out[b] = best;
    }
}

/* ------------------------------------------------------------------------
 * Character-position masks for fixed-format strings (App. K, "constraint-
 * aware dispatch beyond finite sets"): a format of length L is a sequence of
 * byte classes C_0..C_{L-1}; class i allows byte c iff bit (c % 8) of
 * classes[32 * i + c / 8] is set. The strings of the format are the
 * products C_0 x ... x C_{L-1}; the automaton's states are the positions
 * 0..L (position p: p bytes written).
 *
 *  - valid[p]: token v (not EOS) iff 1 <= len(v) <= L - p and byte i of v is
 *    in C_{p+i} for every i (the position-wise character check of App. K);
 *    EOS iff p == L. Every position p < L has a continuation in the format,
 *    so this is the same live-path condition as the trie's (App. G.5).
 *  - advance: a valid token moves p to p + len(v); EOS at L -> FINISHED;
 *    FINISHED + EOS -> FINISHED; DEAD stays DEAD; anything else -> DEAD (one
 *    error per move into DEAD), as for the trie.
 * ---------------------------------------------------------------------- */

static int fmt_class_has(const uint8_t *classes, int32_t i, uint8_t c) {
    return (classes[32 * (int64_t)i + c / 8] >> (c % 8)) & 1;
}

static int fmt_valid(const uint8_t *classes, int32_t L, const uint8_t *vb, const int64_t *vo,
                     int32_t V, int32_t p, int32_t v) {
    if (v == V - 1) return p == L;
    int64_t len = vo[v + 1] - vo[v];
    if (len < 1 || len > (int64_t)(L - p)) return 0;
    for (int64_t i = 0; i < len; i++)
        if (!fmt_class_has(classes, p + (int32_t)i, vb[vo[v] + i])) return 0;
    return 1;
}

static void fmt_row(const uint8_t *classes, int32_t L, const uint8_t *vb, const int64_t *vo, int32_t V,
                    int32_t p, uint32_t *row) {
    int64_t W = (V + 31) / 32;
    memset(row, 0, sizeof(uint32_t) * W);
    if (p < 0 || p > L) {  /* FINISHED, DEAD, not a position: {EOS} */
        row[(V - 1) / 32] |= 1u << ((V - 1) % 32);
        return;
    }
    for (int32_t v = 0; v < V; v++)
        if (fmt_valid(classes, L, vb, vo, V, p, v)) row[v / 32] |= 1u << (v % 32);
}

void oracle_fmt_mask_rows(const uint8_t *classes, int32_t L, const uint8_t *vb, const int64_t *vo,
                          int32_t V, const int32_t *rows, int64_t nrows, uint32_t *out) {
    int64_t W = (V + 31) / 32;
    for (int64_t i = 0; i < nrows; i++) fmt_row(classes, L, vb, vo, V, rows[i], out + i * W);
}

int64_t oracle_fmt_advance(const uint8_t *classes, int32_t L, const uint8_t *vb, const int64_t *vo,
                           int32_t V, int32_t *states, const int32_t *tokens, int64_t B) {
    int64_t errors = 0;
    int32_t eos = V - 1;
    for (int64_t b = 0; b < B; b++) {
        int32_t s = states[b], v = tokens[b], nxt;
        if (s == ORACLE_DEAD) continue;
        if (v < 0 || v >= V) nxt = ORACLE_DEAD;
        else if (s == ORACLE_FINISHED) nxt = v == eos ? ORACLE_FINISHED : ORACLE_DEAD;
        else if (s < 0 || s > L) nxt = ORACLE_DEAD;
        else if (v == eos) nxt = (s == L) ? ORACLE_FINISHED : ORACLE_DEAD;
        else nxt = fmt_valid(classes, L, vb, vo, V, s, v) ? s + (int32_t)(vo[v + 1] - vo[v]) : ORACLE_DEAD;
        errors += nxt == ORACLE_DEAD;
        states[b] = nxt;
    }
    return errors;
}

