/*
 * triemask.h -- C ABI of libtriemask.so: GB300 (sm_103a) trie-automaton token
 * masks for constrained decoding over a finite string set.
 *
 * Method: Xu & Bouyarmane, "Trie Automata for Constrained Decoding over Large
 * Finite Sets". Given an enum set E = {e_1..e_K} of byte strings and a byte
 * vocabulary of V tokens, the library
 *   1. builds the byte trie of E on the host (Sec. 4.1; App. G.1 Step 1),
 *   2. computes valid[n] for every trie node n as a dense bitmask
 *      [num_nodes, ceil(V/32)] uint32 on the GPU (Sec. 4.1-4.2; App. G.1
 *      Steps 3-4; App. G.5 proof conditions (i)+(ii); EOS handling per App.
 *      G.5 "EOS token handling"),
 *   3. advances a batch of decode states by their sampled tokens,
 *      s' = delta*(s, bytes(token)) (Sec. 2, Eq. 1),
 *   4. writes -inf into the logits of every token not in valid[s]
 *      (Sec. 4.2 last paragraph; App. H.3, the cost of applying the bitmask).
 *
 * Conventions shared by every call
 * --------------------------------
 * Strings and tokens are raw bytes (every byte 0x00-0xFF is legal), passed
 * as a concatenated byte array plus int64 offsets[count+1]; string i is
 * bytes[offsets[i] : offsets[i+1]]. Host pointers are read during the call
 * only; the library keeps its own copies.
 *
 * Node ids: breadth-first from the root, siblings by ascending byte, root 0.
 * Equivalently, the distinct prefixes of E sorted by (length, bytes).
 * A forest (trie_build_many) concatenates the tries of its sets in order;
 * states are then global node ids and trie_root() gives each set's root.
 *
 * Token V-1 is EOS: its bytes are ignored. It is allowed at node n iff some
 * e_i ends at n. Any other token with no bytes is never allowed.
 *
 * Mask layout: row n is W = ceil(V/32) uint32 words; token v is bit (v % 32)
 * of word v / 32 (LSB first); bits >= V are zero.
 *
 * States: a node id, TRIE_STATE_FINISHED (EOS was taken at a terminal node)
 * or TRIE_STATE_DEAD (a move the trie does not allow). FINISHED and DEAD
 * rows allow only EOS.
 *
 * Errors: every call returns TRIE_OK (0) or a negative code and never
 * aborts; trie_last_error() gives a message for the calling thread. Argument
 * checks are synchronous. Kernel launch failures return TRIE_ECUDA; faults
 * inside an asynchronous kernel surface on a later CUDA call or sync.
 * Kernels never trap.
 *
 * Ownership: the library owns the trie (host and device copies) and the
 * packed vocabularies (device). The caller owns every device buffer it
 * passes (mask, states, tokens, logits, error counter). The mask passed to
 * trie_compile_masks must stay allocated and unchanged while the handle is
 * used by trie_apply_mask (the handle keeps a non-owning pointer to it).
 * A handle's device memory (trie arrays and per-node tables, 123 B per
 * node, plus a transition table of at least 128 B per node for a single trie;
 * the dense compile's hit buffer, 129 B per node, allocated by the
 * handle's first trie_compile_masks; valid lists; lazy rows) and the
 * scratch of trie_build_many_device come from a memory pool per device that
 * the library creates on first use; up to 8 GiB of memory freed by
 * trie_destroy stays reserved in it for later handles until the process
 * exits, so building and destroying a handle per batch maps no new memory.
 *
 * Streams: device work is enqueued on the given stream (0 = legacy default)
 * and is asynchronous with respect to the host. Concurrent trie_advance /
 * trie_apply_mask calls on one handle are safe (they only read the trie and
 * the mask); trie_compile_masks and trie_destroy must not race with other
 * calls on the same handle.
 */
#ifndef TRIEMASK_H
#define TRIEMASK_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct trie_s *trie_t; /* opaque; owned by the library */

enum {
    TRIE_OK = 0,
    TRIE_EINVAL = -1, /* bad argument (null pointer, bad offsets, size out of range) */
    TRIE_ENOMEM = -2, /* host or device allocation failed */
    TRIE_ECUDA = -3,  /* a CUDA runtime call failed */
    TRIE_ESTATE = -4  /* call out of order (e.g. apply before compile) */
};

enum { TRIE_DTYPE_F32 = 0, TRIE_DTYPE_BF16 = 1 };

#define TRIE_STATE_DEAD (-1)
#define TRIE_STATE_FINISHED (-2)

/* Build the byte trie of K strings (Sec. 4.1: insert each value character by
 * character, merging shared prefixes; App. G.1 Step 1). Host only: no device
 * memory is touched until the first device call on the handle.
 *   bytes    host, offsets[K] bytes (may be NULL when that is 0)
 *   offsets  host int64[K+1], non-decreasing, offsets[0] >= 0
 *   K        >= 0; K = 0 gives a lone root
 *   out      receives the handle (release with trie_destroy)
 * Duplicate strings collapse; the empty string marks the root terminal.
 * Returns TRIE_EINVAL on bad offsets or K < 0, TRIE_ENOMEM on allocation
 * failure or more than 2^31-1 nodes. */
int trie_build(const uint8_t *bytes, const int64_t *offsets, int32_t K, trie_t *out);

/* Build one forest of M independent tries (per-request sets). Set i holds the
 * strings set_offsets[i] .. set_offsets[i+1]-1 of the string list given by
 * (bytes, offsets). Node ids of set i start at trie_root(h, i).
 *   set_offsets  host int32[M+1], non-decreasing, set_offsets[0] = 0
 *   M            >= 1
 * Sets are built on host threads in parallel. Errors as trie_build. */
int trie_build_many(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets,
                    int32_t M, trie_t *out);

/* trie_build_many with the insertion of Sec. 4.1 (App. G.1 Step 1) run on the
 * current device, for per-request sets that change with every batch. The
 * handle's node numbering, terminal flags, roots and statistics equal those
 * of trie_build_many for the same arguments.
 *   Arguments as trie_build_many (all host, read during the call); stream is
 *   the stream the build kernels and the copies run on.
 * The strings are staged on the device and inserted level by level (depth
 * d = 0, 1, ...) for all sets at once; the trie lives on the device only and
 * is bound to the current device. Where the device reads pageable host
 * memory coherently through the host's page tables (Grace CPUs over
 * NVLink-C2C), a kernel reads the strings straight from the caller's arrays;
 * elsewhere they are copied first (TRIEMASK_HOST_READ=copy in the
 * environment forces the copies). The offsets are checked on the device.
 * Returns once the node count and the roots are known on the host (read back
 * after the level insertion; the caller's arrays have been read by then):
 * the last kernels (the breadth-first layout, child links and per-node
 * tables) are still queued on `stream`, so use the handle on `stream` or
 * after synchronising it (calls that copy arrays back synchronise the device
 * first); an error in those kernels surfaces on a later call. Such a
 * forest has no transition table: trie_advance and the fused calls walk the
 * tokens' bytes. Calls that need the host arrays (trie_get_csr,
 * trie_lazy_init) copy them back once. Strings longer than 1024 bytes, more
 * than 2^24 (set, depth) pairs or more than 2^31-3 string bytes plus sets
 * are built by trie_build_many on the host instead. Device scratch (about
 * 20 bytes per string byte plus 90 per string) is taken from the library's
 * device memory pool on `stream` and released there. Errors as
 * trie_build_many; TRIE_ENOMEM if a device allocation fails, TRIE_ECUDA if
 * another CUDA call fails. */
int trie_build_many_device(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets,
                           int32_t M, cudaStream_t stream, trie_t *out);

/* Number of nodes (the mask has this many rows); -1 for a NULL handle. */
int32_t trie_num_nodes(trie_t h);

/* Root node id of set i (0 for a single trie); -1 if i is out of range. */
int32_t trie_root(trie_t h, int32_t i);
/* All roots at once: roots (host int32[trie_num_sets(h)]) receives the root
 * node id of every set, in set order (a forest of many sets, in one call). */
int trie_copy_roots(trie_t h, int32_t *roots);

/* Number of sets in the handle (1 for trie_build). */
int32_t trie_num_sets(trie_t h);

/* Trie statistics: total bytes of the distinct strings (N_chars of Sec. 4.1)
 * and the deepest node's depth. */
int64_t trie_num_chars(trie_t h);
int32_t trie_max_depth(trie_t h);

/* Copy the host CSR out (for inspection and tests). Each pointer may be NULL.
 *   parent       int32[N]   parent id, -1 for a root
 *   label        uint8[N]   byte on the edge into the node (0 for a root)
 *   terminal     uint8[N]   1 where some string of the node's set ends
 *   first_child  int32[N]   id of the first child (children are contiguous
 *                           and sorted by byte); -1 for a leaf */
int trie_get_csr(trie_t h, int32_t *parent, uint8_t *label, uint8_t *terminal,
                 int32_t *first_child);

/* Compute valid[n] for every node n of the handle into a dense bitmask
 * (Sec. 4.2: the per-node valid sets, here for all nodes at once; App. G.1
 * Steps 3-4).
 *   vocab_bytes, vocab_offsets  host; V tokens, token V-1 is EOS
 *   V        2 <= V <= 2^31-32; every token at most 65535 bytes
 *   d_mask   device, caller-allocated, num_nodes * ceil(V/32) uint32,
 *            16-byte aligned for the vector path (any 4-byte alignment works)
 *   stream   CUDA stream for the kernels
 * The vocabulary is packed and uploaded on its first use on the current
 * device (the per-tokenizer step the paper caches, Sec. 4.2) and reused by
 * later calls with byte-identical vocab arrays. The first device call on a
 * handle also uploads the trie. d_mask is written asynchronously on stream;
 * the handle records (d_mask, V, vocabulary) for trie_advance and
 * trie_apply_mask. Errors: TRIE_EINVAL (bad sizes or pointers), TRIE_ENOMEM,
 * TRIE_ECUDA. */
int trie_compile_masks(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets,
                       int32_t V, uint32_t *d_mask, cudaStream_t stream);

/* Vocabulary handles (App. H.4 Phases 2-3: a vocabulary is packed and
 * uploaded once). The entry points that take vocab_bytes / vocab_offsets / V
 * find an uploaded vocabulary by comparing the caller's arrays with the
 * cached copies, byte by byte, on every call (for a 128,000-token vocabulary
 * about 60 us of host time before the first launch). A handle names the
 * vocabulary instead and skips that comparison.
 *   trie_vocab_create  packs and uploads the vocabulary (as the first
 *                      trie_compile_masks would) on the current device, or
 *                      takes the already uploaded copy; arguments as
 *                      trie_compile_masks; *out receives the handle (NULL on
 *                      error). Host-synchronous. Errors: TRIE_EINVAL,
 *                      TRIE_ENOMEM, TRIE_ECUDA.
 *   trie_vocab_size    V of the handle; -1 for NULL.
 *   trie_vocab_destroy releases the handle (NULL is a no-op). The device copy
 *                      is freed when neither the library's cache of recent
 *                      vocabularies nor a trie handle that compiled with it
 *                      still holds it; that cudaFree synchronises the device.
 * The caller's arrays are not referenced after trie_vocab_create returns. */
typedef struct trie_vocab_s *trie_vocab_t; /* opaque; owned by the caller */
int trie_vocab_create(const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                      trie_vocab_t *out);
int32_t trie_vocab_size(trie_vocab_t v);
void trie_vocab_destroy(trie_vocab_t v);

/* trie_compile_masks with the vocabulary of handle v (V = trie_vocab_size(v)).
 * v must belong to the current device (else TRIE_EINVAL); the rest as
 * trie_compile_masks. */
int trie_compile_masks_vocab(trie_t h, trie_vocab_t v, uint32_t *d_mask, cudaStream_t stream);

/* Advance B decode states in place by one token each: s' = delta*(s, bytes(t))
 * (Sec. 2, Eq. 1; the paper's stateless character walk).
 *   d_states  device int32[B], in/out
 *   d_tokens  device int32[B]
 *   d_err     device int32 counter or NULL; incremented once for every state
 *             that moves into DEAD from a state other than DEAD
 * Rules: a token whose bytes walk from node s inside the trie -> the end node;
 * EOS at a terminal node -> FINISHED; FINISHED + EOS -> FINISHED; DEAD stays
 * DEAD; every other move (including a token id outside [0, V) or a state
 * that is not a node) -> DEAD. Needs a prior trie_compile_masks on the handle
 * (for its vocabulary), else TRIE_ESTATE. B = 0 is a no-op. */
int trie_advance(trie_t h, int32_t *d_states, const int32_t *d_tokens, int32_t B,
                 int32_t *d_err, cudaStream_t stream);

/* Mask a batch of logits in place (Sec. 4.2; App. H.3): logits[b][v] becomes
 * -inf (fp32 0xFF800000, bf16 0xFF80) where bit v of the row of d_states[b]
 * is clear; allowed entries keep their bits exactly.
 *   d_logits  device [B, V] contiguous, dtype TRIE_DTYPE_F32 or _BF16
 *   d_states  device int32[B]; FINISHED, DEAD and ids that are not nodes use
 *             the row {EOS}
 *   V         must equal the V of the last trie_compile_masks on the handle
 * Uses the mask recorded by the last trie_compile_masks (TRIE_ESTATE if
 * none), and the summary that compile keeps in the handle of which 1,024-token
 * segments of each row hold an allowed token (segments without one are
 * written without reading the mask). Both belong to the handle's last compile:
 * work captured in a CUDA graph must not outlive a later compile of the handle
 * with another vocabulary. B = 0 is a no-op. */
int trie_apply_mask(trie_t h, void *d_logits, int dtype, const int32_t *d_states, int32_t B,
                    int32_t V, cudaStream_t stream);

/* One decode step in one launch: advance the states by the tokens sampled
 * from the previous logits, then mask the current logits by the new states
 * (trie_advance followed by trie_apply_mask; Sec. 2 Eq. 1, Sec. 4.2, App. H.3).
 *   d_states_in   device int32[B], the states before the move (read only)
 *   d_tokens      device int32[B]
 *   d_states_out  device int32[B], receives the new states; must not be
 *                 d_states_in (TRIE_EINVAL)
 *   d_err         as trie_advance
 *   d_logits      device [B, V], masked in place by the rows of the new states
 * Rules, states, dtype and V as trie_advance / trie_apply_mask; needs a prior
 * trie_compile_masks (TRIE_ESTATE). The transitions recorded by that compile
 * are looked up first; other moves are walked byte by byte. B = 0 is a no-op. */
int trie_advance_apply(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out,
                       int32_t *d_err, void *d_logits, int dtype, int32_t B, int32_t V, cudaStream_t stream);

/* The same mask as trie_compile_masks, computed pair by pair: for every node
 * n and token v the GPU walks v's bytes down from n (the definition of
 * Sec. 4.1: v is allowed iff prefix(n) . bytes(v) is a prefix of some set
 * string, App. G.5), one token per lane, and a warp ballot assembles each
 * 32-bit mask word. It costs N * V walks where trie_compile_masks does a few
 * lookups per node; it is kept as the direct, measured alternative (the
 * design that evaluates every pair) and as a second GPU derivation of the
 * same mask. Arguments, layout, result and errors as trie_compile_masks; it
 * does not record the mask, the vocabulary or transitions in the handle. */
int trie_compile_masks_pairwise(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                                uint32_t *d_mask, cudaStream_t stream);

/* Sparse form of the masks: for every node the ids of its allowed tokens, as
 * the paper stores them (valid[n] as lists of 4-byte token ids, Sec. 4.2;
 * App. H.5), computed on the GPU without the dense bitmask. At K = 10,000 and
 * V = 152,064 the lists hold 56,899 ids (10,000 of them EOS; 228 KB) where the
 * bitmask takes 439 MB.
 *   Arguments as trie_compile_masks; the lists are stored on the device by
 *   the library, with the handle (they replace those of an earlier call).
 *   Layout: offsets int64[num_nodes + 1] and tokens int32[offsets[N]]; the
 *   tokens of node n are tokens[offsets[n] .. offsets[n+1]), EOS (V-1)
 *   included where n is terminal, in no particular order.
 *   Method: the tokens read backwards form a trie (built once per vocabulary
 *   on the host, its edges inserted into a device table); from every node m
 *   the GPU walks it with the labels above m, so that each token ending with
 *   the last k edges into m is found and listed at the node k levels up
 *   (the Aho-Corasick outputs of Sec. 4.2 step 2, found per node). One walk
 *   counts every row's entries, a scan gives the offsets, a second walk
 *   writes the tokens, and beside each the node its token leads to (kept in
 *   the handle, 8 bytes per entry in all, for trie_advance_apply_lists: the
 *   advance is then a look-up in the state's list).
 *   Asynchronous on `stream` while the bound on the entries (a node lists at
 *   most one token string per length up to the longest token, each under
 *   every id that spells it, plus EOS) is at most 2^28 entries or fits the
 *   buffer of an earlier call: the token buffer is sized by it and nothing
 *   is read back; trie_num_valid reads the size when asked. Beyond that the
 *   exact count is read back between the walks (host-synchronous).
 *   Records the vocabulary for trie_advance, like trie_compile_masks (it
 *   neither reads nor fills the transition table).
 *   Errors: TRIE_EINVAL (also for a vocabulary whose reversed-token trie
 *   would exceed 2^24 - 2 nodes), TRIE_ENOMEM, TRIE_ECUDA. */
int trie_compile_lists(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                       cudaStream_t stream);

/* trie_compile_lists with the vocabulary of handle v (see trie_vocab_create);
 * v must belong to the current device (else TRIE_EINVAL). */
int trie_compile_lists_vocab(trie_t h, trie_vocab_t v, cudaStream_t stream);

/* Number of (node, token) entries in the handle's lists; -1 before any
 * trie_compile_lists (or if reading the size back fails). The first call
 * after a trie_compile_lists waits for that build to complete. */
int64_t trie_num_valid(trie_t h);

/* Copy the handle's lists into caller buffers (device; each may be NULL):
 * d_offsets int64[num_nodes + 1], d_tokens int32[trie_num_valid(h)].
 * Asynchronous on `stream`. TRIE_ESTATE before any trie_compile_lists. */
int trie_copy_lists(trie_t h, int64_t *d_offsets, int32_t *d_tokens, cudaStream_t stream);

/* trie_apply_mask driven by the handle's valid lists instead of a bitmask
 * (the decode-time lookup A(s_t) = valid[s_t] of Sec. 4.2, then the -inf
 * write of App. H.3). Arguments, states and result as trie_apply_mask; V
 * must equal the V of the last trie_compile_lists (TRIE_ESTATE if none). */
int trie_apply_lists(trie_t h, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                     cudaStream_t stream);

/* Lazy rows (App. H.5, the memory-constrained mode: valid[n] is computed
 * only when decoding first reaches node n, and kept in an LRU cache of
 * bounded size). No mask of all nodes is built: each call computes the rows
 * of the batch's states that are not cached, on the GPU, and applies them.
 * A row is computed from the node's subtree: the strings of the paths from
 * n down into it that are tokens (App. G.5 condition (i)), plus EOS where n
 * is terminal; the result equals that row of trie_compile_masks.
 *
 * Set-up (host-synchronous; synchronises the device). Allocates, on the
 * current device, (rounded-up cache_rows + max_batch) rows of ceil(V/32)
 * uint32 words plus 16 bytes per trie node and 16 per batch row; replaces the
 * cache of an earlier trie_lazy_init on the handle (starting empty).
 *   vocab_bytes, vocab_offsets, V  as trie_compile_masks, 2 <= V <= 524,288
 *   cache_rows  rows kept between calls, 0 <= cache_rows <= 2^30 (rounded up
 *               to a multiple of 8; 0 = no cache, every row is recomputed;
 *               TRIE_ENOMEM if the rows do not fit). The cache is 8-way set
 *               associative: a node may only use the 8 rows of its set, and
 *               a new row replaces the least recently used of them.
 *   max_batch   largest B of the calls below, 1 <= max_batch <= 4096
 * Errors: TRIE_EINVAL, TRIE_ENOMEM, TRIE_ECUDA. */
int trie_lazy_init(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                   int32_t cache_rows, int32_t max_batch);

/* trie_apply_mask with lazily computed rows (same arguments, states and
 * result; V must equal trie_lazy_init's V; B <= max_batch). Rows of states
 * that are cached are reused; the others are computed and cached, unless all
 * 8 rows of their set are used by this same call (they are then computed for
 * this call only). Three kernels on `stream`; no host synchronisation, no
 * allocation. All lazy calls on one handle share its cache and scratch: they
 * must run one after the other (one stream, or ordered by events), not
 * concurrently. TRIE_ESTATE before trie_lazy_init. */
int trie_lazy_apply(trie_t h, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                    cudaStream_t stream);

/* trie_advance_apply with lazily computed rows: the states are advanced
 * (rules of trie_advance, written to d_states_out, which must differ from
 * d_states_in), then the logits are masked by the rows of the new states as
 * trie_lazy_apply does. d_err as trie_advance. */
int trie_lazy_advance_apply(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out,
                            int32_t *d_err, void *d_logits, int dtype, int32_t B, int32_t V, cudaStream_t stream);

/* The rows themselves (for inspection and tests): d_rows device
 * uint32[B][ceil(V/32)] receives the row of each d_states[b] (FINISHED, DEAD
 * and non-node states: the {EOS} row), computed and cached as by
 * trie_lazy_apply. */
int trie_lazy_rows(trie_t h, const int32_t *d_states, int32_t B, uint32_t *d_rows, cudaStream_t stream);

/* Cache counters since trie_lazy_init: batch rows whose node's row was found
 * in the cache (hits) and batch rows whose node's row had to be computed
 * (misses; batch rows sharing a node in one call all count, the row is
 * computed once). Host-synchronous (synchronises the device). */
int trie_lazy_stats(trie_t h, int64_t *hits, int64_t *misses);

/* trie_advance_apply driven by the handle's valid lists: advance the states
 * by the tokens (rules of trie_advance; d_states_out must differ from
 * d_states_in), then mask the logits by the lists of the new states
 * (trie_apply_lists), in one launch. V must equal the V of the last
 * trie_compile_lists, whose vocabulary the advance uses (TRIE_ESTATE if there
 * was none, or if a later trie_compile_masks took another vocabulary). */
int trie_advance_apply_lists(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out,
                             int32_t *d_err, void *d_logits, int dtype, int32_t B, int32_t V, cudaStream_t stream);

/* Size of the fixed device scratch used by trie_compile_masks_noalloc. */
#define TRIE_NOALLOC_SCRATCH_BYTES (32u << 20)

/* The paper has no counterpart to this entry point; it serves callers that
 * must not have the library allocate device memory.
 *
 * trie_compile_masks keeps device copies of the trie and the packed
 * vocabulary in memory it gets from cudaMalloc. Some callers cannot allow
 * that: a serving engine that has given all free HBM to its own pool (KV
 * cache) and forbids other allocations, a process held to a fixed device
 * memory budget, or a latency-critical loop in which cudaMalloc / cudaFree,
 * which may synchronise the device, must not run. This call computes the
 * same mask as trie_compile_masks without allocating: the trie and the
 * vocabulary are staged in a static host buffer and copied into one
 * fixed-size device array compiled into the library
 * (TRIE_NOALLOC_SCRATCH_BYTES = 32 MiB). Every GPU that loads that array
 * holds it until the process exits (under CUDA's default lazy module loading,
 * from the first call on the device).
 *   Arguments, layout and result are those of trie_compile_masks.
 *   The trie's node arrays (6 bytes per node) plus the packed vocabulary
 *   (6 bytes per token, its bytes rounded up to 16 per token, and a hash
 *   table of 12 bytes per slot, 4 slots per token with bytes) must fit in the
 *   scratch; otherwise TRIE_EINVAL with a message, and nothing is launched.
 *   The first call on a device looks up the device address of the scratch
 *   (cudaGetSymbolAddress) and creates one event, with that device current;
 *   make that first call before any stream capture. Both are kept until the
 *   process exits: after cudaDeviceReset of a device, do not call this entry
 *   point on that device again in the same process.
 *   All calls share the one scratch, which keeps the last call's contents
 *   (every byte a call uses is rewritten by it). Calls whose work overlaps on
 *   the GPU (other streams, other threads) race on it; order them, for
 *   example on one stream.
 *   The host staging buffer is shared too: a call first waits on the host
 *   until the previous call's copy out of it has completed on the GPU (which
 *   includes the work queued before that copy on its stream), so calls queued
 *   back to back on one stream without a synchronisation are safe.
 *   Unlike trie_compile_masks it does not record the mask or the vocabulary
 *   in the handle: trie_advance and trie_apply_mask keep using those of the
 *   last trie_compile_masks.
 *   On success nothing is allocated, on the host or on the device. */
int trie_compile_masks_noalloc(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets,
                               int32_t V, uint32_t *d_mask, cudaStream_t stream);

/* ---- Fixed formats: character-position masks (App. K) ----
 * A format of length L (0 <= L <= 1024) is a sequence of byte classes
 * C_0..C_{L-1}, e.g. YYYY-MM-DD: ten positions, digits but for '-' at 4 and
 * 7. Its strings are the products of its classes; the automaton's states are
 * the positions 0..L (p bytes written). valid[p] holds token v (not EOS) iff
 * 1 <= len(v) <= L - p and byte i of v lies in C_{p+i} for every i (the
 * position-wise check of App. K), and EOS iff p = L. Masks have the trie
 * masks' layout with L + 1 rows; states, FINISHED / DEAD and errors follow
 * the trie calls, with positions in place of node ids. */
typedef struct fmt_s *fmt_t; /* opaque; owned by the library */

/* Build a format from L class bitmaps (host, read during the call):
 *   classes  uint8[L * 32]; byte c is in class i iff bit (c % 8) of
 *            classes[32 * i + c / 8] is set (may be NULL when L = 0)
 * Host only. TRIE_EINVAL for L outside [0, 1024] or NULL pointers. */
int fmt_build(const uint8_t *classes, int32_t L, fmt_t *out);

/* L of the format; -1 for a NULL handle. */
int32_t fmt_length(fmt_t f);

/* valid[p] for every position into the caller's mask d_mask (device,
 * (L + 1) * ceil(V/32) uint32, 4-byte aligned). Vocabulary arguments,
 * caching and errors as trie_compile_masks; the first call uploads the
 * format's classes to the current device. The handle records (d_mask, V,
 * vocabulary) for fmt_advance and fmt_apply_mask. */
int fmt_compile_masks(fmt_t f, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                      uint32_t *d_mask, cudaStream_t stream);

/* Positions in place: p -> p + len(v) for an allowed token; EOS at p = L ->
 * FINISHED; other rules and d_err as trie_advance. Needs a prior
 * fmt_compile_masks (TRIE_ESTATE). */
int fmt_advance(fmt_t f, int32_t *d_states, const int32_t *d_tokens, int32_t B, int32_t *d_err,
                cudaStream_t stream);

/* trie_apply_mask for a format: -inf where bit v of the row of position
 * d_states[b] is clear (positions outside [0, L], FINISHED and DEAD use
 * {EOS}); V must equal the compiled mask's V. */
int fmt_apply_mask(fmt_t f, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                   cudaStream_t stream);

/* Release the format and its device copy. NULL is a no-op. */
int fmt_destroy(fmt_t f);

/* Release the handle, its host arrays and its device copy of the trie.
 * Synchronises the device first if device memory is held. NULL is a no-op. */
int trie_destroy(trie_t h);

/* Release the handle without synchronising: its device memory is freed in
 * stream order on `stream` (it returns to the library's pool once the work
 * queued on `stream` so far has completed); its host arrays, which a queued
 * upload may still be reading, once an event recorded on `stream` now has
 * completed: a later trie_destroy_async or trie_build* call frees them (a
 * handle that never reached a device: at once). Every
 * use of the handle on the device must be on `stream` or ordered before the
 * work queued on it now (for example by an event); the handle must not be
 * used by the host after the call. A server that builds a trie per request
 * batch can then drop the batch's handle right after queueing its last
 * kernel and go on building the next one. NULL is a no-op. */
int trie_destroy_async(trie_t h, cudaStream_t stream);

/* Message of the last error on the calling thread ("" if none). */
const char *trie_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* TRIEMASK_H */
