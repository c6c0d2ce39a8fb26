// Internal structures of libtriemask shared by the host builder, the kernels
// and the C ABI. Not part of the public interface.
#pragma once

#include <stdint.h>

#include <atomic>
#include <memory>
#include <new>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include <cuda_runtime_api.h>

namespace tmk {

#if defined(__CUDACC__)
// Programmatic dependent launch (PDL). Every kernel of the library is launched
// with programmatic stream serialization: it may let the next kernel of its
// stream launch early (pdl_launch_dependents) and waits for the previous one
// (pdl_wait, the hardware grid dependency: the previous grid never waits on
// this one, so the wait always resolves) before it touches memory that kernel
// may write or read.
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... Params, typename... Args>
cudaError_t launch_pdl_smem(void (*kernel)(Params...), int64_t grid, int block, size_t smem, cudaStream_t st,
                            Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(grid < 1 ? 1 : grid));
    cfg.blockDim = dim3(unsigned(block));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Params>(args)...);
}

template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), int64_t grid, int block, cudaStream_t st, Args... args) {
    return launch_pdl_smem(kernel, grid, block, 0, st, args...);
}
#endif

// Blocks of at least 2 MB for the builder's arrays come from a process-wide
// cache of freed blocks (whole 2 MB classes, at most 1 GB held): a server that
// builds a new forest for every batch then reuses pages it has already
// touched instead of faulting in fresh ones. Defined in host_trie.cpp.
void *big_block_alloc(size_t bytes);
void big_block_free(void *p, size_t bytes);
constexpr size_t kBigBlock = size_t(2) << 20;

// std::vector allocator whose resize() leaves trivial elements uninitialised
// (large host arrays are then first touched by the threads that fill them),
// with large blocks from the cache above.
template <class T>
struct DefaultInitAlloc : std::allocator<T> {
    template <class U>
    struct rebind {
        using other = DefaultInitAlloc<U>;
    };
    DefaultInitAlloc() noexcept = default;
    template <class U>
    DefaultInitAlloc(const DefaultInitAlloc<U> &) noexcept {}
    T *allocate(size_t n) {
        const size_t bytes = n * sizeof(T);
        if (bytes < kBigBlock) return std::allocator<T>::allocate(n);
        void *p = big_block_alloc(bytes);
        if (!p) throw std::bad_alloc();
        return static_cast<T *>(p);
    }
    void deallocate(T *p, size_t n) noexcept {
        const size_t bytes = n * sizeof(T);
        if (bytes < kBigBlock) std::allocator<T>::deallocate(p, n);
        else big_block_free(p, bytes);
    }
    template <class U>
    void construct(U *p) noexcept {
        ::new (static_cast<void *>(p)) U;
    }
    template <class U, class... Args>
    void construct(U *p, Args &&...args) {
        ::new (static_cast<void *>(p)) U(std::forward<Args>(args)...);
    }
};
template <class T>
using hvec = std::vector<T, DefaultInitAlloc<T>>;

// ----------------------------------------------------------------- host trie
// Byte trie in breadth-first order, siblings by ascending byte (Sec. 4.1).
// Children of a node are contiguous, so the device derives each node's first
// child and the 256-bit set of its child labels from parent and label
// (launch_trie_links); the child for byte c is then first_child +
// popcount(bits below c).
struct HostTrie {
    int32_t n = 0;                       // nodes (all sets of a forest)
    hvec<int32_t> parent;                // -1 for a root
    hvec<uint8_t> label;                 // byte on the incoming edge
    hvec<uint8_t> terminal;              // some string ends here
    // Depth-first pre-order of the same nodes (the order in which the builder
    // creates them): position i holds node pre_node[i], at depth pre_depth[i],
    // whose subtree is positions i .. i + pre_size[i] - 1. Used by the lazy
    // rows, which enumerate a node's subtree as one interval.
    hvec<int32_t> pre_node;              // [n]
    hvec<int32_t> pre_depth;             // [n]
    hvec<int32_t> pre_size;              // [n]
    std::vector<int32_t> roots;          // root id of each set
    int64_t n_chars = 0;                 // total bytes of the distinct strings
    int32_t max_depth = 0;
};

// Return "" on success, else an error message. build_trie takes strings
// first..last-1; build_forest builds set i from strings
// set_offsets[i]..set_offsets[i+1]-1 on host threads and concatenates them.
std::string build_trie(const uint8_t *bytes, const int64_t *offsets, int32_t first, int32_t last,
                       HostTrie *out);
std::string build_forest(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets,
                         int32_t M, HostTrie *out);

// -------------------------------------------------------------- vocabulary
// Token strings packed for 16-byte vector loads plus an open-addressing hash
// table from (length, bytes) to token id, used to find the tokens that end
// at a trie node.
struct HostVocab {
    int32_t V = 0;
    int32_t max_len = 0;                 // longest token with bytes (EOS excluded)
    std::vector<uint32_t> tok_off;       // [V] start of token bytes in blob (16-byte aligned)
    std::vector<uint16_t> tok_len;       // [V] byte length; EOS and byte-less tokens: 0
    std::vector<uint8_t> blob;           // token bytes, each token 16-byte aligned
    std::vector<uint64_t> ht_key;        // [S] 0 = empty slot
    std::vector<int32_t> ht_val;         // [S] token id
    uint32_t ht_mask = 0;                // S - 1 (S a power of two)
    int32_t dup_keys = 0;                // two tokens share a hash key
};

std::string pack_vocab(const uint8_t *bytes, const int64_t *offsets, int32_t V, HostVocab *out);

// The tokens read backwards, as a trie (root 0): the path from the root
// spelling b_{L-1} .. b_0 ends at the node of token b_0 .. b_{L-1}. Walking it
// with the labels above a node m of a set trie (the label into m first) meets,
// after k steps, exactly the tokens that spell the last k edges into m: the
// Aho-Corasick outputs at m of Sec. 4.2 step 2, without failure links. Node
// ids in pre-order; token[x] = the smallest id whose bytes end at x, or -1;
// next[v] = the next larger id with the same bytes as v, or -1 (empty when
// all token strings differ). Built once per vocabulary, on the host.
constexpr int64_t kRevTrieMaxNodes = (int64_t(1) << 24) - 2;  // edge keys (parent << 8 | byte) + 1 fit 32 bits
struct RevTokenTrie {
    int32_t n = 0;
    hvec<int32_t> parent;
    hvec<uint8_t> label;
    hvec<int32_t> token;
    std::vector<int32_t> next;
    int32_t max_mult = 1;  // most ids sharing one byte string
};
std::string build_reversed_token_trie(const uint8_t *bytes, const int64_t *offsets, int32_t V,
                                      RevTokenTrie *out);

// The two halves of pack_vocab, writing into caller-supplied arrays (the
// no-alloc compile stages into a static buffer). pack_token_bytes: token v's
// bytes at tok_off[v] (16-byte aligned, blob zeroed by the caller), its length
// in tok_len[v]; EOS (V-1) gets length 0. fill_token_table: the (length,
// bytes) -> id table of S slots (token_table_slots), returns whether two
// tokens share a key. Offsets must already be validated.
void pack_token_bytes(const uint8_t *bytes, const int64_t *offsets, int32_t V, uint32_t *tok_off,
                      uint16_t *tok_len, uint8_t *blob);
bool fill_token_table(const uint8_t *bytes, const int64_t *offsets, const uint16_t *tok_len, int32_t V,
                      uint64_t S, uint64_t *key, int32_t *val);
uint64_t token_table_slots(int64_t n_tokens_with_bytes);

// Polynomial string hash used by the table: Horner over (byte + 1) with base
// kHashBase, modulo 2^64, then mixed with the length. The kernel extends it
// one byte to the left per trie edge it climbs.
constexpr uint64_t kHashBase = 0x100000001B3ull;
#if defined(__CUDACC__)
__host__ __device__
#endif
inline uint64_t hash_finish(uint64_t h, uint32_t len) {
    uint64_t z = h ^ (uint64_t(len) * 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 33)) * 0xFF51AFD7ED558CCDull;
    z = (z ^ (z >> 33)) * 0xC4CEB9FE1A85EC53ull;
    z ^= z >> 33;
    return z | 1ull;  // 0 marks an empty slot
}

// ------------------------------------------------------------ device copies
struct DevVocab {
    int device = -1;
    int32_t V = 0;
    int32_t max_len = 0;
    uint32_t ht_mask = 0;
    void *base = nullptr;                // one allocation holding all arrays
    const uint32_t *tok_off = nullptr;
    const uint16_t *tok_len = nullptr;
    const uint8_t *blob = nullptr;
    uint64_t blob_bytes = 0;
    int32_t dup_keys = 0;
    const uint64_t *ht_key = nullptr;
    const int32_t *ht_val = nullptr;
    // per slot: token, min(len, 31) << 27 | blob offset / 16, first 8 bytes
    // (null when the blob exceeds 2 GiB or two tokens share a key)
    const uint4 *ht_pay = nullptr;
    // The reversed-token trie (RevTokenTrie) as an open-addressing edge table
    // for the list compile's walk, built on first use: slot {(parent << 8 |
    // byte) + 1, child, token ending at child or -1, 0}, key 0 = empty.
    std::mutex rt_mu;
    int32_t rt_state = 0;                // 0 not built, 1 built, -1 too large (walk unavailable)
    void *rt_base = nullptr;
    const uint4 *rt_edge = nullptr;
    uint32_t rt_mask = 0;                // slots - 1
    const int32_t *tok_next = nullptr;   // [V] next id with the same bytes, or null (all strings differ)
    int32_t rt_mult = 1;                 // most ids sharing one byte string
    // host copy of the caller's arrays, to recognise the same vocabulary later
    std::vector<uint8_t> src_bytes;
    std::vector<int64_t> src_offsets;
    ~DevVocab();
};

// (row, token) pairs the compile's probe records per node for the scatter; a
// node has at most one per suffix length up to the longest token plus EOS,
// so with tokens of up to 15 bytes no node has more (a node with more is
// searched again by the scatter).
constexpr int kHitSlots = 16;

// The segment summary an apply reads: words per row, the epoch word; words
// null when the compile computed no summary.
struct SegRef {
    const unsigned long long *words = nullptr;
    const uint32_t *epoch = nullptr;
    int32_t per_row = 0;
};

struct DevTrie {
    int device = -1;
    void *base = nullptr;
    const int32_t *parent = nullptr;
    const uint8_t *label = nullptr;
    const uint8_t *terminal = nullptr;
    int32_t *first_child = nullptr;      // built on the device (launch_trie_links)
    uint32_t *child_bits = nullptr;      // [n * 8], built on the device
    // Per node, for the mask compile, built on the device from parent/label
    // (launch_trie_tables): the labels of the last 16 edges into it (byte i =
    // label i levels up, 0 past the root), min(depth, 16), and the ancestors
    // 1..16 levels up (entry k = k + 1 levels up, -1 past the root).
    ulonglong2 *window = nullptr;    // [n]
    uint8_t *depth16 = nullptr;      // [n]
    int4 *anc = nullptr;             // [n * 4]
    ulonglong2 *trans = nullptr;     // transition table {(row << 32 | token) + 1, end node}
    uint32_t trans_mask = 0;         // slots - 1
    // Segment summary of the dense mask (own allocation): per row, words of 32
    // segment bits (1,024 tokens each) tagged in their high half with the
    // epoch of the compile that set them; a word with another tag than the
    // device's current epoch (*seg_epoch, written by each compile's probe)
    // holds no allowed token.
    unsigned long long *seg_any = nullptr;  // seg_cap words
    uint32_t *seg_epoch = nullptr;          // [1] (device), the epoch of the last compile that ran
    uint32_t seg_epoch_next = 1;            // host: the epoch of the next compile (0 is never used)
    int64_t seg_cap = 0;
    void *hits_base = nullptr;       // the two arrays below (allocated by the first dense compile)
    int2 *hits = nullptr;            // compile scratch: kHitSlots (row, token) pairs per node
    uint8_t *hit_count = nullptr;    // compile scratch: hits found per node
};

// Device storage of the sparse valid lists of a handle (library-owned).
struct DevLists {
    void *base = nullptr;           // count, off, tile_sum, total (and a first token buffer)
    size_t base_bytes = 0;
    int32_t *count = nullptr;       // [n] entries per row (the counting walk)
    int64_t *off = nullptr;         // [n + 1]
    int64_t *tile_sum = nullptr;    // [tiles]
    int64_t *total = nullptr;       // [1]
    int32_t *toks = nullptr;        // [tok_cap]: in the block at base, or a separate allocation
    int32_t *ends = nullptr;        // [tok_cap] after toks: the node each entry's token leads to
    int64_t tok_cap = 0;
    bool toks_separate = false;     // toks (with ends) is an allocation of its own
    int64_t n_valid = -1;           // entries of the last build, -1 before any (read back on demand)
    bool n_valid_on_device = false; // n_valid is still only in *total
    cudaEvent_t done = nullptr;     // recorded after the last build's kernels
    int32_t V = 0;
};

// Lazy rows (App. H.5): valid[n] computed when a decode state first reaches
// n, kept in a set-associative cache of rows with least-recently-used
// replacement inside each set.
constexpr int kLazyWays = 8;       // rows per cache set
constexpr int kLazyMaxBatch = 4096;
constexpr int32_t kLazyMaxCacheRows = int32_t(1) << 30;  // cache rows + call rows stay int32
constexpr int64_t kLazyMaxWords = 16384;  // row built in shared memory (64 KB): V <= 524,288
// A missing row whose subtree has more than kLazyPartNodes nodes is computed
// in parts by several CTAs (at most kLazyMaxParts per row), for at most
// kLazySplitRows rows per call (splitting only pays while few rows are
// missing; with many the grid is full anyway).
constexpr int32_t kLazyPartNodes = 1024;
constexpr int32_t kLazyMaxParts = 64;
constexpr int32_t kLazySplitRows = 16;

struct LazyCtrl {
    uint32_t now;                   // call counter (stamps of rows used by this call)
    int32_t n_miss;                 // rows computed by the current call
    int32_t n_tasks;                // CTA tasks of the current call (parts of rows)
    int32_t pad;
    unsigned long long hits;        // batch rows whose node row was cached
    unsigned long long misses;      // batch rows whose node row was computed
};

// One node of the depth-first pre-order, as the lazy-row kernel reads it (a
// subtree is a contiguous run of these, 32 bytes each).
struct LazyNode {
    uint64_t phash;      // Horner hash of the path from the root (unfinished)
    int32_t depth;
    int32_t node;        // breadth-first id
    ulonglong2 window;   // labels of the last 16 edges into the node
};

struct DevLazy {
    int device = -1;
    void *base = nullptr;
    int32_t C = 0;                  // cache rows (a multiple of kLazyWays)
    int32_t max_batch = 0;
    int32_t V = 0;
    int64_t W = 0;
    std::shared_ptr<DevVocab> vocab;
    uint32_t *rows = nullptr;       // [(C + max_batch) * W]: cache rows, then per-call rows
    int32_t *tag = nullptr;         // [C] node of the row, -1 empty
    uint32_t *stamp = nullptr;      // [C] call that last used the row (0 never)
    LazyCtrl *ctrl = nullptr;
    int32_t *slot_of = nullptr;     // [max_batch] row of each batch row, < 0: {EOS}
    int32_t *miss_node = nullptr;   // [max_batch] nodes whose rows the call computes
    int32_t *miss_slot = nullptr;   // [max_batch] where
    int32_t *row_u = nullptr;       // [max_batch] scratch
    int4 *task = nullptr;           // [max_batch + kLazySplitRows * kLazyMaxParts] {miss, part, parts, -}
    int32_t *pre_node = nullptr;    // [n] pre-order tables of the trie (HostTrie)
    int32_t *pre_depth = nullptr;   // [n]
    int32_t *pre_size = nullptr;    // [n]
    int32_t *pos_of = nullptr;      // [n] pre-order position of each node
    LazyNode *pre = nullptr;        // [n] by pre-order position
};

// A forest built on the device (device_build.cu): stage() copies the strings
// into its own scratch (reading the caller's host memory directly when
// `direct`), checks their offsets and returns the longest string's length
// (host-synchronous); levels() runs the level loop and the renumbering and
// returns the node count, the roots and the characters (host-synchronous);
// emit() writes parent, label and terminal of the final layout into the
// caller's device arrays (asynchronous); the destructor frees the scratch on
// the stream after them.
constexpr int32_t kDeviceBuildMaxDepth = 1024;        // longer strings: the host builder
constexpr int64_t kDeviceBuildMaxGroups = int64_t(1) << 24;  // sets x (depths + 1) above: the host builder
class DeviceBuild {
public:
    DeviceBuild() = default;
    DeviceBuild(const DeviceBuild &) = delete;
    DeviceBuild &operator=(const DeviceBuild &) = delete;
    ~DeviceBuild();
    cudaError_t stage(const uint8_t *h_bytes, const int64_t *h_off, const int32_t *h_set_off, int32_t M, int32_t K,
                      int64_t n_bytes, bool direct, int num_sms, cudaMemPool_t pool, cudaStream_t st,
                      int32_t *max_len, bool *offsets_ok);
    cudaError_t levels(int32_t D, int num_sms, int32_t *n_nodes, std::vector<int32_t> *roots, int64_t *n_chars);
    cudaError_t emit(int32_t *parent, uint8_t *label, uint8_t *terminal, int num_sms);

private:
    // forests of small sets: one CTA per set (called by levels())
    cudaError_t sets(int num_sms, int32_t *n_nodes, std::vector<int32_t> *roots, int64_t *n_chars);
    struct Scratch;
    Scratch *s_ = nullptr;
    cudaStream_t stream_ = nullptr;
    cudaMemPool_t pool_ = nullptr;
    int32_t M_ = 0, K_ = 0, D_ = 0, n_ = 0;
    int32_t smax_ = 1;    // strings of the largest set
    bool small_ = false;  // one CTA per set
    int64_t n_bytes_ = 0;
};

// The pre-order tables (pre_node / pre_depth / pre_size) of a trie or forest
// from its breadth-first parent array (a depth-first walk per root).
void pre_order_from_parents(HostTrie *t);

// Character-position masks (App. K): formats of at most kFmtMaxLen positions
// (their classes are staged in shared memory, 32 bytes per position).
constexpr int32_t kFmtMaxLen = 1024;

}  // namespace tmk

// The opaque handle of a fixed format (fmt_* calls).
struct fmt_s {
    std::vector<uint32_t> classes;       // [L * 8] class bitmaps as words
    int32_t L = 0;
    std::mutex mu;                       // guards the fields below
    int device = -1;
    uint32_t *d_classes = nullptr;       // device copy (one allocation)
    std::shared_ptr<tmk::DevVocab> vocab; // vocabulary of the last compile
    uint32_t *mask = nullptr;            // last compiled mask (caller-owned)
    int32_t mask_V = 0;
};

// A vocabulary handle of the C ABI: the packed, uploaded vocabulary of one
// device, shared with the library's vocabulary cache.
struct trie_vocab_s {
    std::shared_ptr<tmk::DevVocab> voc;
};

// The opaque handle of the C ABI.
struct trie_s {
    tmk::HostTrie host;
    std::mutex mu;                       // guards dev / vocab / mask fields
    bool host_arrays = true;             // host parent / label / terminal / pre_* present (else on the device only)
    tmk::DevTrie dev;
    std::shared_ptr<tmk::DevVocab> vocab; // vocabulary of the last compile
    uint32_t *mask = nullptr;            // last compiled mask (caller-owned)
    int32_t mask_V = 0;
    tmk::SegRef mask_seg;                // its segment summary (in dev.seg_any), words null when not computed
    tmk::DevLists lists;                 // last compiled valid lists (library-owned)
    std::shared_ptr<tmk::DevVocab> trans_vocab;  // vocabulary the transition table holds
    bool trans_complete = false;         // filled by a whole compile (else partly, by lazy rows)
    tmk::DevLazy lazy;                   // lazy-row cache (trie_lazy_init)
};

namespace tmk {
// Records msg as the calling thread's last error (trie_last_error) and
// returns code.
int set_error(int code, const char *msg);
// Copies the host arrays of a device-built handle back from the device and
// derives its pre-order tables (no-op for handles built on the host).
int ensure_host_arrays(trie_s *h);
// The library's device memory pool of device dev (created on first use;
// nullptr if it cannot be created).
cudaMemPool_t device_pool(int dev);

// Kernel launchers (kernels.cu). Each returns the launch's cudaError_t.
cudaError_t launch_mask_fill(uint32_t *mask, int64_t n_words, int num_sms, cudaStream_t st);
cudaError_t launch_mask_patch(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                              uint32_t *mask, int64_t W, int num_sms, cudaStream_t st);
// Probe, fill and scatter: the mask compile with the per-node searches running
// beside the fill (needs t.hits / t.hit_count).
cudaError_t launch_mask_compile3(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                                 uint32_t *mask, int64_t W, int num_sms, bool fill_trans, cudaStream_t st,
                                 unsigned long long *seg_any, uint32_t *seg_epoch, uint32_t epoch,
                                 int32_t seg_words, bool *seg_written);
// Writes every entry of t.first_child (-1 for a leaf) and t.child_bits from
// t.parent and t.label; nothing needs clearing first (tables.cu).
cudaError_t launch_trie_links(const DevTrie &t, int32_t n_nodes, int num_sms, cudaStream_t st);
// Fills t.window, t.depth16 and t.anc from t.parent and t.label (tables.cu).
cudaError_t launch_trie_tables(const DevTrie &t, int32_t n_nodes, int num_sms, cudaStream_t st);
// Zeroes the transition table (before it is filled for another vocabulary).
cudaError_t launch_trans_clear(const DevTrie &t, int num_sms, cudaStream_t st);
// Fills the per-slot payload of the vocabulary's token table (S uint4).
cudaError_t launch_vocab_pay(const DevVocab &v, uint4 *pay, int num_sms, cudaStream_t st);
cudaError_t launch_advance(const DevTrie &t, int32_t n_nodes, const DevVocab &v, const int32_t *states_in,
                           int32_t *states_out, const int32_t *tokens, int32_t B, int32_t *err, bool use_trans,
                           cudaStream_t st);
// Advance, then mask the next logits by the new states, in one launch.
cudaError_t launch_advance_apply(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans,
                                 const int32_t *states_in, const int32_t *tokens, int32_t *states_out,
                                 int32_t *err, void *logits, int dtype, const uint32_t *mask, int32_t B,
                                 int num_sms, cudaStream_t st, const SegRef &seg);
cudaError_t launch_apply(void *logits, int dtype, const uint32_t *mask, const int32_t *states,
                         int32_t B, int32_t V, int32_t n_nodes, int num_sms, cudaStream_t st,
                         const SegRef &seg = SegRef());
// Copies (d_k, s_k, b_k bytes), k = 0..2, in one launch; the sources are read
// by the kernel itself (device memory, or host memory the device reads
// coherently), so no copy engine and no host synchronisation is involved.
cudaError_t launch_copy3(void *d0, const void *s0, int64_t b0, void *d1, const void *s1, int64_t b1, void *d2,
                         const void *s2, int64_t b2, int num_sms, cudaStream_t st);
// The pairwise form of the dense compile (one walk per (node, token) pair,
// a warp ballot per mask word), kept for comparison with the suffix search.
cudaError_t launch_mask_pairwise(const DevTrie &t, int32_t n_nodes, const DevVocab &v, uint32_t *mask, int num_sms,
                                 cudaStream_t st);
// Edge table of a reversed-token trie (parent, label, token arrays of n
// nodes on the device): zeroes the S = mask + 1 slots and inserts every edge.
cudaError_t launch_rt_build(const int32_t *parent, const uint8_t *label, const int32_t *token, int32_t n,
                            uint4 *edge, uint32_t mask, int num_sms, cudaStream_t st);
// Valid lists by walking the reversed-token trie from every node. Count:
// zero the per-row counts, count every (row, token) entry, scan the counts
// into L.off (shifted one place up: off[i + 1] = the first position of row
// i) and *L.total. Write: walk again, writing every entry at the position
// claimed from off[row + 1] into L.toks (entries past L.tok_cap are
// dropped); afterwards L.off holds the rows' offsets.
cudaError_t launch_lists_count(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                               const DevLists &L, int num_sms, cudaStream_t st);
cudaError_t launch_lists_write(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                               const DevLists &L, int num_sms, cudaStream_t st);
// Lazy rows: pos_of from the pre-order tables and the path hashes (once, at set-up).
cudaError_t launch_lazy_tables(const DevTrie &t, const DevLazy &L, int32_t n_nodes, cudaStream_t st);
// One lazy call: map the batch's states (after the advance when tokens is not
// null) to cache rows, compute the missing rows, then apply them to the
// logits (logits not null) or copy them out (rows_out not null).
cudaError_t launch_lazy(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans, bool fill_trans,
                        int32_t lmax,
                        const DevLazy &L, const int32_t *states_in, const int32_t *tokens, int32_t *states_out,
                        int32_t *err, int32_t B, void *logits, int dtype, uint32_t *rows_out, int num_sms,
                        cudaStream_t st);
// Fixed formats (fmt.cu): the dense [L + 1, ceil(V/32)] mask, and the advance.
cudaError_t launch_fmt_compile(const uint32_t *classes, int32_t L, const DevVocab &v, uint32_t *mask, int num_sms,
                               cudaStream_t st);
cudaError_t launch_fmt_advance(const uint32_t *classes, int32_t L, const DevVocab &v, const int32_t *states_in,
                               int32_t *states_out, const int32_t *tokens, int32_t B, int32_t *err,
                               cudaStream_t st);
// Advance, then apply from the lists by the new states, in one launch.
cudaError_t launch_advance_apply_lists(const DevTrie &t, int32_t n_nodes, const DevVocab &v, bool use_trans,
                                       const int32_t *states_in, const int32_t *tokens, int32_t *states_out,
                                       int32_t *err, void *logits, int dtype, const DevLists &L, int32_t B,
                                       cudaStream_t st);
cudaError_t launch_apply_lists(void *logits, int dtype, const DevLists &L, const int32_t *states, int32_t B,
                               int32_t V, int32_t n_nodes, cudaStream_t st);
}  // namespace tmk
