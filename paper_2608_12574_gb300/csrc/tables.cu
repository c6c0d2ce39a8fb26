// Per-node tables of a trie on the device, from its parent and label arrays:
// the child links (first child and the 256-bit set of child labels) that the
// character walk of the advance follows (Sec. 2, Eq. 1; Sec. 4.1), and the
// tables that the mask compile's traversal and the list walk read in place of
// the paper's depth-first walk with saved automaton states (App. H.4, Phase
// 4): the last 16 edge labels, min(depth, 16), the 16 nearest ancestors. They
// run once per trie, after its upload or its build on the device, and read
// only parent and label: nodes in breadth-first order within every set,
// siblings by ascending byte, the sets one after another, each root first.
#include <stdint.h>

#include <cuda_runtime.h>

#include "tm_internal.h"

namespace tmk {

namespace {

constexpr int kLinkThreads = 256;
constexpr int kTableThreads = 256;
constexpr int kTableClimb = 16;  // labels in a window, ancestors in a row

inline int grid_size(int64_t work, int64_t per_block, int64_t cap) {
    int64_t g = (work + per_block - 1) / per_block;
    if (g < 1) g = 1;
    if (g > cap) g = cap;
    return int(g);
}

// The key of node c: its parent, or c - 1 for a root. Children of a node are
// contiguous and come in the order of their parents, and a set's root
// follows the last node of the set before it (a leaf, which no node has for
// parent), so the keys never decrease along the ids.
__device__ __forceinline__ int32_t link_key(int32_t p, int32_t c) { return p >= 0 ? p : c - 1; }

// Child links, one warp per 32 consecutive nodes c (a chunk) taken as
// children. The warp owns the parent rows x with key(c0 - 1) < x <= key(c0 +
// 31) (the last chunk up to n - 1): each row has its first child in the
// chunk, or no child, so the chunks' row ranges tile 0 .. n - 1 and every row
// is written whole by one warp, in batches of 32 rows built in shared memory
// (label bits by shared atomics, the first child by a shared minimum) and
// stored as one contiguous run, with no clear of the arrays and no global
// atomics. The children of the last owned row may run past the chunk; the
// warp reads on, 32 nodes at a time, while they last. (Before: clears of the
// two arrays, 171 MB, and one global atomicOr per node.)
__global__ void __launch_bounds__(kLinkThreads) k_trie_links(const int32_t *__restrict__ parent,
                                                             const uint8_t *__restrict__ label, int32_t n,
                                                             int32_t *__restrict__ first_child,
                                                             uint32_t *__restrict__ child_bits) {
    __shared__ uint4 s_bits[kLinkThreads / 32][64];  // per warp: 32 rows of 8 words
    __shared__ int32_t s_first[kLinkThreads / 32][32];
    const int lane = threadIdx.x & 31;
    uint4 *wb4 = s_bits[threadIdx.x >> 5];
    uint32_t *wb = reinterpret_cast<uint32_t *>(wb4);
    int32_t *wf = s_first[threadIdx.x >> 5];
    const int64_t n_chunks = (int64_t(n) + 31) / 32;
    const int64_t warps = (int64_t(gridDim.x) * blockDim.x) >> 5;
    for (int64_t ch = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; ch < n_chunks; ch += warps) {
        const int32_t c0 = int32_t(ch * 32);
        const int32_t c = c0 + lane;
        const int32_t p = c < n ? __ldg(parent + c) : -1;
        const uint32_t lab = c < n ? __ldg(label + c) : 0u;
        const int32_t last = min(c0 + 31, n - 1);
        const int32_t klast = __shfl_sync(0xffffffffu, link_key(p, c), last - c0);
        const int32_t xa = c0 == 0 ? 0 : link_key(__ldg(parent + c0 - 1), c0 - 1) + 1;
        const int32_t xb = last == n - 1 ? n - 1 : klast;
        // the last child of the chunk is a child of xb: its siblings may follow
        const bool runs_on = last < n - 1 && __shfl_sync(0xffffffffu, p, 31) == xb;
        for (int32_t base = xa; base <= xb; base += 32) {
            wb4[lane] = make_uint4(0u, 0u, 0u, 0u);
            wb4[lane + 32] = make_uint4(0u, 0u, 0u, 0u);
            wf[lane] = INT32_MAX;
            __syncwarp();
            if (c < n && p >= base && p <= xb && p - base < 32) {
                atomicOr(wb + (p - base) * 8 + (lab >> 5), 1u << (lab & 31u));
                atomicMin(wf + (p - base), c);
            }
            if (runs_on && xb - base < 32) {
                for (int32_t e0 = c0 + 32; e0 < n; e0 += 32) {
                    const int32_t ce = e0 + lane;
                    const bool mine = ce < n && __ldg(parent + ce) == xb;
                    if (mine) {
                        const uint32_t le = __ldg(label + ce);
                        atomicOr(wb + (xb - base) * 8 + (le >> 5), 1u << (le & 31u));
                    }
                    if (!__all_sync(0xffffffffu, mine)) break;
                }
            }
            __syncwarp();
            const int32_t rows = min(32, xb - base + 1);
            uint4 *dst = reinterpret_cast<uint4 *>(child_bits + int64_t(base) * 8);
            if (lane < 2 * rows) dst[lane] = wb4[lane];
            if (lane + 32 < 2 * rows) dst[lane + 32] = wb4[lane + 32];
            if (lane < rows) first_child[base + lane] = wf[lane] == INT32_MAX ? -1 : wf[lane];
            __syncwarp();  // the batch is stored before the next one is built
        }
    }
}

// Per-node tables of the probe and of the list walk (one thread per node,
// climbing at most 16 parents): the last 16 edge labels into m (byte i = the
// label i levels up, 0 past the root), min(depth, 16), and the 16 nearest
// ancestors (-1 past the root), stored as four 16-byte rows. Siblings and
// cousins are neighbours in breadth-first order, so a warp's climbs read
// neighbouring entries of the parent and label arrays, which stay in L2.
// Each warp stages its 32 ancestor rows (2 KB) in shared memory, a quarter
// row as soon as its four ancestors are known, and writes them out as one
// contiguous 2 KB run: stored straight from the climb, each 16-byte store of
// a warp touched 32 rows 64 bytes apart (117 us on the 4.77 M-node forest
// against 89 us staged). The 16-byte units of a row are swizzled by bits 1-2
// of the row, so that the eight rows of a quarter-warp's stores and the two
// rows of its loads fall on distinct banks. (Measured slower: two or four
// climbs per thread, 97-217 us, and the labels gathered after the climb,
// 105-240 us, both short of registers at full occupancy; rows built by
// doubling from the rows of the ancestors 4, 8 and 12 levels up, 230 us,
// whose reads of the 64-byte ancestor rows come from DRAM.)
__global__ void __launch_bounds__(kTableThreads, 2048 / kTableThreads)
    k_trie_tables(const int32_t *__restrict__ parent, const uint8_t *__restrict__ label, int32_t n,
                  ulonglong2 *__restrict__ window, uint8_t *__restrict__ depth16, int4 *__restrict__ anc) {
    __shared__ int4 stage[kTableThreads * 4];
    const int lane = threadIdx.x & 31;
    int4 *ws = stage + (threadIdx.x >> 5) * 128;  // this warp's 32 rows of four units
    const int32_t stride = gridDim.x * blockDim.x;
    for (int32_t m0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31); m0 < n; m0 += stride) {
        const int32_t m = m0 + lane;
        uint64_t lo = 0, hi = 0;
        int32_t up[4];
        int32_t d = 0;
        int32_t x = m < n ? m : -1;
#pragma unroll
        for (int k = 0; k < kTableClimb; k++) {
            const int32_t p = x >= 0 ? __ldg(parent + x) : -1;
            up[k & 3] = p;
            if (p >= 0) {
                const uint64_t b = __ldg(label + x);
                if (k < 8) lo |= b << (8 * k);
                else hi |= b << (8 * (k - 8));
                d = k + 1;
            }
            x = p;
            if ((k & 3) == 3)
                ws[lane * 4 + ((k >> 2) ^ ((lane >> 1) & 3))] = make_int4(up[0], up[1], up[2], up[3]);
        }
        if (m < n) {
            window[m] = make_ulonglong2(lo, hi);
            depth16[m] = uint8_t(d);
        }
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int u = j * 32 + lane, r = u >> 2, q = u & 3;  // unit u of the warp's 2 KB run
            if (m0 + r < n) anc[int64_t(m0) * 4 + u] = ws[r * 4 + (q ^ ((r >> 1) & 3))];
        }
        __syncwarp();  // the rows are read before the next nodes' climbs overwrite them
    }
}

}  // namespace

cudaError_t launch_trie_links(const DevTrie &t, int32_t n_nodes, int num_sms, cudaStream_t st) {
    if (n_nodes <= 0) return cudaSuccess;
    const int grid = grid_size((int64_t(n_nodes) + 31) / 32, kLinkThreads / 32, int64_t(num_sms) * 8);
    k_trie_links<<<grid, kLinkThreads, 0, st>>>(t.parent, t.label, n_nodes, t.first_child, t.child_bits);
    return cudaGetLastError();
}

cudaError_t launch_trie_tables(const DevTrie &t, int32_t n_nodes, int num_sms, cudaStream_t st) {
    if (n_nodes <= 0) return cudaSuccess;
    const int grid = grid_size(n_nodes, kTableThreads, int64_t(num_sms) * 8);
    k_trie_tables<<<grid, kTableThreads, 0, st>>>(t.parent, t.label, n_nodes, t.window, t.depth16, t.anc);
    return cudaGetLastError();
}

}  // namespace tmk
