// The byte tries of a forest built on the device from the raw strings
// (Sec. 4.1; App. G.1 Step 1), for per-request sets that change every batch.
//
// Level by level over depth d, for all sets at once, without sorting the
// strings: every string of length > d ORs its byte d into the 256-bit
// child-label set of the node it has reached (its parent at depth d); the
// parents of a level, in order, give their children consecutive ids (first
// child = the level's end + an exclusive scan of the sets' popcounts), and a
// string moves to child first_child + popcount(labels below its byte). Level d
// is thus ordered by (set, parent, byte): breadth-first with sorted siblings
// within every set, the sets' nodes interleaved by depth. A final pass
// renumbers every node to base(set) + (its rank within the set's own
// breadth-first order), the layout of the host builder.
#include <stdint.h>

#include <algorithm>
#include <vector>

#include <cuda_runtime.h>

#include "tm_internal.h"

namespace tmk {

namespace {

constexpr int kBThreads = 256;
constexpr int32_t kSetMaxStrings = 4096;  // forests whose sets all hold at most this many strings: one CTA per set
constexpr int kScanTile = 1024;  // parents per tile of the level scan

// Staging: copies the strings' offsets, the set offsets and the bytes into
// the scratch, checks the offsets (non-negative, non-decreasing) and finds
// the longest string. The sources are either the caller's host memory, read
// directly where the device accesses pageable memory coherently (Grace's
// NVLink-C2C), or device copies of it (src_off == off: checked in place;
// n_vec = 0: the bytes are in place). src_vec is the bytes' image in whole
// 16-byte blocks (the first and last block may hold bytes outside the
// strings; a 16-byte block never straddles a page).
__global__ void k_b_stage(const int64_t *src_off, int32_t K, const int32_t *src_soff, int32_t M,
                          const uint4 *src_vec, int64_t n_vec, int64_t *off, int32_t *soff, uint4 *vec,
                          int32_t *__restrict__ flags) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t stride = int64_t(gridDim.x) * blockDim.x;
    const int64_t i0 = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    int32_t longest = 0;
    int32_t bad = 0;
    for (int64_t i = i0; i <= K; i += stride) {
        const int64_t o = src_off[i];
        if (off != src_off) off[i] = o;
        if (o < 0) bad = 1;
        if (i < K) {
            const int64_t o2 = src_off[i + 1];
            if (o2 < o) bad = 1;
            else longest = max(longest, int32_t(min(o2 - o, int64_t(INT32_MAX))));
        }
    }
    if (soff != src_soff)
        for (int64_t i = i0; i <= M; i += stride) soff[i] = src_soff[i];
    for (int64_t k = i0; k < n_vec; k += stride) vec[k] = src_vec[k];
    longest = __reduce_max_sync(0xffffffffu, longest);
    bad = __any_sync(0xffffffffu, bad);
    if ((threadIdx.x & 31) == 0) {
        if (bad) atomicOr(flags, 1);
        if (longest) atomicMax(flags + 1, longest);
    }
}

// Strings: their set (from set_offsets), their node (the set's root), and the
// roots of sets with an empty string are terminal. Level 0 = the M roots;
// every non-empty string sets its first byte in its root's child-label set.
__global__ void k_b_init(const uint8_t *__restrict__ bytes, const int64_t *__restrict__ off,
                         const int32_t *__restrict__ set_off, int32_t M, int32_t K, int32_t *__restrict__ str_set,
                         int32_t *__restrict__ cur, int32_t *__restrict__ parent_g, uint8_t *__restrict__ label_g,
                         uint8_t *__restrict__ term_g, int32_t *__restrict__ set_g, int32_t *__restrict__ depth_g,
                         int32_t *__restrict__ ls, uint32_t *__restrict__ bits0) {
    pdl_launch_dependents();
    pdl_wait();
    const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < M) {
        parent_g[i] = -1;
        label_g[i] = 0;
        set_g[i] = i;
        depth_g[i] = 0;
    }
    if (i == 0) {
        ls[0] = 0;
        ls[1] = M;
    }
    if (i >= K) return;
    int32_t lo = 0, hi = M;  // the set s with set_off[s] <= i < set_off[s + 1]
    while (hi - lo > 1) {
        const int32_t mid = (lo + hi) >> 1;
        if (set_off[mid] <= i) lo = mid;
        else hi = mid;
    }
    str_set[i] = lo;
    cur[i] = lo;
    if (off[i + 1] == off[i]) {
        term_g[lo] = 1;  // the empty string: the root is terminal
    } else {
        const uint32_t b = bytes[off[i] - off[0]];
        atomicOr(bits0 + int64_t(lo) * 8 + (b >> 5), 1u << (b & 31u));
    }
}

__device__ __forceinline__ int32_t row_popc(const uint32_t *bits, int64_t row) {
    const uint4 *r = reinterpret_cast<const uint4 *>(bits + row * 8);
    const uint4 a = r[0], b = r[1];
    return __popc(a.x) + __popc(a.y) + __popc(a.z) + __popc(a.w) + __popc(b.x) + __popc(b.y) + __popc(b.z) +
           __popc(b.w);
}

// Block-wide exclusive scan of one int per thread (kBThreads threads).
__device__ __forceinline__ int32_t block_excl_scan(int32_t v, int32_t *warp_sums, int32_t *total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[wid] = x;
    __syncthreads();
    if (wid == 0) {
        int32_t w = lane < kBThreads / 32 ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < kBThreads / 32) warp_sums[lane] = w;
    }
    __syncthreads();
    const int32_t before = wid > 0 ? warp_sums[wid - 1] : 0;
    if (total) *total = warp_sums[kBThreads / 32 - 1];
    return before + x - v;
}

// Level d, pass 1: the children of every tile of kScanTile parents.
__global__ void __launch_bounds__(kBThreads) k_b_tile_sums(int32_t d, const int32_t *__restrict__ ls,
                                                           const uint32_t *__restrict__ bits,
                                                           int32_t *__restrict__ tile_sum) {
    __shared__ int32_t ws[kBThreads / 32];
    pdl_launch_dependents();
    pdl_wait();
    const int32_t width = ls[d + 1] - ls[d];
    const int32_t t0 = blockIdx.x * kScanTile;
    if (t0 >= width) {
        if (threadIdx.x == 0) tile_sum[blockIdx.x] = 0;
        return;
    }
    int32_t s = 0;
    for (int32_t j = threadIdx.x; j < kScanTile; j += kBThreads)
        if (t0 + j < width) s += row_popc(bits, t0 + j);
    int32_t tot;
    block_excl_scan(s, ws, &tot);
    if (threadIdx.x == 0) tile_sum[blockIdx.x] = tot;
}

// Level d, pass 2: first child of every parent of the level (the level's
// end + the children of the earlier tiles + an exclusive scan within the
// tile); block 0 also writes the end of level d + 1. Clears the other bits
// buffer (level d - 1's rows), into which the moves of level d set the
// child-label sets of level d + 1.
__global__ void __launch_bounds__(kBThreads) k_b_first(int32_t d, int32_t n_tiles, int32_t *__restrict__ ls,
                                                       const uint32_t *__restrict__ bits,
                                                       const int32_t *__restrict__ tile_sum,
                                                       int32_t *__restrict__ first, uint32_t *__restrict__ other) {
    __shared__ int32_t ws[kBThreads / 32];
    __shared__ int32_t carry;
    pdl_launch_dependents();
    pdl_wait();
    const int32_t width = ls[d + 1] - ls[d];
    const int32_t prev = d > 0 ? ls[d] - ls[d - 1] : 0;
    const int32_t t0 = blockIdx.x * kScanTile;
    for (int32_t j = threadIdx.x; j < kScanTile; j += kBThreads)
        if (t0 + j < prev) {
            uint4 *r = reinterpret_cast<uint4 *>(other + int64_t(t0 + j) * 8);
            r[0] = make_uint4(0u, 0u, 0u, 0u);
            r[1] = make_uint4(0u, 0u, 0u, 0u);
        }
    if (t0 >= width && blockIdx.x > 0) return;
    // children of the tiles before this one (all tiles for block 0's total)
    const int32_t upto = blockIdx.x > 0 ? int32_t(blockIdx.x) : n_tiles;
    int32_t part = 0;
    for (int32_t t = threadIdx.x; t < upto; t += kBThreads) part += tile_sum[t];
    int32_t sum;
    block_excl_scan(part, ws, &sum);
    if (threadIdx.x == 0) {
        if (blockIdx.x == 0) {
            ls[d + 2] = ls[d + 1] + sum;
            carry = ls[d + 1];
        } else {
            carry = ls[d + 1] + sum;
        }
    }
    __syncthreads();
    if (t0 >= width) return;
    for (int32_t j0 = 0; j0 < kScanTile; j0 += kBThreads) {
        const int32_t x = t0 + j0 + threadIdx.x;
        const int32_t c = x < width ? row_popc(bits, x) : 0;
        int32_t tot;
        const int32_t ex = block_excl_scan(c, ws, &tot);
        if (x < width) first[x] = carry + ex;
        __syncthreads();
        if (threadIdx.x == 0) carry += tot;
        __syncthreads();
    }
}

// Level d, pass 3: every string of length > d moves to its child at depth
// d + 1, writing the child's parent, label, set, depth and terminal flag
// (all strings through a child write the same values), and sets its byte
// d + 1, if any, in the child's child-label set (level d + 1's rows).
__global__ void k_b_move(const uint8_t *__restrict__ bytes, const int64_t *__restrict__ off, int32_t K, int32_t d,
                         const int32_t *__restrict__ ls, const uint32_t *__restrict__ bits,
                         const int32_t *__restrict__ first, const int32_t *__restrict__ str_set,
                         int32_t *__restrict__ cur, int32_t *__restrict__ parent_g, uint8_t *__restrict__ label_g,
                         uint8_t *__restrict__ term_g, int32_t *__restrict__ set_g, int32_t *__restrict__ depth_g,
                         uint32_t *__restrict__ bits_next) {
    pdl_launch_dependents();
    pdl_wait();
    const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= K) return;
    const int64_t len = off[i + 1] - off[i];
    if (len <= d) return;
    const int64_t a = off[i] - off[0];
    const uint32_t b = bytes[a + d];
    const int32_t x = cur[i];
    const int64_t row = x - ls[d];
    const uint32_t *r = bits + row * 8;
    int32_t below = 0;
#pragma unroll
    for (int w = 0; w < 8; w++) {
        const uint32_t v = r[w];
        const int32_t lo = w * 32;
        if (int32_t(b) >= lo + 32) below += __popc(v);
        else if (int32_t(b) >= lo) below += __popc(v & ((1u << (b - lo)) - 1u));
    }
    const int32_t c = first[row] + below;
    parent_g[c] = x;
    label_g[c] = uint8_t(b);
    set_g[c] = str_set[i];
    depth_g[c] = d + 1;
    cur[i] = c;
    if (len == d + 1) {
        term_g[c] = 1;
    } else {
        const uint32_t b1 = bytes[a + d + 1];
        atomicOr(bits_next + int64_t(c - ls[d + 1]) * 8 + (b1 >> 5), 1u << (b1 & 31u));
    }
}

// Renumbering, pass 1: the level-order range [first, end) of every (set,
// depth) group (level order sorts by depth, then set, so each group is one
// run), and the characters of the distinct strings (depths of terminals).
__global__ void k_b_count(const int32_t *__restrict__ ls, int32_t D, const int32_t *__restrict__ set_g,
                          const int32_t *__restrict__ depth_g, const uint8_t *__restrict__ term_g,
                          int32_t *__restrict__ first_sd, int32_t *__restrict__ end_sd,
                          unsigned long long *__restrict__ n_chars) {
    pdl_launch_dependents();
    pdl_wait();
    const int32_t n = ls[D + 1];
    unsigned long long chars = 0;
    for (int32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < n; g += gridDim.x * blockDim.x) {
        const int32_t k = set_g[g] * (D + 1) + depth_g[g];
        if (g == 0 || set_g[g - 1] * (D + 1) + depth_g[g - 1] != k) first_sd[k] = g;
        if (g == n - 1 || set_g[g + 1] * (D + 1) + depth_g[g + 1] != k) end_sd[k] = g + 1;
        if (term_g[g]) chars += unsigned(depth_g[g]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) chars += __shfl_down_sync(0xffffffffu, chars, o);
    if ((threadIdx.x & 31) == 0 && chars) atomicAdd(n_chars, chars);
}

__device__ __forceinline__ int32_t group_size(const int32_t *first_sd, const int32_t *end_sd, int32_t k) {
    const int32_t e = end_sd[k];
    return e > 0 ? e - first_sd[k] : 0;  // end 0: no node of that set at that depth
}

// Renumbering, pass 2 (one CTA): the offset of every (set, depth) in the
// final layout (set after set, each in breadth-first order), and the roots.
__global__ void __launch_bounds__(kBThreads) k_b_offsets(int32_t M, int32_t D, const int32_t *__restrict__ first_sd,
                                                         const int32_t *__restrict__ end_sd,
                                                         int32_t *__restrict__ off_sd, int32_t *__restrict__ roots) {
    __shared__ int32_t ws[kBThreads / 32];
    __shared__ int32_t carry;
    pdl_launch_dependents();
    pdl_wait();
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int32_t s0 = 0; s0 < M; s0 += kBThreads) {
        const int32_t s = s0 + threadIdx.x;
        int32_t n_s = 0;
        if (s < M)
            for (int32_t d = 0; d <= D; d++) n_s += group_size(first_sd, end_sd, s * (D + 1) + d);
        int32_t tot;
        const int32_t base = carry + block_excl_scan(n_s, ws, &tot);
        if (s < M) {
            roots[s] = base;
            int32_t o = base;
            for (int32_t d = 0; d <= D; d++) {
                off_sd[s * (D + 1) + d] = o;
                o += group_size(first_sd, end_sd, s * (D + 1) + d);
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) carry += tot;
        __syncthreads();
    }
}

// Renumbering, pass 3: final id of every level-order id.
__global__ void k_b_map(const int32_t *__restrict__ ls, int32_t D, const int32_t *__restrict__ set_g,
                        const int32_t *__restrict__ depth_g, const int32_t *__restrict__ first_sd,
                        const int32_t *__restrict__ off_sd, int32_t *__restrict__ map) {
    pdl_launch_dependents();
    pdl_wait();
    const int32_t n = ls[D + 1];
    for (int32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < n; g += gridDim.x * blockDim.x) {
        const int32_t k = set_g[g] * (D + 1) + depth_g[g];
        map[g] = off_sd[k] + (g - first_sd[k]);
    }
}

// Renumbering, pass 4: parent, label and terminal in the final layout.
__global__ void k_b_permute(const int32_t *__restrict__ ls, int32_t D, const int32_t *__restrict__ map,
                            const int32_t *__restrict__ parent_g, const uint8_t *__restrict__ label_g,
                            const uint8_t *__restrict__ term_g, int32_t *__restrict__ parent,
                            uint8_t *__restrict__ label, uint8_t *__restrict__ terminal) {
    pdl_launch_dependents();
    pdl_wait();
    const int32_t n = ls[D + 1];
    for (int32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < n; g += gridDim.x * blockDim.x) {
        const int32_t f = map[g];
        const int32_t p = parent_g[g];
        parent[f] = p < 0 ? -1 : map[p];
        label[f] = label_g[g];
        terminal[f] = term_g[g];
    }
}

// ---- Forests of small sets: one CTA per set (kSetThreads threads, each
// owning up to kSetPer strings), the levels of that set in shared memory. The
// set's nodes are created in the order of the level path restricted to the
// set (breadth-first, sorted siblings) at local ids 0, 1, ..., written at
// ub(s) = (bytes before set s) + s, room for the set's at most 1 + bytes
// nodes; a scan of the node counts then gives every set its base.
constexpr int kSetThreads = 512;
constexpr int kSetPer = int(kSetMaxStrings / kSetThreads);

__device__ __forceinline__ int32_t block_reduce_max(int32_t v, int32_t *ws) {
    v = __reduce_max_sync(0xffffffffu, v);
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = v;
    __syncthreads();
    int32_t m = 0;
    for (int w = 0; w < int(blockDim.x >> 5); w++) m = max(m, ws[w]);
    __syncthreads();
    return m;
}

// Exclusive scan of one int per thread over a block of kSetThreads.
__device__ __forceinline__ int32_t set_excl_scan(int32_t v, int32_t *ws, int32_t *total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) ws[wid] = x;
    __syncthreads();
    if (wid == 0) {
        int32_t w = lane < kSetThreads / 32 ? ws[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < kSetThreads / 32) ws[lane] = w;
    }
    __syncthreads();
    const int32_t before = wid > 0 ? ws[wid - 1] : 0;
    *total = ws[kSetThreads / 32 - 1];
    __syncthreads();  // ws is reused by the next scan
    return before + x - v;
}

// Dynamic shared memory: the child-label sets of the current level
// (smax rows of 8 words), for each row the labels counted in its words before
// each word (8 bytes), the first child of each of its nodes, and a flag per
// node of the next level that some string ends at.
__global__ void __launch_bounds__(kSetThreads) k_b_sets(const uint8_t *__restrict__ bytes,
                                                        const int64_t *__restrict__ off,
                                                        const int32_t *__restrict__ set_off, int32_t M, int32_t smax,
                                                        int32_t *__restrict__ parent_ub, uint8_t *__restrict__ label_ub,
                                                        uint8_t *__restrict__ term_ub, int32_t *__restrict__ count,
                                                        unsigned long long *__restrict__ chars) {
    extern __shared__ uint4 dyn[];
    uint32_t *bits = reinterpret_cast<uint32_t *>(dyn);
    uint2 *cum = reinterpret_cast<uint2 *>(bits + int64_t(smax) * 8);
    int32_t *first = reinterpret_cast<int32_t *>(cum + smax);
    uint8_t *ends = reinterpret_cast<uint8_t *>(first + smax);
    __shared__ int32_t ws[kSetThreads / 32];
    __shared__ int32_t root_term;
    pdl_launch_dependents();
    pdl_wait();
    const int tid = threadIdx.x;
    for (int32_t r = tid; r < smax * 8; r += kSetThreads) bits[r] = 0u;
    for (int32_t r = tid; r < smax; r += kSetThreads) ends[r] = 0;
    for (int32_t s = blockIdx.x; s < M; s += gridDim.x) {
        const int32_t i0 = set_off[s], Ks = set_off[s + 1] - i0;
        const int64_t ub = off[i0] - off[0] + s;
        if (tid == 0) root_term = 0;
        __syncthreads();
        int32_t st[kSetPer], len[kSetPer], cur[kSetPer], nb[kSetPer];
        int32_t longest = 0;
#pragma unroll
        for (int k = 0; k < kSetPer; k++) {
            const int32_t j = tid + k * kSetThreads;
            len[k] = -1;
            cur[k] = 0;
            nb[k] = 0;
            st[k] = 0;
            if (j < Ks) {
                const int64_t a = off[i0 + j], e = off[i0 + j + 1];
                st[k] = int32_t(a - off[0]);
                len[k] = int32_t(e - a);
                longest = max(longest, len[k]);
                if (len[k] == 0) root_term = 1;
                else nb[k] = bytes[st[k]];
            }
        }
        const int32_t dmax = block_reduce_max(longest, ws);  // also orders root_term
        if (tid == 0) {
            parent_ub[ub] = -1;
            label_ub[ub] = 0;
            term_ub[ub] = uint8_t(root_term);
        }
        int32_t level_start = 0, level_end = 1;
        unsigned long long my_chars = 0;
        for (int32_t d = 0; d < dmax; d++) {
            const int32_t width = level_end - level_start;
#pragma unroll
            for (int k = 0; k < kSetPer; k++)
                if (len[k] > d)
                    atomicOr(bits + (cur[k] - level_start) * 8 + (nb[k] >> 5), 1u << (nb[k] & 31));
            __syncthreads();
            // first child of every node of the level: a contiguous chunk of rows per thread
            const int32_t per = (width + kSetThreads - 1) / kSetThreads;
            const int32_t r0 = min(tid * per, width), r1 = min(r0 + per, width);
            int32_t c = 0;
            for (int32_t r = r0; r < r1; r++) c += row_popc(bits, r);
            int32_t total;
            int32_t at = level_end + set_excl_scan(c, ws, &total);
            for (int32_t r = r0; r < r1; r++) {
                const uint4 *rw = reinterpret_cast<const uint4 *>(bits + int64_t(r) * 8);
                const uint4 lo = rw[0], hi = rw[1];
                const uint32_t p1 = __popc(lo.x), p2 = p1 + __popc(lo.y), p3 = p2 + __popc(lo.z),
                               p4 = p3 + __popc(lo.w), p5 = p4 + __popc(hi.x), p6 = p5 + __popc(hi.y),
                               p7 = p6 + __popc(hi.z);
                cum[r] = make_uint2((p1 << 8) | (p2 << 16) | (p3 << 24), p4 | (p5 << 8) | (p6 << 16) | (p7 << 24));
                first[r] = at;
                at += int32_t(p7 + __popc(hi.w));
            }
            __syncthreads();
#pragma unroll
            for (int k = 0; k < kSetPer; k++) {
                if (len[k] <= d) continue;
                const uint32_t b = uint32_t(nb[k]);
                const int32_t row = cur[k] - level_start;
                const uint32_t wi = b >> 5;
                const uint2 cm = cum[row];
                const uint32_t before = ((wi < 4 ? cm.x : cm.y) >> (8 * (wi & 3))) & 0xFFu;
                const int32_t below = int32_t(before + __popc(bits[row * 8 + wi] & ((1u << (b & 31)) - 1u)));
                const int32_t ch = first[row] + below;
                const int64_t g = ub + ch;
                parent_ub[g] = cur[k];
                label_ub[g] = uint8_t(b);
                if (len[k] == d + 1) {
                    term_ub[g] = 1;
                    ends[ch - level_end] = 1;
                } else {
                    nb[k] = bytes[st[k] + d + 1];
                }
                cur[k] = ch;
            }
            __syncthreads();
            for (int32_t r = tid; r < width * 8; r += kSetThreads) bits[r] = 0u;
            for (int32_t x = tid; x < total; x += kSetThreads)
                if (ends[x]) {
                    my_chars += unsigned(d + 1);
                    ends[x] = 0;
                }
            level_start = level_end;
            level_end += total;
            __syncthreads();
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) my_chars += __shfl_down_sync(0xffffffffu, my_chars, o);
        if ((tid & 31) == 0 && my_chars) atomicAdd(chars, my_chars);
        if (tid == 0) count[s] = level_end;
        __syncthreads();
    }
}

// One CTA: every set's base (exclusive scan of the node counts) = its root,
// and the total.
__global__ void __launch_bounds__(kBThreads) k_b_set_scan(int32_t M, const int32_t *__restrict__ count,
                                                          int32_t *__restrict__ roots, int32_t *__restrict__ total) {
    __shared__ int32_t ws[kBThreads / 32];
    __shared__ int32_t carry;
    pdl_launch_dependents();
    pdl_wait();
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int32_t s0 = 0; s0 < M; s0 += kBThreads) {
        const int32_t s = s0 + threadIdx.x;
        int32_t tot;
        const int32_t ex = block_excl_scan(s < M ? count[s] : 0, ws, &tot);
        if (s < M) roots[s] = carry + ex;
        __syncthreads();
        if (threadIdx.x == 0) carry += tot;
        __syncthreads();
    }
    if (threadIdx.x == 0) *total = carry;
}

// Every set's nodes from ub(s) + i to base(s) + i (kEmitParts CTAs per set,
// each a share of the set's nodes: one CTA per set left each thread ~70
// dependent copies at 256 sets of ~19,000 nodes).
constexpr int32_t kEmitParts = 8;
__global__ void k_b_set_emit(const int64_t *__restrict__ off, const int32_t *__restrict__ set_off, int32_t M,
                             const int32_t *__restrict__ count, const int32_t *__restrict__ roots,
                             const int32_t *__restrict__ parent_ub, const uint8_t *__restrict__ label_ub,
                             const uint8_t *__restrict__ term_ub, int32_t *__restrict__ parent,
                             uint8_t *__restrict__ label, uint8_t *__restrict__ terminal) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t u = blockIdx.x; u < int64_t(M) * kEmitParts; u += gridDim.x) {
        const int32_t s = int32_t(u / kEmitParts), part = int32_t(u % kEmitParts);
        const int64_t ub = off[set_off[s]] - off[0] + s;
        const int32_t base = roots[s], n = count[s];
        for (int32_t i = part * int32_t(blockDim.x) + threadIdx.x; i < n; i += kEmitParts * int32_t(blockDim.x)) {
            const int32_t p = parent_ub[ub + i];
            parent[base + i] = p < 0 ? -1 : base + p;
            label[base + i] = label_ub[ub + i];
            terminal[base + i] = term_ub[ub + i];
        }
    }
}

}  // namespace

// Scratch of one device build. Staging part: the strings, level-order node
// arrays (at most n_bytes + M nodes), two child-label buffers of
// max(K, M) rows, the level scans, the flags. Level part (once the longest
// string D is known): the level ends and the (set, depth) tables.
struct DeviceBuild::Scratch {
    void *base = nullptr, *base2 = nullptr;
    uint8_t *bytes;
    uint4 *image;
    int64_t *off;
    int32_t *set_off, *str_set, *cur, *parent_g, *set_g, *depth_g, *first, *tile_sum, *ls, *flags;
    uint8_t *label_g, *term_g;
    uint32_t *bits[2];
    int32_t *end_sd, *first_sd, *off_sd, *roots, *map;
    int32_t *count, *total;  // small-set path: nodes per set, all nodes
    unsigned long long *n_chars;
};

DeviceBuild::~DeviceBuild() {
    if (s_) {
        if (s_->base) cudaFreeAsync(s_->base, stream_);
        if (s_->base2) cudaFreeAsync(s_->base2, stream_);
        delete s_;
    }
}

namespace {

struct Carver {
    size_t total = 0;
    size_t add(size_t b) {
        const size_t o = total;
        total += (b + 255) / 256 * 256;
        return o;
    }
};

}  // namespace

cudaError_t DeviceBuild::stage(const uint8_t *h_bytes, const int64_t *h_off, const int32_t *h_set_off, int32_t M,
                               int32_t K, int64_t n_bytes, bool direct, int num_sms, cudaMemPool_t pool,
                               cudaStream_t st, int32_t *max_len, bool *offsets_ok) {
    stream_ = st;
    pool_ = pool;
    M_ = M;
    K_ = K;
    n_bytes_ = n_bytes;
    smax_ = 1;
    for (int32_t i = 0; i < M; i++) smax_ = std::max(smax_, h_set_off[i + 1] - h_set_off[i]);
    small_ = smax_ <= kSetMaxStrings;
    s_ = new Scratch();
    const int64_t U = n_bytes + M;               // nodes at most
    const int64_t W = std::max<int64_t>(K, M);   // parents of one level at most
    const int64_t tiles = (W + kScanTile - 1) / kScanTile + 1;
    Carver c;
    const size_t o_img = c.add(size_t(n_bytes) + 32), o_off = c.add(8 * (size_t(K) + 1)),
                 o_soff = c.add(4 * (size_t(M) + 1)), o_sset = c.add(4 * size_t(K)), o_cur = c.add(4 * size_t(K)),
                 o_par = c.add(4 * size_t(U)), o_set = c.add(4 * size_t(U)), o_dep = c.add(4 * size_t(U)),
                 o_first = c.add(4 * size_t(W)), o_ts = c.add(4 * size_t(tiles)), o_lab = c.add(size_t(U)),
                 o_term = c.add(size_t(U)), o_b0 = c.add(32 * size_t(W) + 32), o_b1 = c.add(32 * size_t(W) + 32),
                 o_roots = c.add(4 * size_t(M)), o_map = c.add(4 * size_t(U)), o_nch = c.add(8), o_flags = c.add(8);
    cudaError_t e = cudaMallocFromPoolAsync(&s_->base, c.total, pool, st);
    if (e != cudaSuccess) return e;
    char *b = static_cast<char *>(s_->base);
    const size_t mis = reinterpret_cast<uintptr_t>(h_bytes) & 15u;  // the image keeps the source's alignment
    s_->image = reinterpret_cast<uint4 *>(b + o_img);
    s_->bytes = reinterpret_cast<uint8_t *>(b + o_img) + mis;
    s_->off = reinterpret_cast<int64_t *>(b + o_off);
    s_->set_off = reinterpret_cast<int32_t *>(b + o_soff);
    s_->str_set = reinterpret_cast<int32_t *>(b + o_sset);
    s_->cur = reinterpret_cast<int32_t *>(b + o_cur);
    s_->parent_g = reinterpret_cast<int32_t *>(b + o_par);
    s_->set_g = reinterpret_cast<int32_t *>(b + o_set);
    s_->depth_g = reinterpret_cast<int32_t *>(b + o_dep);
    s_->first = reinterpret_cast<int32_t *>(b + o_first);
    s_->tile_sum = reinterpret_cast<int32_t *>(b + o_ts);
    s_->label_g = reinterpret_cast<uint8_t *>(b + o_lab);
    s_->term_g = reinterpret_cast<uint8_t *>(b + o_term);
    s_->bits[0] = reinterpret_cast<uint32_t *>(b + o_b0);
    s_->bits[1] = reinterpret_cast<uint32_t *>(b + o_b1);
    s_->roots = reinterpret_cast<int32_t *>(b + o_roots);
    s_->map = reinterpret_cast<int32_t *>(b + o_map);
    s_->n_chars = reinterpret_cast<unsigned long long *>(b + o_nch);
    s_->flags = reinterpret_cast<int32_t *>(b + o_flags);
    if ((e = cudaMemsetAsync(s_->term_g, 0, size_t(U), st)) != cudaSuccess ||
        (e = cudaMemsetAsync(s_->bits[0], 0, 32 * size_t(W) + 32, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(s_->bits[1], 0, 32 * size_t(W) + 32, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(s_->n_chars, 0, 8, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(s_->flags, 0, 8, st)) != cudaSuccess)
        return e;
    const int64_t n_vec = n_bytes > 0 ? (int64_t(mis) + n_bytes + 15) / 16 : 0;
    const int64_t items = std::max<int64_t>(std::max<int64_t>(K, M) + 1, n_vec);
    const int64_t grid = std::min<int64_t>((items + kBThreads - 1) / kBThreads, int64_t(num_sms) * 16);
    if (direct) {
        e = launch_pdl(k_b_stage, grid, kBThreads, st, h_off, K, h_set_off, M,
                   reinterpret_cast<const uint4 *>(h_bytes - mis), n_vec, s_->off, s_->set_off, s_->image, s_->flags);
    } else {
        if ((n_bytes > 0 && (e = cudaMemcpyAsync(s_->bytes, h_bytes, size_t(n_bytes), cudaMemcpyHostToDevice, st)) !=
                                cudaSuccess) ||
            (e = cudaMemcpyAsync(s_->off, h_off, 8 * (size_t(K) + 1), cudaMemcpyHostToDevice, st)) != cudaSuccess ||
            (e = cudaMemcpyAsync(s_->set_off, h_set_off, 4 * (size_t(M) + 1), cudaMemcpyHostToDevice, st)) !=
                cudaSuccess)
            return e;
        e = launch_pdl(k_b_stage, grid, kBThreads, st, static_cast<const int64_t *>(s_->off), K,
                   static_cast<const int32_t *>(s_->set_off), M, static_cast<const uint4 *>(nullptr), int64_t(0),
                   s_->off, s_->set_off, s_->image, s_->flags);
    }
    if (e != cudaSuccess) return e;
    int32_t flags[2] = {0, 0};
    if ((e = cudaMemcpyAsync(flags, s_->flags, sizeof(flags), cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess)
        return e;
    *offsets_ok = flags[0] == 0;
    *max_len = flags[1];
    return cudaSuccess;
}

cudaError_t DeviceBuild::levels(int32_t D, int num_sms, int32_t *n_nodes, std::vector<int32_t> *roots,
                                int64_t *n_chars) {
    const cudaStream_t st = stream_;
    const int32_t M = M_, K = K_;
    D_ = D;
    if (small_) return sets(num_sms, n_nodes, roots, n_chars);
    const int64_t U = n_bytes_ + M;
    const int64_t W = std::max<int64_t>(K, M);
    const int64_t sd = int64_t(M) * (D + 1);
    Carver c;
    const size_t o_ls = c.add(4 * (size_t(D) + 2)), o_end = c.add(4 * size_t(sd)), o_fsd = c.add(4 * size_t(sd)),
                 o_osd = c.add(4 * size_t(sd));
    cudaError_t e = cudaMallocFromPoolAsync(&s_->base2, c.total, pool_, st);
    if (e != cudaSuccess) return e;
    char *b = static_cast<char *>(s_->base2);
    s_->ls = reinterpret_cast<int32_t *>(b + o_ls);
    s_->end_sd = reinterpret_cast<int32_t *>(b + o_end);
    s_->first_sd = reinterpret_cast<int32_t *>(b + o_fsd);
    s_->off_sd = reinterpret_cast<int32_t *>(b + o_osd);
    if ((e = cudaMemsetAsync(s_->end_sd, 0, 4 * size_t(sd), st)) != cudaSuccess) return e;
    const int64_t sgrid = (W + kBThreads - 1) / kBThreads;
    if ((e = launch_pdl(k_b_init, sgrid, kBThreads, st, static_cast<const uint8_t *>(s_->bytes),
                    static_cast<const int64_t *>(s_->off), static_cast<const int32_t *>(s_->set_off), M, K,
                    s_->str_set, s_->cur, s_->parent_g, s_->label_g, s_->term_g, s_->set_g, s_->depth_g, s_->ls,
                    s_->bits[0])) != cudaSuccess)
        return e;
    const int64_t kgrid = (int64_t(K) + kBThreads - 1) / kBThreads;
    const int32_t n_tiles = int32_t((W + kScanTile - 1) / kScanTile);
    for (int32_t d = 0; d < D; d++) {  // level d: bits[d & 1] holds its child-label sets
        uint32_t *bits = s_->bits[d & 1], *next = s_->bits[(d + 1) & 1];
        if ((e = launch_pdl(k_b_tile_sums, n_tiles, kBThreads, st, d, static_cast<const int32_t *>(s_->ls),
                        static_cast<const uint32_t *>(bits), s_->tile_sum)) != cudaSuccess ||
            (e = launch_pdl(k_b_first, n_tiles, kBThreads, st, d, n_tiles, s_->ls, static_cast<const uint32_t *>(bits),
                        static_cast<const int32_t *>(s_->tile_sum), s_->first, next)) != cudaSuccess ||
            (e = launch_pdl(k_b_move, kgrid, kBThreads, st, static_cast<const uint8_t *>(s_->bytes),
                        static_cast<const int64_t *>(s_->off), K, d, static_cast<const int32_t *>(s_->ls),
                        static_cast<const uint32_t *>(bits), static_cast<const int32_t *>(s_->first),
                        static_cast<const int32_t *>(s_->str_set), s_->cur, s_->parent_g, s_->label_g, s_->term_g,
                        s_->set_g, s_->depth_g, next)) != cudaSuccess)
            return e;
    }
    const int64_t ngrid = std::min<int64_t>((U + kBThreads - 1) / kBThreads, int64_t(num_sms) * 16);
    if ((e = launch_pdl(k_b_count, ngrid, kBThreads, st, static_cast<const int32_t *>(s_->ls), D,
                    static_cast<const int32_t *>(s_->set_g), static_cast<const int32_t *>(s_->depth_g),
                    static_cast<const uint8_t *>(s_->term_g), s_->first_sd, s_->end_sd, s_->n_chars)) != cudaSuccess ||
        (e = launch_pdl(k_b_offsets, 1, kBThreads, st, M, D, static_cast<const int32_t *>(s_->first_sd),
                    static_cast<const int32_t *>(s_->end_sd), s_->off_sd, s_->roots)) != cudaSuccess ||
        (e = launch_pdl(k_b_map, ngrid, kBThreads, st, static_cast<const int32_t *>(s_->ls), D,
                    static_cast<const int32_t *>(s_->set_g), static_cast<const int32_t *>(s_->depth_g),
                    static_cast<const int32_t *>(s_->first_sd), static_cast<const int32_t *>(s_->off_sd), s_->map)) !=
            cudaSuccess)
        return e;
    // the node count, the roots and the characters (host-synchronous)
    int32_t n = 0;
    unsigned long long nc = 0;
    roots->resize(size_t(M));
    if ((e = cudaMemcpyAsync(&n, s_->ls + D + 1, 4, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(roots->data(), s_->roots, 4 * size_t(M), cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(&nc, s_->n_chars, 8, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess)
        return e;
    *n_nodes = n;
    *n_chars = int64_t(nc);
    n_ = n;
    return cudaSuccess;
}

cudaError_t DeviceBuild::sets(int num_sms, int32_t *n_nodes, std::vector<int32_t> *roots, int64_t *n_chars) {
    const cudaStream_t st = stream_;
    const int32_t M = M_;
    Carver c;
    const size_t o_cnt = c.add(4 * size_t(M)), o_tot = c.add(4);
    cudaError_t e = cudaMallocFromPoolAsync(&s_->base2, c.total, pool_, st);
    if (e != cudaSuccess) return e;
    char *b = static_cast<char *>(s_->base2);
    s_->count = reinterpret_cast<int32_t *>(b + o_cnt);
    s_->total = reinterpret_cast<int32_t *>(b + o_tot);
    const size_t smem = size_t(smax_) * (8 * sizeof(uint32_t) + sizeof(uint2) + sizeof(int32_t) + 1);
    int per_sm = 0;
    if ((e = cudaFuncSetAttribute(k_b_sets, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem))) !=
            cudaSuccess ||
        (e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_b_sets, kSetThreads, smem)) != cudaSuccess)
        return e;
    const int64_t grid = std::min<int64_t>(M, int64_t(num_sms) * std::max(per_sm, 1));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(grid));
    cfg.blockDim = dim3(unsigned(kSetThreads));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if ((e = cudaLaunchKernelEx(&cfg, k_b_sets, static_cast<const uint8_t *>(s_->bytes),
                                static_cast<const int64_t *>(s_->off), static_cast<const int32_t *>(s_->set_off), M,
                                smax_, s_->parent_g, s_->label_g, s_->term_g, s_->count, s_->n_chars)) !=
            cudaSuccess ||
        (e = launch_pdl(k_b_set_scan, 1, kBThreads, st, M, static_cast<const int32_t *>(s_->count), s_->roots,
                    s_->total)) != cudaSuccess)
        return e;
    int32_t n = 0;
    unsigned long long nc = 0;
    roots->resize(size_t(M));
    if ((e = cudaMemcpyAsync(&n, s_->total, 4, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(roots->data(), s_->roots, 4 * size_t(M), cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(&nc, s_->n_chars, 8, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess)
        return e;
    *n_nodes = n;
    *n_chars = int64_t(nc);
    n_ = n;
    return cudaSuccess;
}

cudaError_t DeviceBuild::emit(int32_t *parent, uint8_t *label, uint8_t *terminal, int num_sms) {
    if (small_)
        return launch_pdl(k_b_set_emit, std::min<int64_t>(int64_t(M_) * kEmitParts, int64_t(num_sms) * 16), kBThreads,
                          stream_,
                      static_cast<const int64_t *>(s_->off), static_cast<const int32_t *>(s_->set_off), M_,
                      static_cast<const int32_t *>(s_->count), static_cast<const int32_t *>(s_->roots),
                      static_cast<const int32_t *>(s_->parent_g), static_cast<const uint8_t *>(s_->label_g),
                      static_cast<const uint8_t *>(s_->term_g), parent, label, terminal);
    const int64_t ngrid = std::min<int64_t>((int64_t(n_) + kBThreads - 1) / kBThreads, int64_t(num_sms) * 16);
    return launch_pdl(k_b_permute, ngrid, kBThreads, stream_, static_cast<const int32_t *>(s_->ls), D_,
                  static_cast<const int32_t *>(s_->map), static_cast<const int32_t *>(s_->parent_g),
                  static_cast<const uint8_t *>(s_->label_g), static_cast<const uint8_t *>(s_->term_g), parent, label,
                  terminal);
}

}  // namespace tmk
