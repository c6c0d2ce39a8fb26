// sm_103a kernels of libtriemask.
//
//  k_mask_fill   dense part of the mask compile: writes every mask word once
//                (zero) with 16-byte streaming stores. HBM-write bound.
//  k_mask_patch  sparse part: one thread per trie node m finds every token
//                whose bytes spell the last k edges into m (k = 1..lmax) and
//                sets that token's bit in the row of the node k edges above m.
//                These are exactly the Aho-Corasick outputs of Sec. 4.2 step
//                2 ("a vocabulary token's characters end at the current trie
//                node; that token started |token| characters earlier, at its
//                start node", App. G.1 Step 3), found by a hash lookup per
//                suffix instead of by failure links, so that every node is
//                independent. Cost O(N * min(depth, l)) lookups, the paper's
//                O(N_chars * l) traversal bound.
//  k_advance     delta*(s, bytes(token)) per request (Sec. 2, Eq. 1).
//  k_apply_vec   -inf into the logits of disallowed tokens (Sec. 4.2; App.
//                H.3); one warp per 1024-token segment of a row, 16-byte
//                stores, the logits are read only where some token of the
//                16-byte chunk is allowed.
#include <stdint.h>

#include <cuda_runtime.h>

#include "tm_internal.h"

namespace tmk {

namespace {

constexpr int kThreads = 256;
constexpr int32_t kDead = -1;
constexpr int32_t kFinished = -2;

__global__ void __launch_bounds__(kThreads) k_mask_fill(uint32_t *__restrict__ mask, int64_t n_words,
                                                        int64_t head) {
    const int64_t tid = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    const int64_t nth = int64_t(gridDim.x) * blockDim.x;
    if (tid < head) mask[tid] = 0u;
    uint4 *v = reinterpret_cast<uint4 *>(mask + head);
    const int64_t n4 = (n_words - head) >> 2;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    int64_t i = tid;
    for (; i + 3 * nth < n4; i += 4 * nth) {
        __stcs(v + i, z);
        __stcs(v + i + nth, z);
        __stcs(v + i + 2 * nth, z);
        __stcs(v + i + 3 * nth, z);
    }
    for (; i < n4; i += nth) __stcs(v + i, z);
    const int64_t tail0 = head + (n4 << 2);
    if (tid < n_words - tail0) mask[tail0 + tid] = 0u;
}

// True iff the token bytes tok[0..k) equal the labels of the k edges that end
// at node m (read bottom-up).
__device__ __forceinline__ bool path_equals(const int32_t *__restrict__ parent,
                                            const uint8_t *__restrict__ label, int32_t m,
                                            const uint8_t *__restrict__ tok, int32_t k) {
    int32_t y = m;
    for (int32_t j = k - 1; j >= 0; j--) {
        if (y < 0 || label[y] != tok[j]) return false;
        y = parent[y];
    }
    return true;
}

__global__ void __launch_bounds__(kThreads) k_mask_patch(
    const int32_t *__restrict__ parent, const uint8_t *__restrict__ label,
    const uint8_t *__restrict__ terminal, int32_t n_nodes, const uint64_t *__restrict__ ht_key,
    const int32_t *__restrict__ ht_val, uint32_t ht_mask, const uint32_t *__restrict__ tok_off,
    const uint16_t *__restrict__ tok_len, const uint8_t *__restrict__ blob, int32_t lmax,
    uint32_t *__restrict__ mask, int64_t W, int32_t eos) {
    const int32_t stride = gridDim.x * blockDim.x;
    for (int32_t m = blockIdx.x * blockDim.x + threadIdx.x; m < n_nodes; m += stride) {
        // EOS is allowed exactly at terminal nodes (App. G.5, EOS handling)
        if (terminal[m]) atomicOr(mask + int64_t(m) * W + (eos >> 5), 1u << (eos & 31));
        uint64_t h = 0, pw = 1;
        int32_t x = m;
        for (int32_t k = 1; k <= lmax; k++) {
            const int32_t p = parent[x];
            if (p < 0) break;
            h += (uint64_t(label[x]) + 1ull) * pw;  // prepend one byte to the suffix
            pw *= kHashBase;
            x = p;  // the suffix of length k starts at node x
            const uint64_t key = hash_finish(h, uint32_t(k));
            uint32_t slot = uint32_t(key) & ht_mask;
            for (uint32_t probe = 0; probe <= ht_mask; probe++) {  // ends at an empty slot
                const uint64_t kk = ht_key[slot];
                if (kk == 0ull) break;
                if (kk == key) {
                    const int32_t t = ht_val[slot];
                    if (int32_t(tok_len[t]) == k && path_equals(parent, label, m, blob + tok_off[t], k))
                        atomicOr(mask + int64_t(x) * W + (t >> 5), 1u << (t & 31));
                }
                slot = (slot + 1u) & ht_mask;
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads) k_advance(
    const int32_t *__restrict__ first_child, const uint32_t *__restrict__ child_bits,
    const uint8_t *__restrict__ terminal, int32_t n_nodes, const uint32_t *__restrict__ tok_off,
    const uint16_t *__restrict__ tok_len, const uint8_t *__restrict__ blob, int32_t V,
    int32_t *__restrict__ states, const int32_t *__restrict__ tokens, int32_t B,
    int32_t *__restrict__ err) {
    const int32_t b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    const int32_t s = states[b];
    if (s == kDead) return;
    const int32_t v = tokens[b];
    const int32_t eos = V - 1;
    int32_t nxt;
    if (v < 0 || v >= V) {
        nxt = kDead;
    } else if (s == kFinished) {
        nxt = (v == eos) ? kFinished : kDead;
    } else if (s < 0 || s >= n_nodes) {
        nxt = kDead;
    } else if (v == eos) {
        nxt = terminal[s] ? kFinished : kDead;
    } else {
        const int32_t L = tok_len[v];
        const uint8_t *p = blob + tok_off[v];
        int32_t x = s;
        nxt = L > 0 ? s : kDead;
        for (int32_t j = 0; j < L; j++) {
            const uint32_t c = p[j];
            const uint4 *cb = reinterpret_cast<const uint4 *>(child_bits + int64_t(x) * 8);
            const uint4 lo = cb[0], hi = cb[1];
            const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
            const uint32_t wi = c >> 5, bit = c & 31u;
            uint32_t below = 0, cur = 0;
#pragma unroll
            for (uint32_t i = 0; i < 8; i++) {
                below += (i < wi) ? __popc(w[i]) : 0u;
                cur = (i == wi) ? w[i] : cur;
            }
            if (!((cur >> bit) & 1u)) {
                nxt = kDead;
                break;
            }
            x = first_child[x] + int32_t(below + __popc(cur & ((1u << bit) - 1u)));
            nxt = x;
        }
    }
    if (nxt == kDead && err) atomicAdd(err, 1);
    states[b] = nxt;
}

// Mask word of (state, word index w): the node's row, or {EOS} for FINISHED,
// DEAD and ids that are not nodes.
__device__ __forceinline__ uint32_t row_word(const uint32_t *__restrict__ mask, int32_t s,
                                             int32_t n_nodes, int64_t W, int64_t w, int32_t eos) {
    if (w >= W) return 0u;
    if (s >= 0 && s < n_nodes) return __ldg(mask + int64_t(s) * W + w);
    return (w == (eos >> 5)) ? (1u << (eos & 31)) : 0u;
}

// kElt = 2 (bf16) or 4 (fp32). Requires V % (16 / kElt) == 0 and a 16-byte
// aligned logits base, so that every row starts on a 16-byte boundary.
template <int kElt>
__global__ void __launch_bounds__(kThreads) k_apply_vec(uint4 *__restrict__ logits,
                                                        const uint32_t *__restrict__ mask,
                                                        const int32_t *__restrict__ states, int32_t B,
                                                        int32_t V, int64_t W, int32_t n_nodes,
                                                        int32_t segs_per_row) {
    constexpr int kPer = 16 / kElt;             // tokens per 16-byte chunk
    constexpr int kChunks = 1024 / kPer / 32;   // chunks per lane per segment
    const int64_t gw = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (gw >= int64_t(B) * segs_per_row) return;  // uniform per warp
    const int32_t b = int32_t(gw / segs_per_row);
    const int32_t seg = int32_t(gw % segs_per_row);
    const int32_t s = __ldg(states + b);
    const int32_t eos = V - 1;
    const uint32_t word = row_word(mask, s, n_nodes, W, int64_t(seg) * 32 + lane, eos);
    const int64_t row_chunks = int64_t(V) / kPer;
    uint4 *row = logits + int64_t(b) * row_chunks;
    const uint4 ninf = (kElt == 2) ? make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u)
                                   : make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
#pragma unroll
    for (int j = 0; j < kChunks; j++) {
        const int q = j * 32 + lane;                        // chunk within the segment
        const uint32_t wv = __shfl_sync(0xffffffffu, word, (q * kPer) >> 5);
        const uint32_t bits = (wv >> ((q * kPer) & 31)) & ((1u << kPer) - 1u);
        const int64_t chunk = int64_t(seg) * (1024 / kPer) + q;
        if (chunk >= row_chunks) continue;
        if (bits == 0u) {
            row[chunk] = ninf;
        } else {
            uint4 x = row[chunk];
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
            row[chunk] = make_uint4(e[0], e[1], e[2], e[3]);
        }
    }
}

// Any V and alignment: one thread per logit.
template <int kElt>
__global__ void __launch_bounds__(kThreads) k_apply_scalar(void *__restrict__ logits,
                                                           const uint32_t *__restrict__ mask,
                                                           const int32_t *__restrict__ states, int32_t B,
                                                           int32_t V, int64_t W, int32_t n_nodes) {
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

inline int grid_for(int64_t work, int64_t per_block, int64_t cap) {
    int64_t g = (work + per_block - 1) / per_block;
    if (g < 1) g = 1;
    if (g > cap) g = cap;
    return int(g);
}

}  // namespace

cudaError_t launch_mask_fill(uint32_t *mask, int64_t n_words, int num_sms, cudaStream_t st) {
    const uintptr_t a = reinterpret_cast<uintptr_t>(mask);
    int64_t head = int64_t(((16u - (a & 15u)) & 15u) >> 2);
    if (head > n_words) head = n_words;
    const int64_t n4 = (n_words - head) >> 2;
    const int grid = grid_for(n4, kThreads, int64_t(num_sms) * 8);
    k_mask_fill<<<grid, kThreads, 0, st>>>(mask, n_words, head);
    return cudaGetLastError();
}

cudaError_t launch_mask_patch(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t lmax,
                              uint32_t *mask, int64_t W, int num_sms, cudaStream_t st) {
    const int grid = grid_for(n_nodes, kThreads, int64_t(num_sms) * 64);
    k_mask_patch<<<grid, kThreads, 0, st>>>(t.parent, t.label, t.terminal, n_nodes, v.ht_key, v.ht_val,
                                            v.ht_mask, v.tok_off, v.tok_len, v.blob, lmax, mask, W,
                                            v.V - 1);
    return cudaGetLastError();
}

cudaError_t launch_advance(const DevTrie &t, int32_t n_nodes, const DevVocab &v, int32_t *states,
                           const int32_t *tokens, int32_t B, int32_t *err, cudaStream_t st) {
    const int grid = (B + kThreads - 1) / kThreads;
    k_advance<<<grid, kThreads, 0, st>>>(t.first_child, t.child_bits, t.terminal, n_nodes, v.tok_off,
                                         v.tok_len, v.blob, v.V, states, tokens, B, err);
    return cudaGetLastError();
}

cudaError_t launch_apply(void *logits, int dtype, const uint32_t *mask, const int32_t *states,
                         int32_t B, int32_t V, int32_t n_nodes, int num_sms, cudaStream_t st) {
    const int64_t W = (int64_t(V) + 31) / 32;
    const int elt = dtype == 0 ? 4 : 2;
    const bool vec = (reinterpret_cast<uintptr_t>(logits) & 15u) == 0 && (int64_t(V) * elt) % 16 == 0;
    if (vec) {
        const int32_t segs = int32_t((W + 31) / 32);
        const int64_t warps = int64_t(B) * segs;
        const int grid = grid_for(warps * 32, kThreads, INT32_MAX);
        if (elt == 2)
            k_apply_vec<2><<<grid, kThreads, 0, st>>>(static_cast<uint4 *>(logits), mask, states, B, V, W,
                                                      n_nodes, segs);
        else
            k_apply_vec<4><<<grid, kThreads, 0, st>>>(static_cast<uint4 *>(logits), mask, states, B, V, W,
                                                      n_nodes, segs);
    } else {
        const int grid = grid_for(int64_t(B) * V, kThreads, int64_t(num_sms) * 16);
        if (elt == 2)
            k_apply_scalar<2><<<grid, kThreads, 0, st>>>(logits, mask, states, B, V, W, n_nodes);
        else
            k_apply_scalar<4><<<grid, kThreads, 0, st>>>(logits, mask, states, B, V, W, n_nodes);
    }
    return cudaGetLastError();
}

}  // namespace tmk
