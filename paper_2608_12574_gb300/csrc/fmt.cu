// sm_103a kernels of the character-position masks for fixed-format strings
// (App. K, constraint-aware dispatch beyond finite sets): a format of length
// L is a sequence of byte classes C_0..C_{L-1}; the automaton's states are
// the positions 0..L. Token v (not EOS) is allowed at position p iff
// 1 <= len(v) <= L - p and byte i of v lies in C_{p+i}; EOS iff p = L.
//
//  k_fmt_compile  the dense mask [L + 1, ceil(V/32)]: one warp per 32 tokens
//                 (one per lane, its first 16 bytes loaded once into
//                 registers); for formats of at most 63 positions the set of
//                 positions where a token fits is one AND of 64-bit masks per
//                 byte, longer formats check every position against the
//                 classes in shared memory; each position's word is written
//                 by a ballot.
//  k_fmt_advance  p -> p + len(v) for allowed tokens, with the FINISHED /
//                 DEAD rules of the trie automaton.
// The masks have the trie masks' layout, so the apply kernels serve both.
#include <stdint.h>

#include <cuda_runtime.h>

#include "tm_internal.h"

namespace tmk {

namespace {

constexpr int32_t kFmtDead = -1;
constexpr int32_t kFmtFinished = -2;
constexpr int kFmtThreads = 256;

struct FmtArgs {
    const uint32_t *classes;  // [L * 8] words: byte c of class i is bit c % 32 of word 8 i + c / 32
    int32_t L;
    const uint32_t *tok_off;
    const uint16_t *tok_len;
    const uint8_t *blob;      // token bytes, each token 16-byte aligned
    int32_t V;
};


// Every byte of token v (len bytes at blob + off) lies in the class of its
// position, starting at position p (the caller has checked p + len <= L).
__device__ __forceinline__ bool token_fits(const uint32_t *cls, int32_t p, const uint8_t *blob, uint32_t off,
                                           int32_t len) {
    for (int32_t c0 = 0; c0 < len; c0 += 16) {
        const uint4 q = __ldg(reinterpret_cast<const uint4 *>(blob + off + c0));
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int i = 0; i < 16; i++) {
            if (c0 + i >= len) break;
            const uint32_t b = (w[i >> 2] >> ((i & 3) * 8)) & 0xFFu;
            if (!((cls[(p + c0 + i) * 8 + int32_t(b >> 5)] >> (b & 31u)) & 1u)) return false;
        }
    }
    return true;
}

__device__ __forceinline__ bool fmt_allows(const FmtArgs &a, const uint32_t *cls, int32_t p, int32_t v) {
    if (v == a.V - 1) return p == a.L;
    const int32_t len = a.tok_len[v];
    if (len < 1 || len > a.L - p) return false;
    return token_fits(cls, p, a.blob, a.tok_off[v], len);
}

// Positions at which a token fits, for formats of at most 63 positions:
// pos_of_byte[b] has bit q set iff byte b lies in class q, so the token
// b_0..b_{n-1} fits at p iff bit p of AND_i (pos_of_byte[b_i] >> i) is set,
// and p <= L - n. q holds the token's first 16 bytes; later ones are loaded.
__device__ __forceinline__ uint64_t token_positions(const uint64_t *pos_of_byte, int32_t L, uint4 q,
                                                    const uint8_t *blob, uint32_t off, int32_t len) {
    if (len < 1 || len > L) return 0ull;
    uint64_t S = (2ull << (L - len)) - 1ull;  // p = 0 .. L - len
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 16; i++)
        if (i < len) S &= pos_of_byte[(w[i >> 2] >> ((i & 3) * 8)) & 0xFFu] >> i;
    for (int32_t c0 = 16; c0 < len && S; c0 += 16) {
        const uint4 r = __ldg(reinterpret_cast<const uint4 *>(blob + off + c0));
        const uint32_t x[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int i = 0; i < 16; i++)
            if (c0 + i < len) S &= pos_of_byte[(x[i >> 2] >> ((i & 3) * 8)) & 0xFFu] >> (c0 + i);
    }
    return S;
}

__global__ void __launch_bounds__(kFmtThreads) k_fmt_compile(FmtArgs a, uint32_t *__restrict__ mask, int64_t W) {
    __shared__ uint32_t cls[kFmtMaxLen * 8];
    __shared__ uint64_t pos_of_byte[256];
    for (int32_t i = threadIdx.x; i < a.L * 8; i += blockDim.x) cls[i] = __ldg(a.classes + i);
    const bool short_fmt = a.L <= 63;
    if (short_fmt) {
        for (int32_t c = threadIdx.x; c < 256; c += blockDim.x) {
            uint64_t m = 0ull;
            for (int32_t p = 0; p < a.L; p++) m |= uint64_t((__ldg(a.classes + p * 8 + (c >> 5)) >> (c & 31)) & 1u) << p;
            pos_of_byte[c] = m;
        }
    }
    __syncthreads();
    pdl_launch_dependents();
    pdl_wait();  // an earlier kernel may still read the mask
    const int lane = threadIdx.x & 31;
    const int64_t warps = int64_t(gridDim.x) * (blockDim.x / 32);
    for (int64_t w = int64_t(blockIdx.x) * (blockDim.x / 32) + (threadIdx.x >> 5); w < W; w += warps) {
        const int64_t t = w * 32 + lane;
        const bool eos = t == a.V - 1;
        const int32_t len = (t < a.V - 1) ? int32_t(__ldg(a.tok_len + t)) : 0;
        const uint32_t off = len > 0 ? __ldg(a.tok_off + t) : 0u;
        const uint4 q = len > 0 ? __ldg(reinterpret_cast<const uint4 *>(a.blob + off)) : make_uint4(0u, 0u, 0u, 0u);
        if (short_fmt) {
            const uint64_t S = eos ? (1ull << a.L) : token_positions(pos_of_byte, a.L, q, a.blob, off, len);
            for (int32_t p = 0; p <= a.L; p++) {
                const uint32_t word = __ballot_sync(0xffffffffu, (S >> p) & 1ull);
                if (lane == 0) mask[int64_t(p) * W + w] = word;
            }
        } else {
            for (int32_t p = 0; p <= a.L; p++) {
                const bool ok = eos ? p == a.L
                                    : (len >= 1 && len <= a.L - p && token_fits(cls, p, a.blob, off, len));
                const uint32_t word = __ballot_sync(0xffffffffu, ok);
                if (lane == 0) mask[int64_t(p) * W + w] = word;
            }
        }
    }
}

// states_out[b] = the position after tokens[b] (in place allowed).
__global__ void __launch_bounds__(kFmtThreads) k_fmt_advance(FmtArgs a, const int32_t *states_in,
                                                             int32_t *states_out,
                                                             const int32_t *__restrict__ tokens, int32_t B,
                                                             int32_t *__restrict__ err) {
    pdl_launch_dependents();
    pdl_wait();  // states and tokens come from earlier kernels
    const int32_t b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    const int32_t s = states_in[b], v = tokens[b];
    int32_t nxt;
    if (s == kFmtDead) nxt = kFmtDead;
    else if (v < 0 || v >= a.V) nxt = kFmtDead;
    else if (s == kFmtFinished) nxt = (v == a.V - 1) ? kFmtFinished : kFmtDead;
    else if (s < 0 || s > a.L) nxt = kFmtDead;
    else if (v == a.V - 1) nxt = (s == a.L) ? kFmtFinished : kFmtDead;
    else nxt = fmt_allows(a, a.classes, s, v) ? s + int32_t(a.tok_len[v]) : kFmtDead;
    if (nxt == kFmtDead && s != kFmtDead && err) atomicAdd(err, 1);
    states_out[b] = nxt;
}

FmtArgs fmt_args(const uint32_t *classes, int32_t L, const DevVocab &v) {
    FmtArgs a;
    a.classes = classes;
    a.L = L;
    a.tok_off = v.tok_off;
    a.tok_len = v.tok_len;
    a.blob = v.blob;
    a.V = v.V;
    return a;
}

}  // namespace

cudaError_t launch_fmt_compile(const uint32_t *classes, int32_t L, const DevVocab &v, uint32_t *mask, int num_sms,
                               cudaStream_t st) {
    const int64_t W = (int64_t(v.V) + 31) / 32;
    int64_t grid = (W + kFmtThreads / 32 - 1) / (kFmtThreads / 32);
    if (grid > int64_t(num_sms) * 8) grid = int64_t(num_sms) * 8;
    if (grid < 1) grid = 1;
    return launch_pdl(k_fmt_compile, int(grid), kFmtThreads, st, fmt_args(classes, L, v), mask, W);
}

cudaError_t launch_fmt_advance(const uint32_t *classes, int32_t L, const DevVocab &v, const int32_t *states_in,
                               int32_t *states_out, const int32_t *tokens, int32_t B, int32_t *err,
                               cudaStream_t st) {
    const int grid = (B + kFmtThreads - 1) / kFmtThreads;
    return launch_pdl(k_fmt_advance, grid, kFmtThreads, st, fmt_args(classes, L, v), states_in, states_out, tokens, B,
                  err);
}

}  // namespace tmk
