// trie_compile_masks_noalloc: the mask compile without any device allocation.
//
// trie_compile_masks keeps device copies of the trie and of the packed
// vocabulary in memory it obtains with cudaMalloc. Some callers cannot let a
// library do that: a serving engine that has handed all free HBM to its own
// pool (KV cache) and forbids other allocations, a process whose device memory
// is accounted to a fixed budget, or a latency-critical loop where cudaMalloc /
// cudaFree, which may synchronise the device, must not run. This entry point
// serves them: the trie and vocabulary go into one fixed-size array declared
// in this file (g_scratch, TRIE_NOALLOC_SCRATCH_BYTES), reserved when the
// library's module is loaded on a device and held until the process exits.
// The host packing likewise goes through a static staging buffer. Only the
// caller's inputs and output are touched besides.
#include <stdint.h>
#include <string.h>

#include <mutex>

#include <cuda_runtime.h>

#include "../../include/triemask.h"
#include "tm_internal.h"

namespace {

// The device scratch: trie arrays and the packed vocabulary of the current
// call. Shared by every call on a device; holds the last call's contents.
__device__ __align__(256) unsigned char g_scratch[TRIE_NOALLOC_SCRATCH_BYTES];

// Host staging area with the same layout, copied to g_scratch in one go.
alignas(256) unsigned char g_stage[TRIE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;                          // serialises use of g_stage and g_dev_ptr
void *g_dev_ptr[kMaxDevices] = {nullptr};  // device address of g_scratch per device

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// Device address of g_scratch on `dev` (the current device). The host-side
// name g_scratch is only a stand-in for the symbol, so the address is looked
// up once per device with that device current.
int scratch_ptr(int dev, void **out) {
    if (dev < 0 || dev >= kMaxDevices) return tmk::set_error(TRIE_EINVAL, "device ordinal out of range");
    if (!g_dev_ptr[dev]) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
        if (e != cudaSuccess || !p) {
            cudaGetLastError();
            return tmk::set_error(TRIE_ECUDA, "cudaGetSymbolAddress of the no-alloc scratch failed");
        }
        g_dev_ptr[dev] = p;
    }
    *out = g_dev_ptr[dev];
    return TRIE_OK;
}

}  // namespace

extern "C" int trie_compile_masks_noalloc(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets,
                                          int32_t V, uint32_t *d_mask, cudaStream_t stream) {
    if (!h) return tmk::set_error(TRIE_EINVAL, "handle is NULL");
    if (!vocab_offsets) return tmk::set_error(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || V > INT32_MAX - 32) return tmk::set_error(TRIE_EINVAL, "V must be in [2, 2^31-32]");
    if (!d_mask) return tmk::set_error(TRIE_EINVAL, "d_mask is NULL");
    if (reinterpret_cast<uintptr_t>(d_mask) & 3u) return tmk::set_error(TRIE_EINVAL, "d_mask must be 4-byte aligned");
    if (vocab_offsets[0] < 0 || vocab_offsets[V] < vocab_offsets[0])
        return tmk::set_error(TRIE_EINVAL, "vocab offsets must be non-negative and non-decreasing");
    if (vocab_offsets[V] > vocab_offsets[0] && !vocab_bytes) return tmk::set_error(TRIE_EINVAL, "vocab_bytes is NULL");

    // sizes: tokens with bytes (EOS = V-1 excluded), blob, hash table
    int64_t n_ins = 0, blob = 0;
    int32_t max_len = 0;
    for (int32_t v = 0; v < V; v++) {
        const int64_t L = vocab_offsets[v + 1] - vocab_offsets[v];
        if (L < 0) return tmk::set_error(TRIE_EINVAL, "vocab offsets must be non-decreasing");
        if (v == V - 1) break;
        if (L > 65535) return tmk::set_error(TRIE_EINVAL, "a token is longer than 65535 bytes");
        if (L > 0) {
            n_ins++;
            blob += (L + 15) / 16 * 16;
            if (L > max_len) max_len = int32_t(L);
        }
    }
    uint64_t S = 16;
    while (S < uint64_t(4 * n_ins)) S <<= 1;
    const tmk::HostTrie &t = h->host;
    const size_t n = size_t(t.n);
    size_t off = 0;
    const size_t o_par = off; off = align256(off + 4 * n);
    const size_t o_lab = off; off = align256(off + n);
    const size_t o_term = off; off = align256(off + n);
    const size_t o_toff = off; off = align256(off + 4 * size_t(V));
    const size_t o_tlen = off; off = align256(off + 2 * size_t(V));
    const size_t o_blob = off; off = align256(off + size_t(blob) + 16);
    const size_t o_key = off; off = align256(off + 8 * size_t(S));
    const size_t o_val = off; off = align256(off + 4 * size_t(S));
    const size_t total = off;
    if (total > TRIE_NOALLOC_SCRATCH_BYTES)
        return tmk::set_error(TRIE_EINVAL, "trie + vocabulary need more than the no-alloc scratch "
                                           "(TRIE_NOALLOC_SCRATCH_BYTES = 32 MiB); use trie_compile_masks");

    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return tmk::set_error(TRIE_ECUDA, "cudaGetDevice failed");
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) sms = 1;

    std::lock_guard<std::mutex> lk(g_mu);
    void *dscratch = nullptr;
    int rc = scratch_ptr(dev, &dscratch);
    if (rc != TRIE_OK) return rc;

    // stage: trie arrays from the handle's host copy; a forest built on the
    // device has none, and its device arrays are copied within the device
    bool on_device;
    {
        std::lock_guard<std::mutex> hl(h->mu);
        on_device = !h->host_arrays;
    }
    if (on_device && h->dev.device != dev)
        return tmk::set_error(TRIE_EINVAL, "handle was built on another device");
    unsigned char *st = g_stage;
    if (!on_device) {
        memcpy(st + o_par, t.parent.data(), 4 * n);
        memcpy(st + o_lab, t.label.data(), n);
        memcpy(st + o_term, t.terminal.data(), n);
    }
    // stage: tokens 16-byte aligned, EOS and byte-less tokens with length 0
    uint32_t *toff = reinterpret_cast<uint32_t *>(st + o_toff);
    uint16_t *tlen = reinterpret_cast<uint16_t *>(st + o_tlen);
    unsigned char *bl = st + o_blob;
    memset(bl, 0, size_t(blob) + 16);
    uint32_t pos = 0;
    for (int32_t v = 0; v < V; v++) {
        const int64_t L = (v == V - 1) ? 0 : vocab_offsets[v + 1] - vocab_offsets[v];
        toff[v] = pos;
        tlen[v] = uint16_t(L);
        if (L > 0) memcpy(bl + pos, vocab_bytes + vocab_offsets[v], size_t(L));
        pos += uint32_t((L + 15) / 16 * 16);
    }
    // stage: (length, bytes) -> id table in aligned slot pairs, load <= 1/4,
    // the same hash and probe order as the kernel's lookups
    uint64_t *key = reinterpret_cast<uint64_t *>(st + o_key);
    int32_t *val = reinterpret_cast<int32_t *>(st + o_val);
    memset(key, 0, 8 * size_t(S));
    memset(val, 0xff, 4 * size_t(S));
    const uint64_t pairs_mask = S / 2 - 1;
    for (int32_t v = 0; v + 1 < V; v++) {
        const uint32_t L = tlen[v];
        if (!L) continue;
        const uint8_t *p = vocab_bytes + vocab_offsets[v];
        uint64_t hsh = 0;
        for (uint32_t j = 0; j < L; j++) hsh = hsh * tmk::kHashBase + uint64_t(p[j]) + 1;
        const uint64_t k = tmk::hash_finish(hsh, L);
        uint64_t pair = (k >> 1) & pairs_mask;
        for (;;) {
            if (!key[2 * pair]) { key[2 * pair] = k; val[2 * pair] = v; break; }
            if (!key[2 * pair + 1]) { key[2 * pair + 1] = k; val[2 * pair + 1] = v; break; }
            pair = (pair + 1) & pairs_mask;
        }
    }
    // one copy into the device scratch, ordered on the caller's stream; from
    // pageable memory it returns once the staging buffer has been read
    e = cudaMemcpyAsync(dscratch, g_stage, total, cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return tmk::set_error(TRIE_ECUDA, "copy into the no-alloc scratch failed");
    }

    unsigned char *d = static_cast<unsigned char *>(dscratch);
    if (on_device && n > 0 &&
        ((e = cudaMemcpyAsync(d + o_par, h->dev.parent, 4 * n, cudaMemcpyDeviceToDevice, stream)) != cudaSuccess ||
         (e = cudaMemcpyAsync(d + o_lab, h->dev.label, n, cudaMemcpyDeviceToDevice, stream)) != cudaSuccess ||
         (e = cudaMemcpyAsync(d + o_term, h->dev.terminal, n, cudaMemcpyDeviceToDevice, stream)) != cudaSuccess)) {
        cudaGetLastError();
        return tmk::set_error(TRIE_ECUDA, "copy of the device-built trie into the no-alloc scratch failed");
    }
    tmk::DevTrie dt;
    dt.device = dev;
    dt.parent = reinterpret_cast<const int32_t *>(d + o_par);
    dt.label = d + o_lab;
    dt.terminal = d + o_term;
    tmk::DevVocab dv;  // a view: base stays null, so nothing is freed
    dv.device = dev;
    dv.V = V;
    dv.max_len = max_len;
    dv.ht_mask = uint32_t(S - 1);
    dv.tok_off = reinterpret_cast<const uint32_t *>(d + o_toff);
    dv.tok_len = reinterpret_cast<const uint16_t *>(d + o_tlen);
    dv.blob = d + o_blob;
    dv.ht_key = reinterpret_cast<const uint64_t *>(d + o_key);
    dv.ht_val = reinterpret_cast<const int32_t *>(d + o_val);
    const int64_t W = (int64_t(V) + 31) / 32;
    const int32_t lmax = max_len < t.max_depth ? max_len : t.max_depth;
    e = tmk::launch_mask_fill(d_mask, int64_t(t.n) * W, sms, stream);
    if (e != cudaSuccess) return tmk::set_error(TRIE_ECUDA, "mask fill launch failed");
    e = tmk::launch_mask_patch(dt, t.n, dv, lmax, d_mask, W, sms, stream);
    if (e != cudaSuccess) return tmk::set_error(TRIE_ECUDA, "mask patch launch failed");
    return TRIE_OK;
}
