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
// The host packing likewise goes through a static staging buffer, which a call
// rewrites only after the previous call's copy out of it has completed (an
// event recorded after that copy). Only the caller's inputs and output are
// touched besides.
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
std::mutex g_mu;  // serialises use of g_stage and of the per-device state

// Per device, set up by its first call with the device current: the device
// address of g_scratch and an event recorded after each copy out of g_stage.
struct DevState {
    void *scratch = nullptr;
    cudaEvent_t staged = nullptr;
};
DevState g_dev[kMaxDevices];
cudaEvent_t g_pending = nullptr;  // event of the last copy out of g_stage (any device)

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// The host-side name g_scratch is only a stand-in for the symbol, so its
// device address is looked up once per device; the address and the event are
// kept for the life of the process (they do not survive cudaDeviceReset).
int device_state(int dev, DevState **out) {
    if (dev < 0 || dev >= kMaxDevices) return tmk::set_error(TRIE_EINVAL, "device ordinal out of range");
    DevState &d = g_dev[dev];
    if (!d.scratch) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
        if (e != cudaSuccess || !p) {
            cudaGetLastError();
            return tmk::set_error(TRIE_ECUDA, "cudaGetSymbolAddress of the no-alloc scratch failed");
        }
        cudaEvent_t ev = nullptr;
        if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming)) != cudaSuccess) {
            cudaGetLastError();
            return tmk::set_error(TRIE_ECUDA, "creating the no-alloc staging event failed");
        }
        d.scratch = p;
        d.staged = ev;
    }
    *out = &d;
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
    const uint64_t S = tmk::token_table_slots(n_ins);
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
    DevState *ds = nullptr;
    int rc = device_state(dev, &ds);
    if (rc != TRIE_OK) return rc;
    void *dscratch = ds->scratch;

    bool on_device;
    {
        std::lock_guard<std::mutex> hl(h->mu);
        on_device = !h->host_arrays;
    }
    if (on_device && h->dev.device != dev)
        return tmk::set_error(TRIE_EINVAL, "handle was built on another device");
    // the previous call's copy may still be reading g_stage (an asynchronous
    // copy from pageable memory need not have staged it before returning)
    if (g_pending) {
        e = cudaEventSynchronize(g_pending);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return tmk::set_error(TRIE_ECUDA, "waiting for the previous no-alloc copy failed");
        }
        g_pending = nullptr;
    }
    // stage: trie arrays from the handle's host copy; a forest built on the
    // device has none, and its device arrays are copied within the device
    unsigned char *st = g_stage;
    if (!on_device) {
        memcpy(st + o_par, t.parent.data(), 4 * n);
        memcpy(st + o_lab, t.label.data(), n);
        memcpy(st + o_term, t.terminal.data(), n);
    }
    // stage: tokens 16-byte aligned (EOS and byte-less tokens with length 0)
    // and the (length, bytes) -> id table, as trie_compile_masks packs them
    uint32_t *toff = reinterpret_cast<uint32_t *>(st + o_toff);
    uint16_t *tlen = reinterpret_cast<uint16_t *>(st + o_tlen);
    memset(st + o_blob, 0, size_t(blob) + 16);
    tmk::pack_token_bytes(vocab_bytes, vocab_offsets, V, toff, tlen, st + o_blob);
    const bool dup_keys = tmk::fill_token_table(vocab_bytes, vocab_offsets, tlen, V, S,
                                                reinterpret_cast<uint64_t *>(st + o_key),
                                                reinterpret_cast<int32_t *>(st + o_val));
    // one copy into the device scratch, ordered on the caller's stream; the
    // next call waits for its event before it rewrites g_stage
    e = cudaMemcpyAsync(dscratch, g_stage, total, cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return tmk::set_error(TRIE_ECUDA, "copy into the no-alloc scratch failed");
    }
    if ((e = cudaEventRecord(ds->staged, stream)) != cudaSuccess) {
        cudaGetLastError();
        cudaStreamSynchronize(stream);  // no event to wait for: g_stage must be free on return
        cudaGetLastError();
        return tmk::set_error(TRIE_ECUDA, "recording the no-alloc staging event failed");
    }
    g_pending = ds->staged;

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
    dv.dup_keys = dup_keys ? 1 : 0;
    const int64_t W = (int64_t(V) + 31) / 32;
    const int32_t lmax = max_len < t.max_depth ? max_len : t.max_depth;
    e = tmk::launch_mask_fill(d_mask, int64_t(t.n) * W, sms, stream);
    if (e != cudaSuccess) return tmk::set_error(TRIE_ECUDA, "mask fill launch failed");
    e = tmk::launch_mask_patch(dt, t.n, dv, lmax, d_mask, W, sms, stream);
    if (e != cudaSuccess) return tmk::set_error(TRIE_ECUDA, "mask patch launch failed");
    return TRIE_OK;
}
