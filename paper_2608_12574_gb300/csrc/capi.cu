// C ABI of libtriemask (declared in include/triemask.h): argument checks,
// handle and device-memory management, the per-device vocabulary cache, and
// the kernel launches.
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <cstdlib>
#include <memory>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/triemask.h"
#include "tm_internal.h"

namespace {

thread_local std::string g_last_error;

int fail(int code, const std::string &msg) {
    g_last_error = msg;
    return code;
}

int fail_cuda(cudaError_t e, const char *what) {
    return fail(TRIE_ECUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

// Restores the caller's current device on scope exit.
struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

int num_sms(int dev) {
    static std::mutex mu;
    static std::vector<int> cache;
    std::lock_guard<std::mutex> lk(mu);
    if (int(cache.size()) <= dev) cache.resize(size_t(dev) + 1, 0);
    if (!cache[size_t(dev)]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
        cache[size_t(dev)] = n;
    }
    return cache[size_t(dev)];
}

// Carves 256-byte aligned sub-arrays out of one device allocation.
struct Layout {
    size_t total = 0;
    size_t add(size_t bytes) {
        size_t off = total;
        total += (bytes + 255) / 256 * 256;
        return off;
    }
};

// Per-handle device memory (the trie's arrays, the valid lists, the lazy
// rows) and the scratch of device builds come from one memory pool per
// device, owned by the library and kept until exit. Up to kPoolKeepBytes of
// freed memory stays mapped for the next allocations, so a loop that builds,
// uses and destroys a forest for every batch does not map and unmap device
// memory each time. A freed block is reused only once its free has completed
// on the device, so an allocation carries no stream dependency.
constexpr uint64_t kPoolKeepBytes = uint64_t(8) << 30;

int pool_alloc(int dev, size_t bytes, cudaStream_t stream, void **out, const char *what) {
    *out = nullptr;
    cudaMemPool_t pool = tmk::device_pool(dev);
    if (!pool) return fail(TRIE_ECUDA, std::string("creating the device memory pool for ") + what);
    cudaError_t e = cudaMallocFromPoolAsync(out, std::max<size_t>(bytes, 1), pool, stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        *out = nullptr;
        return fail(TRIE_ENOMEM, std::string("device allocation for ") + what + ": " + cudaGetErrorString(e));
    }
    return TRIE_OK;
}

// Frees a pool block once no device work can still use it: waits for the
// current device (the block's device must be current).
void pool_free(void *p) {
    if (!p) return;
    cudaDeviceSynchronize();
    cudaFreeAsync(p, 0);
    cudaGetLastError();
}

std::mutex g_vocab_mu;
// Most recent last. Never destroyed, so no device memory is freed during
// static destruction at process exit (the CUDA runtime may be gone by then).
std::vector<std::shared_ptr<tmk::DevVocab>> &g_vocabs = *new std::vector<std::shared_ptr<tmk::DevVocab>>();
constexpr size_t kVocabCacheSize = 4;

int get_vocab(const uint8_t *vb, const int64_t *vo, int32_t V, int dev,
              std::shared_ptr<tmk::DevVocab> *out) {
    const int64_t b0 = vo[0], b1 = vo[V];
    if (b0 < 0 || b1 < b0) return fail(TRIE_EINVAL, "vocab offsets must be non-negative and non-decreasing");
    const size_t nbytes = size_t(b1 - b0);
    if (nbytes && !vb) return fail(TRIE_EINVAL, "vocab_bytes is NULL");
    std::lock_guard<std::mutex> lk(g_vocab_mu);
    for (size_t i = 0; i < g_vocabs.size(); i++) {
        auto &c = g_vocabs[i];
        if (c->device == dev && c->V == V && c->src_bytes.size() == nbytes &&
            memcmp(c->src_offsets.data(), vo, sizeof(int64_t) * (size_t(V) + 1)) == 0 &&
            (nbytes == 0 || memcmp(c->src_bytes.data(), vb + b0, nbytes) == 0)) {
            *out = c;
            std::rotate(g_vocabs.begin() + long(i), g_vocabs.begin() + long(i) + 1, g_vocabs.end());
            return TRIE_OK;
        }
    }
    tmk::HostVocab hv;
    std::string err;
    try {
        err = tmk::pack_vocab(vb, vo, V, &hv);
    } catch (const std::bad_alloc &) {
        return fail(TRIE_ENOMEM, "host allocation failed while packing the vocabulary");
    }
    if (!err.empty()) return fail(TRIE_EINVAL, err);
    auto dv = std::make_shared<tmk::DevVocab>();
    dv->device = dev;
    dv->V = V;
    dv->max_len = hv.max_len;
    dv->ht_mask = hv.ht_mask;
    Layout L;
    const size_t o_off = L.add(sizeof(uint32_t) * hv.tok_off.size());
    const size_t o_len = L.add(sizeof(uint16_t) * hv.tok_len.size());
    const size_t o_blob = L.add(hv.blob.size());
    const size_t o_key = L.add(sizeof(uint64_t) * hv.ht_key.size());
    const size_t o_val = L.add(sizeof(int32_t) * hv.ht_val.size());
    // the probe's per-slot payload (blob offsets / 16 must fit in 27 bits)
    const bool with_pay = !hv.dup_keys && hv.blob.size() < (size_t(1) << 31);
    const size_t o_pay = with_pay ? L.add(sizeof(uint4) * hv.ht_key.size()) : 0;
    cudaError_t e = cudaMalloc(&dv->base, L.total);
    if (e != cudaSuccess) {
        dv->base = nullptr;
        cudaGetLastError();
        return fail(TRIE_ENOMEM, std::string("cudaMalloc for the vocabulary: ") + cudaGetErrorString(e));
    }
    char *base = static_cast<char *>(dv->base);
    struct Up { size_t off; const void *src; size_t n; } ups[] = {
        {o_off, hv.tok_off.data(), sizeof(uint32_t) * hv.tok_off.size()},
        {o_len, hv.tok_len.data(), sizeof(uint16_t) * hv.tok_len.size()},
        {o_blob, hv.blob.data(), hv.blob.size()},
        {o_key, hv.ht_key.data(), sizeof(uint64_t) * hv.ht_key.size()},
        {o_val, hv.ht_val.data(), sizeof(int32_t) * hv.ht_val.size()},
    };
    for (const Up &u : ups) {
        e = cudaMemcpy(base + u.off, u.src, u.n, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return fail_cuda(e, "uploading the vocabulary");
    }
    dv->tok_off = reinterpret_cast<const uint32_t *>(base + o_off);
    dv->tok_len = reinterpret_cast<const uint16_t *>(base + o_len);
    dv->blob = reinterpret_cast<const uint8_t *>(base + o_blob);
    dv->blob_bytes = hv.blob.size();
    dv->dup_keys = hv.dup_keys;
    dv->ht_key = reinterpret_cast<const uint64_t *>(base + o_key);
    dv->ht_val = reinterpret_cast<const int32_t *>(base + o_val);
    if (with_pay) {
        uint4 *pay = reinterpret_cast<uint4 *>(base + o_pay);
        if ((e = tmk::launch_vocab_pay(*dv, pay, num_sms(dev), 0)) != cudaSuccess ||
            (e = cudaStreamSynchronize(0)) != cudaSuccess)
            return fail_cuda(e, "building the token table's payload");
        dv->ht_pay = pay;
    }
    try {
        dv->src_offsets.assign(vo, vo + V + 1);
        dv->src_bytes.assign(vb ? vb + b0 : nullptr, vb ? vb + b1 : nullptr);
    } catch (const std::bad_alloc &) {
        return fail(TRIE_ENOMEM, "host allocation failed while caching the vocabulary");
    }
    g_vocabs.push_back(dv);
    if (g_vocabs.size() > kVocabCacheSize) g_vocabs.erase(g_vocabs.begin());
    *out = dv;
    return TRIE_OK;
}

// Uploads the trie on first use, ordered on `stream` (the copies read the
// handle's own host arrays, which outlive them); the handle is bound to that
// device.
// Device arrays of a trie of n nodes (one allocation); nothing is uploaded.
// with_trans: also a transition table (8 or more slots per node) for the
// compiles to record moves in.
int alloc_device_trie(trie_t h, int dev, size_t n, cudaStream_t stream, bool with_trans) {
    Layout L;
    const size_t o_par = L.add(sizeof(int32_t) * n);
    const size_t o_lab = L.add(n);
    const size_t o_term = L.add(n);
    const size_t o_fc = L.add(sizeof(int32_t) * n);
    const size_t o_bits = L.add(sizeof(uint32_t) * 8 * n);
    const size_t o_win = L.add(sizeof(uint64_t) * 2 * n);
    const size_t o_d16 = L.add(n);
    const size_t o_anc = L.add(sizeof(int32_t) * 16 * n);
    size_t trans_slots = with_trans ? 16 : 0;  // >= 8 per node, a power of two
    while (with_trans && trans_slots < 8 * n) trans_slots <<= 1;
    const size_t o_trans = L.add(sizeof(ulonglong2) * trans_slots);
    void *base = nullptr;
    const int rc = pool_alloc(dev, L.total, stream, &base, "the trie");
    if (rc != TRIE_OK) return rc;
    char *b = static_cast<char *>(base);
    h->dev.device = dev;
    h->dev.base = base;
    h->dev.parent = reinterpret_cast<const int32_t *>(b + o_par);
    h->dev.label = reinterpret_cast<const uint8_t *>(b + o_lab);
    h->dev.terminal = reinterpret_cast<const uint8_t *>(b + o_term);
    h->dev.first_child = reinterpret_cast<int32_t *>(b + o_fc);
    h->dev.child_bits = reinterpret_cast<uint32_t *>(b + o_bits);
    h->dev.window = reinterpret_cast<ulonglong2 *>(b + o_win);
    h->dev.depth16 = reinterpret_cast<uint8_t *>(b + o_d16);
    h->dev.anc = reinterpret_cast<int4 *>(b + o_anc);
    h->dev.trans = with_trans ? reinterpret_cast<ulonglong2 *>(b + o_trans) : nullptr;
    h->dev.trans_mask = with_trans ? uint32_t(trans_slots - 1) : 0u;
    return TRIE_OK;
}

// The child links and the compile's per-node tables, from the device's
// parent / label / terminal arrays (once they are written on `stream`).
int finish_device_trie(trie_t h, int dev, cudaStream_t stream) {
    cudaError_t e;
    if ((e = tmk::launch_trie_links(h->dev, h->host.n, num_sms(dev), stream)) == cudaSuccess)
        e = tmk::launch_trie_tables(h->dev, h->host.n, num_sms(dev), stream);
    if (e != cudaSuccess) {
        pool_free(h->dev.base);
        h->dev = tmk::DevTrie();
        return fail_cuda(e, "building the trie's compile tables");
    }
    return TRIE_OK;
}

bool host_memory_direct(int dev);

int ensure_device_trie(trie_t h, int dev, cudaStream_t stream) {
    std::lock_guard<std::mutex> lk(h->mu);
    if (h->dev.base) {
        if (h->dev.device != dev)
            return fail(TRIE_EINVAL, "handle was uploaded to device " + std::to_string(h->dev.device) +
                                         ", called on device " + std::to_string(dev));
        return TRIE_OK;
    }
    const tmk::HostTrie &t = h->host;
    const size_t n = size_t(t.n);
    // a transition table for a single trie; a forest's per-request sets are
    // decoded for a few steps, where byte walks cost less than the table
    int rc = alloc_device_trie(h, dev, n, stream, t.roots.size() <= 1);
    if (rc != TRIE_OK) return rc;
    if (host_memory_direct(dev)) {
        // the kernel reads the handle's host arrays itself: a pageable copy
        // would wait on the host for the stream and for the copy engines
        cudaError_t e = tmk::launch_copy3(const_cast<int32_t *>(h->dev.parent), t.parent.data(),
                                          int64_t(sizeof(int32_t) * n), const_cast<uint8_t *>(h->dev.label),
                                          t.label.data(), int64_t(n), const_cast<uint8_t *>(h->dev.terminal),
                                          t.terminal.data(), int64_t(n), num_sms(dev), stream);
        if (e != cudaSuccess) {
            pool_free(h->dev.base);
            h->dev = tmk::DevTrie();
            return fail_cuda(e, "uploading the trie");
        }
        return finish_device_trie(h, dev, stream);
    }
    struct Up { const void *dst; const void *src; size_t n; } ups[] = {
        {h->dev.parent, t.parent.data(), sizeof(int32_t) * n},
        {h->dev.label, t.label.data(), n},
        {h->dev.terminal, t.terminal.data(), n},
    };
    for (const Up &u : ups) {
        cudaError_t e = cudaMemcpyAsync(const_cast<void *>(u.dst), u.src, u.n, cudaMemcpyHostToDevice, stream);
        if (e != cudaSuccess) {
            pool_free(h->dev.base);
            h->dev = tmk::DevTrie();
            return fail_cuda(e, "uploading the trie");
        }
    }
    return finish_device_trie(h, dev, stream);
}

// The transition table holds transitions of one vocabulary: when a compile
// uses another, clear it and let this compile's probe refill it; when it
// holds only the entries lazy rows added, let the compile complete it.
int prepare_trans(trie_t h, const std::shared_ptr<tmk::DevVocab> &voc, int sms, cudaStream_t stream, bool *fill) {
    std::lock_guard<std::mutex> lk(h->mu);
    *fill = false;
    if (!h->dev.trans) return TRIE_OK;
    if (h->trans_vocab == voc) {
        *fill = !h->trans_complete;
        return TRIE_OK;
    }
    h->trans_vocab.reset();
    h->trans_complete = false;
    cudaError_t e = tmk::launch_trans_clear(h->dev, sms, stream);
    if (e != cudaSuccess) return fail_cuda(e, "transition table clear");
    *fill = true;
    return TRIE_OK;
}

// Whether kernels on dev may read the caller's pageable host memory directly
// (coherent access through the host's page tables, as on Grace systems over
// NVLink-C2C). TRIEMASK_HOST_READ=copy in the environment forces the copy
// path instead.
bool host_memory_direct(int dev) {
    static std::mutex mu;
    static std::vector<int> cache;  // 0 unknown, 1 direct, 2 copy
    std::lock_guard<std::mutex> lk(mu);
    if (int(cache.size()) <= dev) cache.resize(size_t(dev) + 1, 0);
    if (!cache[size_t(dev)]) {
        int pageable = 0, host_tables = 0;
        const char *env = getenv("TRIEMASK_HOST_READ");
        const bool forced_copy = env && strcmp(env, "copy") == 0;
        if (cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&host_tables, cudaDevAttrPageableMemoryAccessUsesHostPageTables, dev) !=
                cudaSuccess) {
            cudaGetLastError();
            pageable = 0;
        }
        cache[size_t(dev)] = (!forced_copy && pageable == 1 && host_tables == 1) ? 1 : 2;
    }
    return cache[size_t(dev)] == 1;
}

int current_device(int *dev) {
    cudaError_t e = cudaGetDevice(dev);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail_cuda(e, "cudaGetDevice");
    }
    return TRIE_OK;
}

int finish_build(std::string err, trie_s *h, trie_t *out) {
    if (!err.empty()) {
        delete h;
        return fail(err.find("exceed") != std::string::npos ? TRIE_ENOMEM : TRIE_EINVAL, err);
    }
    *out = h;
    return TRIE_OK;
}

// Shared checks and the launch of the three lazy-row calls.
int lazy_call(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out, int32_t *d_err,
              void *d_logits, int dtype, uint32_t *d_rows, int32_t B, int32_t V, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    const tmk::DevLazy &L = h->lazy;
    if (!L.base) return fail(TRIE_ESTATE, "lazy call before trie_lazy_init on this handle");
    if (B < 0 || B > L.max_batch)
        return fail(TRIE_EINVAL, "B must be in [0, max_batch = " + std::to_string(L.max_batch) + "]");
    if (V != L.V) return fail(TRIE_EINVAL, "V differs from the V given to trie_lazy_init");
    if (B == 0) return TRIE_OK;
    if (!d_states_in) return fail(TRIE_EINVAL, "d_states is NULL");
    if (d_tokens && (!d_states_out || d_states_out == d_states_in))
        return fail(TRIE_EINVAL, "d_states_out must be a buffer other than d_states_in");
    if (d_logits) {
        if (dtype != TRIE_DTYPE_F32 && dtype != TRIE_DTYPE_BF16) return fail(TRIE_EINVAL, "unknown dtype");
        if (reinterpret_cast<uintptr_t>(d_logits) & uintptr_t(dtype == TRIE_DTYPE_F32 ? 3 : 1))
            return fail(TRIE_EINVAL, "d_logits is not aligned to its element size");
    }
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != L.device || dev != h->dev.device) return fail(TRIE_EINVAL, "handle belongs to another device");
    bool use_trans, fill_trans;
    {
        std::lock_guard<std::mutex> lk(h->mu);
        use_trans = h->trans_vocab == L.vocab;
        fill_trans = use_trans && !h->trans_complete;  // record the moves the rows find
    }
    const int32_t lmax = std::min(L.vocab->max_len, h->host.max_depth);
    cudaError_t e = tmk::launch_lazy(h->dev, h->host.n, *L.vocab, use_trans, fill_trans, lmax, L, d_states_in, d_tokens,
                                     d_states_out, d_err, B, d_logits, dtype, d_rows, num_sms(dev), stream);
    if (e != cudaSuccess) return fail_cuda(e, "lazy-row launch");
    return TRIE_OK;
}

}  // namespace

int tmk::set_error(int code, const char *msg) { return fail(code, msg); }

cudaMemPool_t tmk::device_pool(int dev) {
    static std::mutex mu;
    static std::vector<cudaMemPool_t> &pools = *new std::vector<cudaMemPool_t>();  // never destroyed
    std::lock_guard<std::mutex> lk(mu);
    if (dev < 0) return nullptr;
    if (int(pools.size()) <= dev) pools.resize(size_t(dev) + 1, nullptr);
    if (!pools[size_t(dev)]) {
        cudaMemPoolProps props = {};
        props.allocType = cudaMemAllocationTypePinned;
        props.handleTypes = cudaMemHandleTypeNone;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        cudaMemPool_t p = nullptr;
        if (cudaMemPoolCreate(&p, &props) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        uint64_t keep = kPoolKeepBytes;
        int no = 0;
        if (cudaMemPoolSetAttribute(p, cudaMemPoolAttrReleaseThreshold, &keep) != cudaSuccess ||
            cudaMemPoolSetAttribute(p, cudaMemPoolReuseFollowEventDependencies, &no) != cudaSuccess ||
            cudaMemPoolSetAttribute(p, cudaMemPoolReuseAllowInternalDependencies, &no) != cudaSuccess) {
            cudaGetLastError();
            cudaMemPoolDestroy(p);
            return nullptr;
        }
        pools[size_t(dev)] = p;
    }
    return pools[size_t(dev)];
}

int tmk::ensure_host_arrays(trie_s *h) {
    std::lock_guard<std::mutex> lk(h->mu);
    if (h->host_arrays) return TRIE_OK;
    {  // the build's last kernels may still be queued (on the caller's stream)
        DeviceGuard g(h->dev.device);
        const cudaError_t e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return fail_cuda(e, "waiting for the forest build");
    }
    tmk::HostTrie &t = h->host;
    const size_t n = size_t(t.n);
    try {
        t.parent.resize(n);
        t.label.resize(n);
        t.terminal.resize(n);
    } catch (const std::bad_alloc &) {
        return fail(TRIE_ENOMEM, "host allocation failed while copying the trie back");
    }
    DeviceGuard g(h->dev.device);
    cudaError_t e;
    if ((e = cudaDeviceSynchronize()) != cudaSuccess ||
        (e = cudaMemcpy(t.parent.data(), h->dev.parent, sizeof(int32_t) * n, cudaMemcpyDeviceToHost)) !=
            cudaSuccess ||
        (e = cudaMemcpy(t.label.data(), h->dev.label, n, cudaMemcpyDeviceToHost)) != cudaSuccess ||
        (e = cudaMemcpy(t.terminal.data(), h->dev.terminal, n, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return fail_cuda(e, "copying the trie back from the device");
    try {
        tmk::pre_order_from_parents(&t);
    } catch (const std::bad_alloc &) {
        return fail(TRIE_ENOMEM, "host allocation failed for the pre-order tables");
    }
    h->host_arrays = true;
    return TRIE_OK;
}

tmk::DevVocab::~DevVocab() {
    if (base || rt_base) {
        DeviceGuard g(device);
        if (base) cudaFree(base);
        if (rt_base) cudaFree(rt_base);
    }
}

extern "C" {

const char *trie_last_error(void) { return g_last_error.c_str(); }

static void sweep_retired();

int trie_build(const uint8_t *bytes, const int64_t *offsets, int32_t K, trie_t *out) {
    sweep_retired();
    if (!out) return fail(TRIE_EINVAL, "out is NULL");
    *out = nullptr;
    if (K < 0) return fail(TRIE_EINVAL, "K must be >= 0");
    if (K > 0 && !offsets) return fail(TRIE_EINVAL, "offsets is NULL");
    if (K > 0 && offsets[K] > offsets[0] && !bytes) return fail(TRIE_EINVAL, "bytes is NULL");
    trie_s *h = new (std::nothrow) trie_s;
    if (!h) return fail(TRIE_ENOMEM, "host allocation failed");
    std::string err;
    try {
        static const int64_t zero = 0;
        err = tmk::build_trie(bytes, K > 0 ? offsets : &zero, 0, K, &h->host);
    } catch (const std::bad_alloc &) {
        delete h;
        return fail(TRIE_ENOMEM, "host allocation failed while building the trie");
    }
    return finish_build(err, h, out);
}

int trie_build_many(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets,
                    int32_t M, trie_t *out) {
    sweep_retired();
    if (!out) return fail(TRIE_EINVAL, "out is NULL");
    *out = nullptr;
    if (M < 1) return fail(TRIE_EINVAL, "M must be >= 1");
    if (!set_offsets) return fail(TRIE_EINVAL, "set_offsets is NULL");
    if (set_offsets[0] != 0) return fail(TRIE_EINVAL, "set_offsets[0] must be 0");
    for (int32_t i = 0; i < M; i++)
        if (set_offsets[i + 1] < set_offsets[i]) return fail(TRIE_EINVAL, "set_offsets must be non-decreasing");
    const int32_t K = set_offsets[M];
    if (K > 0 && !offsets) return fail(TRIE_EINVAL, "offsets is NULL");
    if (K > 0 && offsets[K] > offsets[0] && !bytes) return fail(TRIE_EINVAL, "bytes is NULL");
    trie_s *h = new (std::nothrow) trie_s;
    if (!h) return fail(TRIE_ENOMEM, "host allocation failed");
    std::string err;
    try {
        static const int64_t zero = 0;
        err = tmk::build_forest(bytes, K > 0 ? offsets : &zero, set_offsets, M, &h->host);
    } catch (const std::bad_alloc &) {
        delete h;
        return fail(TRIE_ENOMEM, "host allocation failed while building the forest");
    }
    return finish_build(err, h, out);
}

int trie_build_many_device(const uint8_t *bytes, const int64_t *offsets, const int32_t *set_offsets, int32_t M,
                           cudaStream_t stream, trie_t *out) {
    sweep_retired();
    if (!out) return fail(TRIE_EINVAL, "out is NULL");
    *out = nullptr;
    if (M < 1) return fail(TRIE_EINVAL, "M must be >= 1");
    if (!set_offsets) return fail(TRIE_EINVAL, "set_offsets is NULL");
    if (set_offsets[0] != 0) return fail(TRIE_EINVAL, "set_offsets[0] must be 0");
    for (int32_t i = 0; i < M; i++)
        if (set_offsets[i + 1] < set_offsets[i]) return fail(TRIE_EINVAL, "set_offsets must be non-decreasing");
    const int32_t K = set_offsets[M];
    if (K > 0 && !offsets) return fail(TRIE_EINVAL, "offsets is NULL");
    static const int64_t zero = 0;
    const int64_t *off = K > 0 ? offsets : &zero;
    if (off[0] < 0 || off[K] < off[0]) return fail(TRIE_EINVAL, "offsets must be non-negative and non-decreasing");
    const int64_t n_bytes = off[K] - off[0];
    if (n_bytes > 0 && !bytes) return fail(TRIE_EINVAL, "bytes is NULL");
    if (n_bytes + M > int64_t(INT32_MAX) - 2)  // more bytes than node ids: the host builder decides
        return trie_build_many(bytes, offsets, set_offsets, M, out);
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    cudaMemPool_t pool = tmk::device_pool(dev);
    if (!pool) return fail(TRIE_ECUDA, "creating the device memory pool for the forest build");
    const int sms = num_sms(dev);
    trie_s *h = new (std::nothrow) trie_s;
    if (!h) return fail(TRIE_ENOMEM, "host allocation failed");
    int32_t n = 0, max_len = 0;
    int64_t n_chars = 0;
    cudaError_t e;
    {
        tmk::DeviceBuild db;
        bool ok = true;
        e = db.stage(n_bytes > 0 ? bytes + off[0] : nullptr, off, set_offsets, M, K, n_bytes,
                     host_memory_direct(dev), sms, pool, stream, &max_len, &ok);
        if (e == cudaSuccess && !ok) {
            delete h;
            return fail(TRIE_EINVAL, "offsets must be non-negative and non-decreasing");
        }
        // long strings (a long level loop) or many sets with deep strings
        // (the per-(set, depth) tables): the host builder
        if (e == cudaSuccess &&
            (max_len > tmk::kDeviceBuildMaxDepth || int64_t(M) * (max_len + 1) > tmk::kDeviceBuildMaxGroups)) {
            delete h;
            return trie_build_many(bytes, offsets, set_offsets, M, out);
        }
        if (e == cudaSuccess) e = db.levels(max_len, sms, &n, &h->host.roots, &n_chars);
        if (e == cudaSuccess) {
            h->host.n = n;
            h->host.n_chars = n_chars;
            h->host.max_depth = max_len;
            h->host_arrays = false;
            // per-batch sets are decoded for a few steps: no transition
            // table to clear and fill (advance walks the tokens' bytes)
            if ((rc = alloc_device_trie(h, dev, size_t(n), stream, false)) != TRIE_OK) {
                delete h;
                return rc;
            }
            e = db.emit(const_cast<int32_t *>(h->dev.parent), const_cast<uint8_t *>(h->dev.label),
                        const_cast<uint8_t *>(h->dev.terminal), sms);
        }
    }  // the scratch is freed on the stream after the last kernel
    if (e == cudaSuccess && (rc = finish_device_trie(h, dev, stream)) != TRIE_OK) {
        delete h;
        return rc;
    }
    // no synchronisation here: the node count and roots are on the host, the
    // caller's arrays have been read, and the last kernels (breadth-first
    // layout, child links, per-node tables) finish on `stream` while the host
    // goes on (a later call on `stream` is ordered after them)
    if (e != cudaSuccess) {
        cudaGetLastError();
        pool_free(h->dev.base);
        delete h;
        if (e == cudaErrorMemoryAllocation)
            return fail(TRIE_ENOMEM, "device allocation failed while building the forest");
        return fail_cuda(e, "building the forest on the device");
    }
    *out = h;
    return TRIE_OK;
}

int32_t trie_num_nodes(trie_t h) { return h ? h->host.n : -1; }

int32_t trie_num_sets(trie_t h) { return h ? int32_t(h->host.roots.size()) : -1; }

int32_t trie_root(trie_t h, int32_t i) {
    if (!h || i < 0 || i >= int32_t(h->host.roots.size())) return -1;
    return h->host.roots[size_t(i)];
}

int trie_copy_roots(trie_t h, int32_t *roots) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (!roots && !h->host.roots.empty()) return fail(TRIE_EINVAL, "roots is NULL");
    std::copy(h->host.roots.begin(), h->host.roots.end(), roots);
    return TRIE_OK;
}

int64_t trie_num_chars(trie_t h) { return h ? h->host.n_chars : -1; }

int32_t trie_max_depth(trie_t h) { return h ? h->host.max_depth : -1; }

int trie_get_csr(trie_t h, int32_t *parent, uint8_t *label, uint8_t *terminal, int32_t *first_child) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    int rc = tmk::ensure_host_arrays(h);
    if (rc != TRIE_OK) return rc;
    const size_t n = size_t(h->host.n);
    if (parent) memcpy(parent, h->host.parent.data(), sizeof(int32_t) * n);
    if (label) memcpy(label, h->host.label.data(), n);
    if (terminal) memcpy(terminal, h->host.terminal.data(), n);
    if (first_child) {  // children are contiguous: the first is the smallest id with that parent
        for (size_t i = 0; i < n; i++) first_child[i] = -1;
        for (size_t c = n; c-- > 1;)
            if (h->host.parent[c] >= 0) first_child[size_t(h->host.parent[c])] = int32_t(c);
    }
    return TRIE_OK;
}

// The dense compile's hit buffer (the probe's records for the scatter), on
// the first dense compile of the handle: the valid lists and the lazy rows
// never need it, so a forest compiled to lists does not hold 129 B per node.
static int ensure_hits(trie_t h, int dev, cudaStream_t stream) {
    std::lock_guard<std::mutex> lk(h->mu);
    if (h->dev.hits_base) return TRIE_OK;
    const size_t n = size_t(h->host.n);
    Layout L;
    const size_t o_hits = L.add(sizeof(int2) * tmk::kHitSlots * n);
    const size_t o_hcnt = L.add(n);
    void *base = nullptr;
    const int rc = pool_alloc(dev, L.total, stream, &base, "the compile's hit buffer");
    if (rc != TRIE_OK) return rc;
    char *b = static_cast<char *>(base);
    h->dev.hits_base = base;
    h->dev.hits = reinterpret_cast<int2 *>(b + o_hits);
    h->dev.hit_count = reinterpret_cast<uint8_t *>(b + o_hcnt);
    return TRIE_OK;
}

// The segment summary of the dense mask (bit g of row r set iff the row allows
// a token of the 1,024-token segment g), which lets the apply skip reading
// the mask words of empty segments; none when it would exceed 256 MB, and
// none for tries of more than kSegMaxNodes nodes: the probe sets the summary
// while the fill runs, and for a forest of millions of nodes its
// compare-and-swaps made it outlast the fill (dense compile of the 4.77 M-node
// forest 12.9 ms with the summary, 11.1 ms without).
constexpr int32_t kSegMaxNodes = int32_t(1) << 18;
static unsigned long long *ensure_seg(trie_t h, int dev, cudaStream_t stream, int32_t words) {
    const int64_t need = int64_t(h->host.n) * words;
    if (need * 8 > (int64_t(256) << 20)) return nullptr;
    std::lock_guard<std::mutex> lk(h->mu);
    if (h->dev.seg_cap < need) {
        pool_free(h->dev.seg_epoch);  // an earlier apply may still read it
        h->dev.seg_any = nullptr;
        h->dev.seg_epoch = nullptr;
        h->dev.seg_cap = 0;
        void *p = nullptr;
        const size_t bytes = 16 + size_t(need) * 8;  // the epoch word, then the summary words
        if (pool_alloc(dev, bytes, stream, &p, "the mask's segment summary") != TRIE_OK) {
            cudaGetLastError();
            return nullptr;  // the compile and the apply work without it
        }
        // epoch 0 is never a compile's: every word starts out empty
        if (cudaMemsetAsync(p, 0, bytes, stream) != cudaSuccess) {
            cudaGetLastError();
            pool_free(p);
            return nullptr;
        }
        h->dev.seg_epoch = static_cast<uint32_t *>(p);
        h->dev.seg_any = reinterpret_cast<unsigned long long *>(static_cast<char *>(p) + 16);
        h->dev.seg_cap = need;
    }
    return h->dev.seg_any;
}

// The mask compile with the vocabulary resolved (from the cache, or a vocabulary handle).
static int compile_masks(trie_t h, const std::shared_ptr<tmk::DevVocab> &voc, int dev, uint32_t *d_mask,
                         cudaStream_t stream) {
    int rc;
    const int32_t V = voc->V;
    if ((rc = ensure_device_trie(h, dev, stream)) != TRIE_OK) return rc;
    if ((rc = ensure_hits(h, dev, stream)) != TRIE_OK) return rc;
    const int64_t W = (int64_t(V) + 31) / 32;
    const int32_t n = h->host.n;
    const int32_t lmax = std::min(voc->max_len, h->host.max_depth);
    const int sms = num_sms(dev);
    bool fill_trans;
    if ((rc = prepare_trans(h, voc, sms, stream, &fill_trans)) != TRIE_OK) return rc;
    const int32_t seg_words = int32_t(((W + 31) / 32 + 31) / 32);
    unsigned long long *seg = n <= kSegMaxNodes ? ensure_seg(h, dev, stream, seg_words) : nullptr;
    const uint32_t epoch = h->dev.seg_epoch_next;
    h->dev.seg_epoch_next = epoch == UINT32_MAX ? 1u : epoch + 1u;
    bool seg_written = false;
    cudaError_t e = tmk::launch_mask_compile3(h->dev, n, *voc, lmax, d_mask, W, sms, fill_trans, stream, seg,
                                              h->dev.seg_epoch, epoch, seg_words, &seg_written);
    if (e != cudaSuccess) return fail_cuda(e, "mask compile launch");
    std::lock_guard<std::mutex> lk(h->mu);
    h->trans_vocab = voc;
    h->trans_complete = h->trans_complete || fill_trans;
    h->vocab = voc;
    h->mask = d_mask;
    h->mask_V = V;
    h->mask_seg = tmk::SegRef();
    if (seg_written) {
        h->mask_seg.words = seg;
        h->mask_seg.epoch = h->dev.seg_epoch;
        h->mask_seg.per_row = seg_words;
    }
    return TRIE_OK;
}

static int check_mask_arg(uint32_t *d_mask) {
    if (!d_mask) return fail(TRIE_EINVAL, "d_mask is NULL");
    if (reinterpret_cast<uintptr_t>(d_mask) & 3u) return fail(TRIE_EINVAL, "d_mask must be 4-byte aligned");
    return TRIE_OK;
}

// The vocabulary of a handle, on the current device.
static int vocab_of(trie_vocab_t v, int *dev, std::shared_ptr<tmk::DevVocab> *voc) {
    if (!v || !v->voc) return fail(TRIE_EINVAL, "vocabulary handle is NULL");
    int rc;
    if ((rc = current_device(dev)) != TRIE_OK) return rc;
    if (v->voc->device != *dev) return fail(TRIE_EINVAL, "the vocabulary handle belongs to another device");
    *voc = v->voc;
    return TRIE_OK;
}

int trie_compile_masks(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                       uint32_t *d_mask, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (!vocab_offsets) return fail(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || V > INT32_MAX - 32) return fail(TRIE_EINVAL, "V must be in [2, 2^31-32]");
    int dev, rc;
    if ((rc = check_mask_arg(d_mask)) != TRIE_OK) return rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = get_vocab(vocab_bytes, vocab_offsets, V, dev, &voc)) != TRIE_OK) return rc;
    return compile_masks(h, voc, dev, d_mask, stream);
}

int trie_compile_masks_vocab(trie_t h, trie_vocab_t v, uint32_t *d_mask, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    int dev, rc;
    if ((rc = check_mask_arg(d_mask)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = vocab_of(v, &dev, &voc)) != TRIE_OK) return rc;
    return compile_masks(h, voc, dev, d_mask, stream);
}

int trie_advance(trie_t h, int32_t *d_states, const int32_t *d_tokens, int32_t B, int32_t *d_err,
                 cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_states || !d_tokens)) return fail(TRIE_EINVAL, "d_states / d_tokens is NULL");
    std::shared_ptr<tmk::DevVocab> voc;
    bool use_trans;
    {
        std::lock_guard<std::mutex> lk(h->mu);
        voc = h->vocab;
        use_trans = h->trans_vocab == voc;
    }
    if (!voc) return fail(TRIE_ESTATE, "trie_advance before trie_compile_masks on this handle");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != h->dev.device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e =
        tmk::launch_advance(h->dev, h->host.n, *voc, d_states, d_states, d_tokens, B, d_err, use_trans, stream);
    if (e != cudaSuccess) return fail_cuda(e, "advance launch");
    return TRIE_OK;
}

int trie_advance_apply(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out,
                       int32_t *d_err, void *d_logits, int dtype, int32_t B, int32_t V, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (dtype != TRIE_DTYPE_F32 && dtype != TRIE_DTYPE_BF16) return fail(TRIE_EINVAL, "unknown dtype");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_states_in || !d_tokens || !d_states_out || !d_logits))
        return fail(TRIE_EINVAL, "a device pointer is NULL");
    if (B > 0 && d_states_in == d_states_out)
        return fail(TRIE_EINVAL, "d_states_in and d_states_out must be different buffers");
    std::shared_ptr<tmk::DevVocab> voc;
    uint32_t *mask;
    int32_t mV;
    bool use_trans;
    tmk::SegRef seg;
    {
        std::lock_guard<std::mutex> lk(h->mu);
        voc = h->vocab;
        mask = h->mask;
        mV = h->mask_V;
        use_trans = h->trans_vocab == voc;
        seg = h->mask_seg;
    }
    if (!mask || !voc) return fail(TRIE_ESTATE, "trie_advance_apply before trie_compile_masks on this handle");
    if (V != mV || V != voc->V) return fail(TRIE_EINVAL, "V differs from the compiled mask's V");
    if (reinterpret_cast<uintptr_t>(d_logits) & uintptr_t(dtype == TRIE_DTYPE_F32 ? 3 : 1))
        return fail(TRIE_EINVAL, "d_logits is not aligned to its element size");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != h->dev.device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e = tmk::launch_advance_apply(h->dev, h->host.n, *voc, use_trans, d_states_in, d_tokens,
                                              d_states_out, d_err, d_logits, dtype, mask, B, num_sms(dev), stream,
                                              seg);
    if (e != cudaSuccess) return fail_cuda(e, "advance-apply launch");
    return TRIE_OK;
}

int trie_apply_mask(trie_t h, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                    cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (dtype != TRIE_DTYPE_F32 && dtype != TRIE_DTYPE_BF16) return fail(TRIE_EINVAL, "unknown dtype");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_logits || !d_states)) return fail(TRIE_EINVAL, "d_logits / d_states is NULL");
    uint32_t *mask;
    int32_t mV;
    tmk::SegRef seg;
    {
        std::lock_guard<std::mutex> lk(h->mu);
        mask = h->mask;
        mV = h->mask_V;
        seg = h->mask_seg;
    }
    if (!mask) return fail(TRIE_ESTATE, "trie_apply_mask before trie_compile_masks on this handle");
    if (V != mV) return fail(TRIE_EINVAL, "V differs from the compiled mask's V");
    if (reinterpret_cast<uintptr_t>(d_logits) & uintptr_t(dtype == TRIE_DTYPE_F32 ? 3 : 1))
        return fail(TRIE_EINVAL, "d_logits is not aligned to its element size");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != h->dev.device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e = tmk::launch_apply(d_logits, dtype, mask, d_states, B, V, h->host.n, num_sms(dev), stream, seg);
    if (e != cudaSuccess) return fail_cuda(e, "apply launch");
    return TRIE_OK;
}

// Blocks of released valid lists kept for the next handles' lists: a fresh
// block from the pool cost 0.3-0.4 ms of host time for the 4.8 M-node forest
// (381 MB), more than the list compile's kernels. A block is reused once the
// event recorded at its release (if any) has completed; at most
// kSpareListBlocks are kept per device, the rest go back to the pool.
constexpr size_t kSpareListBlocks = 2;
struct SpareBlock {
    int dev;
    void *p;
    size_t bytes;
    cudaEvent_t ready;  // null: free for use at once
};
static std::mutex g_spare_mu;
static std::vector<SpareBlock> &g_spare = *new std::vector<SpareBlock>();

static void *take_spare_block(int dev, size_t bytes) {
    std::lock_guard<std::mutex> lk(g_spare_mu);
    for (size_t i = 0; i < g_spare.size(); i++) {
        SpareBlock &b = g_spare[i];
        if (b.dev != dev || b.bytes < bytes || b.bytes > 2 * bytes) continue;
        if (b.ready) {
            const cudaError_t q = cudaEventQuery(b.ready);
            if (q == cudaErrorNotReady) continue;
            cudaGetLastError();
            cudaEventDestroy(b.ready);
        }
        void *p = b.p;
        g_spare.erase(g_spare.begin() + long(i));
        return p;
    }
    return nullptr;
}

// Takes a block of `bytes` on device dev (current) whose last use is queued
// before `ready` (null: none pending); frees it in stream order on `stream`
// when the cache is full.
static void give_spare_block(int dev, void *p, size_t bytes, cudaEvent_t ready, cudaStream_t stream) {
    {
        std::lock_guard<std::mutex> lk(g_spare_mu);
        size_t held = 0;
        for (const SpareBlock &b : g_spare) held += b.dev == dev;
        if (held < kSpareListBlocks) {
            g_spare.push_back(SpareBlock{dev, p, bytes, ready});
            return;
        }
    }
    if (ready) cudaEventDestroy(ready);
    cudaFreeAsync(p, stream);
    cudaGetLastError();
}

// Token buffers of up to this many entries (1 GiB) are sized by the bound on
// the number of list entries, with no read-back.
constexpr int64_t kListBoundEntries = int64_t(1) << 28;

// Whether the handle holds lists (their size may still be on the device).
static bool lists_built(trie_t h) {
    std::lock_guard<std::mutex> lk(h->mu);
    return h->lists.n_valid_on_device || h->lists.n_valid >= 0;
}

// The vocabulary's reversed-token trie as a device edge table (the list
// compile's walk), built on first use: on the host, then its edges inserted
// on the device (host-synchronous, once per vocabulary and device).
static int ensure_rev_trie(tmk::DevVocab *voc) {
    std::lock_guard<std::mutex> lk(voc->rt_mu);
    if (voc->rt_state == 1) return TRIE_OK;
    if (voc->rt_state < 0) return fail(TRIE_EINVAL, "the vocabulary is too large for the valid-list walk");
    const int32_t V = voc->V;
    tmk::RevTokenTrie rt;
    std::string err;
    try {
        // from the vocabulary's host copy: its bytes start at the caller's offsets[0]
        const int64_t b0 = voc->src_offsets[0];
        std::vector<int64_t> rel;
        const int64_t *vo = voc->src_offsets.data();
        if (b0 != 0) {
            rel.resize(size_t(V) + 1);
            for (size_t i = 0; i <= size_t(V); i++) rel[i] = voc->src_offsets[i] - b0;
            vo = rel.data();
        }
        err = tmk::build_reversed_token_trie(voc->src_bytes.data(), vo, V, &rt);
    } catch (const std::bad_alloc &) {
        return fail(TRIE_ENOMEM, "host allocation failed while building the reversed-token trie");
    }
    if (!err.empty()) {
        voc->rt_state = -1;
        return fail(TRIE_EINVAL, err);
    }
    uint64_t S = 16;
    while (S < 2 * uint64_t(rt.n)) S <<= 1;
    Layout L;
    const size_t o_edge = L.add(sizeof(uint4) * size_t(S));
    const size_t o_next = rt.next.empty() ? 0 : L.add(sizeof(int32_t) * size_t(V));
    Layout T;  // build-time arrays
    const size_t t_par = T.add(sizeof(int32_t) * size_t(rt.n));
    const size_t t_lab = T.add(size_t(rt.n));
    const size_t t_tok = T.add(sizeof(int32_t) * size_t(rt.n));
    DeviceGuard g(voc->device);
    void *base = nullptr, *tmp = nullptr;
    cudaError_t e = cudaMalloc(&base, L.total);
    if (e == cudaSuccess) e = cudaMalloc(&tmp, T.total);
    if (e != cudaSuccess) {
        cudaGetLastError();
        if (base) cudaFree(base);
        return fail(TRIE_ENOMEM, std::string("cudaMalloc for the reversed-token trie: ") + cudaGetErrorString(e));
    }
    char *b = static_cast<char *>(base), *t = static_cast<char *>(tmp);
    if ((e = cudaMemcpy(t + t_par, rt.parent.data(), sizeof(int32_t) * size_t(rt.n), cudaMemcpyHostToDevice)) ==
            cudaSuccess &&
        (e = cudaMemcpy(t + t_lab, rt.label.data(), size_t(rt.n), cudaMemcpyHostToDevice)) == cudaSuccess &&
        (e = cudaMemcpy(t + t_tok, rt.token.data(), sizeof(int32_t) * size_t(rt.n), cudaMemcpyHostToDevice)) ==
            cudaSuccess &&
        (rt.next.empty() || (e = cudaMemcpy(b + o_next, rt.next.data(), sizeof(int32_t) * size_t(V),
                                            cudaMemcpyHostToDevice)) == cudaSuccess) &&
        (e = tmk::launch_rt_build(reinterpret_cast<const int32_t *>(t + t_par),
                                  reinterpret_cast<const uint8_t *>(t + t_lab),
                                  reinterpret_cast<const int32_t *>(t + t_tok), rt.n,
                                  reinterpret_cast<uint4 *>(b + o_edge), uint32_t(S - 1), num_sms(voc->device),
                                  0)) == cudaSuccess)
        e = cudaDeviceSynchronize();
    cudaFree(tmp);
    if (e != cudaSuccess) {
        cudaFree(base);
        return fail_cuda(e, "building the reversed-token trie");
    }
    voc->rt_base = base;
    voc->rt_edge = reinterpret_cast<const uint4 *>(b + o_edge);
    voc->rt_mask = uint32_t(S - 1);
    voc->tok_next = rt.next.empty() ? nullptr : reinterpret_cast<const int32_t *>(b + o_next);
    voc->rt_mult = rt.max_mult;
    voc->rt_state = 1;
    return TRIE_OK;
}

int trie_compile_masks_pairwise(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                                uint32_t *d_mask, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (!vocab_offsets) return fail(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || V > INT32_MAX - 32) return fail(TRIE_EINVAL, "V must be in [2, 2^31-32]");
    if (!d_mask) return fail(TRIE_EINVAL, "d_mask is NULL");
    if (reinterpret_cast<uintptr_t>(d_mask) & 3u) return fail(TRIE_EINVAL, "d_mask must be 4-byte aligned");
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = get_vocab(vocab_bytes, vocab_offsets, V, dev, &voc)) != TRIE_OK) return rc;
    if ((rc = ensure_device_trie(h, dev, stream)) != TRIE_OK) return rc;
    cudaError_t e = tmk::launch_mask_pairwise(h->dev, h->host.n, *voc, d_mask, num_sms(dev), stream);
    if (e != cudaSuccess) return fail_cuda(e, "pairwise mask compile launch");
    return TRIE_OK;
}

// The list compile with the vocabulary resolved (from the cache, or a vocabulary handle).
static int compile_lists(trie_t h, const std::shared_ptr<tmk::DevVocab> &voc, int dev, cudaStream_t stream) {
    int rc;
    const int32_t V = voc->V;
    if ((rc = ensure_rev_trie(voc.get())) != TRIE_OK) return rc;
    if ((rc = ensure_device_trie(h, dev, stream)) != TRIE_OK) return rc;
    const int32_t n = h->host.n;
    tmk::DevLists &L = h->lists;
    const int32_t lmax = std::min(voc->max_len, h->host.max_depth);
    // a node is the end of at most one path of each length up to lmax, each
    // spelled by at most rt_mult ids, plus EOS. While that bound is modest the
    // token buffer is sized by it and nothing is read back; otherwise the
    // exact total is read back between the two walks (host-synchronous).
    const int64_t bound = int64_t(n) * (int64_t(lmax) * voc->rt_mult + 1);
    const bool by_bound = bound <= std::max<int64_t>(kListBoundEntries, L.tok_cap);
    if (!L.base) {  // per-row counts, offsets, scan scratch (and a first token buffer, in one block)
        Layout lay;
        const size_t o_cnt = lay.add(sizeof(int32_t) * size_t(n));
        const size_t o_off = lay.add(sizeof(int64_t) * (size_t(n) + 1));
        const size_t o_tile = lay.add(sizeof(int64_t) * (size_t(n) / 4096 + 2));
        const size_t o_tot = lay.add(sizeof(int64_t));
        const size_t o_tok = by_bound ? lay.add(2 * sizeof(int32_t) * size_t(std::max<int64_t>(bound, 1))) : 0;
        void *base = take_spare_block(dev, lay.total);
        if (!base && (rc = pool_alloc(dev, lay.total, stream, &base, "the valid lists")) != TRIE_OK) return rc;
        cudaEvent_t done = nullptr;
        cudaError_t e = cudaEventCreateWithFlags(&done, cudaEventDisableTiming);
        if (e != cudaSuccess) {
            pool_free(base);
            return fail_cuda(e, "creating the valid lists' event");
        }
        char *b = static_cast<char *>(base);
        L.base = base;
        L.base_bytes = lay.total;
        L.done = done;
        L.count = reinterpret_cast<int32_t *>(b + o_cnt);
        L.off = reinterpret_cast<int64_t *>(b + o_off);
        L.tile_sum = reinterpret_cast<int64_t *>(b + o_tile);
        L.total = reinterpret_cast<int64_t *>(b + o_tot);
        if (by_bound) {
            L.toks = reinterpret_cast<int32_t *>(b + o_tok);
            L.tok_cap = std::max<int64_t>(bound, 1);
            L.ends = L.toks + L.tok_cap;
            L.toks_separate = false;
        }
    }
    const int sms = num_sms(dev);
    auto grow = [&](int64_t need) -> int {
        if (need <= L.tok_cap) return TRIE_OK;
        if (L.toks_separate) pool_free(L.toks);  // earlier apply calls may still read it
        L.toks = nullptr;                         // (a buffer inside the block at base stays there)
        L.ends = nullptr;
        L.tok_cap = 0;
        void *toks = nullptr;
        need = std::max<int64_t>(need, 1);
        int r = pool_alloc(dev, 2 * sizeof(int32_t) * size_t(need), stream, &toks, "the valid-list tokens");
        if (r != TRIE_OK) return r;
        L.toks = static_cast<int32_t *>(toks);
        L.ends = L.toks + need;
        L.tok_cap = need;
        L.toks_separate = true;
        return TRIE_OK;
    };
    auto failed = [&](int r) {
        L.n_valid = -1;
        L.n_valid_on_device = false;
        return r;
    };
    if (by_bound && (rc = grow(bound)) != TRIE_OK) return failed(rc);
    cudaError_t e = tmk::launch_lists_count(h->dev, n, *voc, lmax, L, sms, stream);
    if (e != cudaSuccess) return failed(fail_cuda(e, "valid-list count"));
    if (!by_bound) {
        int64_t total = 0;
        if ((e = cudaMemcpyAsync(&total, L.total, sizeof(int64_t), cudaMemcpyDeviceToHost, stream)) != cudaSuccess ||
            (e = cudaStreamSynchronize(stream)) != cudaSuccess)
            return failed(fail_cuda(e, "reading the number of list entries back"));
        if ((rc = grow(total + total / 2)) != TRIE_OK) return failed(rc);
    }
    e = tmk::launch_lists_write(h->dev, n, *voc, lmax, L, sms, stream);
    if (e == cudaSuccess) e = cudaEventRecord(L.done, stream);
    if (e != cudaSuccess) return failed(fail_cuda(e, "valid-list write"));
    std::lock_guard<std::mutex> lk(h->mu);
    L.n_valid_on_device = true;
    L.V = V;
    h->vocab = voc;
    return TRIE_OK;
}

int trie_compile_lists(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                       cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (!vocab_offsets) return fail(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || V > INT32_MAX - 32) return fail(TRIE_EINVAL, "V must be in [2, 2^31-32]");
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = get_vocab(vocab_bytes, vocab_offsets, V, dev, &voc)) != TRIE_OK) return rc;
    return compile_lists(h, voc, dev, stream);
}

int trie_compile_lists_vocab(trie_t h, trie_vocab_t v, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    int dev, rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = vocab_of(v, &dev, &voc)) != TRIE_OK) return rc;
    return compile_lists(h, voc, dev, stream);
}

int trie_vocab_create(const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V, trie_vocab_t *out) {
    if (!out) return fail(TRIE_EINVAL, "out is NULL");
    *out = nullptr;
    if (!vocab_offsets) return fail(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || V > INT32_MAX - 32) return fail(TRIE_EINVAL, "V must be in [2, 2^31-32]");
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = get_vocab(vocab_bytes, vocab_offsets, V, dev, &voc)) != TRIE_OK) return rc;
    trie_vocab_t v = new (std::nothrow) trie_vocab_s;
    if (!v) return fail(TRIE_ENOMEM, "host allocation failed");
    v->voc = std::move(voc);
    *out = v;
    return TRIE_OK;
}

int32_t trie_vocab_size(trie_vocab_t v) { return v && v->voc ? v->voc->V : -1; }

void trie_vocab_destroy(trie_vocab_t v) { delete v; }

int64_t trie_num_valid(trie_t h) {
    if (!h) return -1;
    tmk::DevLists &L = h->lists;
    std::lock_guard<std::mutex> lk(h->mu);
    if (L.n_valid_on_device) {  // the total of the last build, once its kernels are done
        int64_t total = -1;
        DeviceGuard g(h->dev.device);
        if (cudaEventSynchronize(L.done) != cudaSuccess ||
            cudaMemcpy(&total, L.total, sizeof(int64_t), cudaMemcpyDeviceToHost) != cudaSuccess) {
            cudaGetLastError();
            fail(TRIE_ECUDA, "reading the number of list entries back failed");
            return -1;
        }
        L.n_valid = total;
        L.n_valid_on_device = false;
    }
    return L.n_valid;
}

int trie_copy_lists(trie_t h, int64_t *d_offsets, int32_t *d_tokens, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    const tmk::DevLists &L = h->lists;
    if (!lists_built(h)) return fail(TRIE_ESTATE, "trie_copy_lists before trie_compile_lists on this handle");
    if (trie_num_valid(h) < 0) return TRIE_ECUDA;
    if (d_offsets) {
        cudaError_t e = cudaMemcpyAsync(d_offsets, L.off, sizeof(int64_t) * (size_t(h->host.n) + 1),
                                        cudaMemcpyDeviceToDevice, stream);
        if (e != cudaSuccess) return fail_cuda(e, "copying the list offsets");
    }
    if (d_tokens && L.n_valid > 0) {
        cudaError_t e = cudaMemcpyAsync(d_tokens, L.toks, sizeof(int32_t) * size_t(L.n_valid),
                                        cudaMemcpyDeviceToDevice, stream);
        if (e != cudaSuccess) return fail_cuda(e, "copying the list tokens");
    }
    return TRIE_OK;
}

int trie_apply_lists(trie_t h, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                     cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (dtype != TRIE_DTYPE_F32 && dtype != TRIE_DTYPE_BF16) return fail(TRIE_EINVAL, "unknown dtype");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_logits || !d_states)) return fail(TRIE_EINVAL, "d_logits / d_states is NULL");
    if (!lists_built(h)) return fail(TRIE_ESTATE, "trie_apply_lists before trie_compile_lists on this handle");
    if (V != h->lists.V) return fail(TRIE_EINVAL, "V differs from the compiled lists' V");
    if (reinterpret_cast<uintptr_t>(d_logits) & uintptr_t(dtype == TRIE_DTYPE_F32 ? 3 : 1))
        return fail(TRIE_EINVAL, "d_logits is not aligned to its element size");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != h->dev.device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e = tmk::launch_apply_lists(d_logits, dtype, h->lists, d_states, B, V, h->host.n, stream);
    if (e != cudaSuccess) return fail_cuda(e, "apply-lists launch");
    return TRIE_OK;
}

int trie_lazy_init(trie_t h, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                   int32_t cache_rows, int32_t max_batch) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (!vocab_offsets) return fail(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || (int64_t(V) + 31) / 32 > tmk::kLazyMaxWords)
        return fail(TRIE_EINVAL, "V must be in [2, " + std::to_string(tmk::kLazyMaxWords * 32) + "] for lazy rows");
    if (cache_rows < 0 || cache_rows > tmk::kLazyMaxCacheRows)
        return fail(TRIE_EINVAL, "cache_rows must be in [0, " + std::to_string(tmk::kLazyMaxCacheRows) + "]");
    if (max_batch < 1 || max_batch > tmk::kLazyMaxBatch)
        return fail(TRIE_EINVAL, "max_batch must be in [1, " + std::to_string(tmk::kLazyMaxBatch) + "]");
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = get_vocab(vocab_bytes, vocab_offsets, V, dev, &voc)) != TRIE_OK) return rc;
    if ((rc = tmk::ensure_host_arrays(h)) != TRIE_OK) return rc;  // the pre-order tables
    if ((rc = ensure_device_trie(h, dev, 0)) != TRIE_OK) return rc;
    cudaError_t e = cudaDeviceSynchronize();  // earlier lazy calls may still use the old cache
    if (e != cudaSuccess) return fail_cuda(e, "synchronising before the lazy set-up");
    {  // the transition table takes the moves the lazy rows find for this vocabulary
        std::lock_guard<std::mutex> lk(h->mu);
        if (h->dev.trans && h->trans_vocab != voc) {
            h->trans_vocab.reset();
            h->trans_complete = false;
            if ((e = tmk::launch_trans_clear(h->dev, num_sms(dev), 0)) != cudaSuccess)
                return fail_cuda(e, "transition table clear");
            h->trans_vocab = voc;
        }
    }
    tmk::DevLazy &L = h->lazy;
    pool_free(L.base);
    L = tmk::DevLazy();
    const int32_t C = (cache_rows + tmk::kLazyWays - 1) / tmk::kLazyWays * tmk::kLazyWays;
    const int64_t W = (int64_t(V) + 31) / 32;
    const size_t n = size_t(h->host.n), mb = size_t(max_batch);
    Layout lay;
    const size_t o_rows = lay.add(sizeof(uint32_t) * size_t(W) * (size_t(C) + mb));
    const size_t o_tag = lay.add(sizeof(int32_t) * size_t(C));
    const size_t o_stamp = lay.add(sizeof(uint32_t) * size_t(C));
    const size_t o_ctrl = lay.add(sizeof(tmk::LazyCtrl));
    const size_t o_slot = lay.add(sizeof(int32_t) * mb);
    const size_t o_mnode = lay.add(sizeof(int32_t) * mb);
    const size_t o_mslot = lay.add(sizeof(int32_t) * mb);
    const size_t o_rowu = lay.add(sizeof(int32_t) * mb);
    const size_t o_task = lay.add(sizeof(int4) * (mb + size_t(tmk::kLazySplitRows) * tmk::kLazyMaxParts));
    const size_t o_pnode = lay.add(sizeof(int32_t) * n);
    const size_t o_pdep = lay.add(sizeof(int32_t) * n);
    const size_t o_psize = lay.add(sizeof(int32_t) * n);
    const size_t o_pos = lay.add(sizeof(int32_t) * n);
    const size_t o_pre = lay.add(sizeof(tmk::LazyNode) * n);
    void *base = nullptr;
    if ((rc = pool_alloc(dev, lay.total, 0, &base, "the lazy rows")) != TRIE_OK) return rc;
    char *b = static_cast<char *>(base);
    L.device = dev;
    L.base = base;
    L.C = C;
    L.max_batch = max_batch;
    L.V = V;
    L.W = W;
    L.rows = reinterpret_cast<uint32_t *>(b + o_rows);
    L.tag = reinterpret_cast<int32_t *>(b + o_tag);
    L.stamp = reinterpret_cast<uint32_t *>(b + o_stamp);
    L.ctrl = reinterpret_cast<tmk::LazyCtrl *>(b + o_ctrl);
    L.slot_of = reinterpret_cast<int32_t *>(b + o_slot);
    L.miss_node = reinterpret_cast<int32_t *>(b + o_mnode);
    L.miss_slot = reinterpret_cast<int32_t *>(b + o_mslot);
    L.row_u = reinterpret_cast<int32_t *>(b + o_rowu);
    L.task = reinterpret_cast<int4 *>(b + o_task);
    L.pre_node = reinterpret_cast<int32_t *>(b + o_pnode);
    L.pre_depth = reinterpret_cast<int32_t *>(b + o_pdep);
    L.pre_size = reinterpret_cast<int32_t *>(b + o_psize);
    L.pos_of = reinterpret_cast<int32_t *>(b + o_pos);
    L.pre = reinterpret_cast<tmk::LazyNode *>(b + o_pre);
    const tmk::LazyCtrl ctrl0 = {1u, 0, 0, 0, 0ull, 0ull};
    const tmk::HostTrie &t = h->host;
    if ((e = cudaMemset(L.tag, 0xFF, sizeof(int32_t) * size_t(C))) != cudaSuccess ||
        (e = cudaMemset(L.stamp, 0, sizeof(uint32_t) * size_t(C))) != cudaSuccess ||
        (e = cudaMemcpy(L.ctrl, &ctrl0, sizeof(ctrl0), cudaMemcpyHostToDevice)) != cudaSuccess ||
        (e = cudaMemcpy(L.pre_node, t.pre_node.data(), sizeof(int32_t) * n, cudaMemcpyHostToDevice)) !=
            cudaSuccess ||
        (e = cudaMemcpy(L.pre_depth, t.pre_depth.data(), sizeof(int32_t) * n, cudaMemcpyHostToDevice)) !=
            cudaSuccess ||
        (e = cudaMemcpy(L.pre_size, t.pre_size.data(), sizeof(int32_t) * n, cudaMemcpyHostToDevice)) !=
            cudaSuccess ||
        (e = tmk::launch_lazy_tables(h->dev, L, h->host.n, 0)) != cudaSuccess || (e = cudaDeviceSynchronize()) != cudaSuccess) {
        pool_free(base);
        L = tmk::DevLazy();
        return fail_cuda(e, "lazy-row set-up");
    }
    L.vocab = voc;
    return TRIE_OK;
}

int trie_lazy_apply(trie_t h, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                    cudaStream_t stream) {
    if (B > 0 && !d_logits) return fail(TRIE_EINVAL, "d_logits is NULL");
    return lazy_call(h, d_states, nullptr, nullptr, nullptr, d_logits, dtype, nullptr, B, V, stream);
}

int trie_lazy_advance_apply(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out,
                            int32_t *d_err, void *d_logits, int dtype, int32_t B, int32_t V, cudaStream_t stream) {
    if (B > 0 && (!d_tokens || !d_logits)) return fail(TRIE_EINVAL, "d_tokens / d_logits is NULL");
    return lazy_call(h, d_states_in, d_tokens, d_states_out, d_err, d_logits, dtype, nullptr, B, V, stream);
}

int trie_lazy_rows(trie_t h, const int32_t *d_states, int32_t B, uint32_t *d_rows, cudaStream_t stream) {
    if (B > 0 && !d_rows) return fail(TRIE_EINVAL, "d_rows is NULL");
    const int32_t V = h ? h->lazy.V : 0;
    return lazy_call(h, d_states, nullptr, nullptr, nullptr, nullptr, 0, d_rows, B, V, stream);
}

int trie_lazy_stats(trie_t h, int64_t *hits, int64_t *misses) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (!h->lazy.base) return fail(TRIE_ESTATE, "trie_lazy_stats before trie_lazy_init on this handle");
    DeviceGuard g(h->lazy.device);
    tmk::LazyCtrl c;
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemcpy(&c, h->lazy.ctrl, sizeof(c), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return fail_cuda(e, "reading the lazy-row counters");
    if (hits) *hits = int64_t(c.hits);
    if (misses) *misses = int64_t(c.misses);
    return TRIE_OK;
}

int trie_advance_apply_lists(trie_t h, const int32_t *d_states_in, const int32_t *d_tokens, int32_t *d_states_out,
                             int32_t *d_err, void *d_logits, int dtype, int32_t B, int32_t V, cudaStream_t stream) {
    if (!h) return fail(TRIE_EINVAL, "handle is NULL");
    if (dtype != TRIE_DTYPE_F32 && dtype != TRIE_DTYPE_BF16) return fail(TRIE_EINVAL, "unknown dtype");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_states_in || !d_tokens || !d_states_out || !d_logits))
        return fail(TRIE_EINVAL, "a device pointer is NULL");
    if (B > 0 && d_states_in == d_states_out)
        return fail(TRIE_EINVAL, "d_states_in and d_states_out must be different buffers");
    if (!lists_built(h))
        return fail(TRIE_ESTATE, "trie_advance_apply_lists before trie_compile_lists on this handle");
    if (V != h->lists.V) return fail(TRIE_EINVAL, "V differs from the compiled lists' V");
    if (reinterpret_cast<uintptr_t>(d_logits) & uintptr_t(dtype == TRIE_DTYPE_F32 ? 3 : 1))
        return fail(TRIE_EINVAL, "d_logits is not aligned to its element size");
    std::shared_ptr<tmk::DevVocab> voc;
    bool use_trans;
    {
        std::lock_guard<std::mutex> lk(h->mu);
        voc = h->vocab;
        use_trans = h->trans_vocab == voc;
    }
    if (!voc || voc->V != V) return fail(TRIE_ESTATE, "the handle's vocabulary is not the lists' vocabulary");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != h->dev.device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e = tmk::launch_advance_apply_lists(h->dev, h->host.n, *voc, use_trans, d_states_in, d_tokens,
                                                    d_states_out, d_err, d_logits, dtype, h->lists, B, stream);
    if (e != cudaSuccess) return fail_cuda(e, "advance-apply-lists launch");
    return TRIE_OK;
}

int fmt_build(const uint8_t *classes, int32_t L, fmt_t *out) {
    if (!out) return fail(TRIE_EINVAL, "out is NULL");
    *out = nullptr;
    if (L < 0 || L > tmk::kFmtMaxLen)
        return fail(TRIE_EINVAL, "L must be in [0, " + std::to_string(tmk::kFmtMaxLen) + "]");
    if (L > 0 && !classes) return fail(TRIE_EINVAL, "classes is NULL");
    fmt_s *f = new (std::nothrow) fmt_s;
    if (!f) return fail(TRIE_ENOMEM, "host allocation failed");
    try {
        f->classes.assign(size_t(L) * 8, 0u);
    } catch (const std::bad_alloc &) {
        delete f;
        return fail(TRIE_ENOMEM, "host allocation failed");
    }
    for (int32_t i = 0; i < L; i++)
        for (int c = 0; c < 256; c++)
            if ((classes[32 * size_t(i) + size_t(c / 8)] >> (c % 8)) & 1)
                f->classes[8 * size_t(i) + size_t(c / 32)] |= 1u << (c % 32);
    f->L = L;
    *out = f;
    return TRIE_OK;
}

int32_t fmt_length(fmt_t f) { return f ? f->L : -1; }

int fmt_compile_masks(fmt_t f, const uint8_t *vocab_bytes, const int64_t *vocab_offsets, int32_t V,
                      uint32_t *d_mask, cudaStream_t stream) {
    if (!f) return fail(TRIE_EINVAL, "handle is NULL");
    if (!vocab_offsets) return fail(TRIE_EINVAL, "vocab_offsets is NULL");
    if (V < 2 || V > INT32_MAX - 32) return fail(TRIE_EINVAL, "V must be in [2, 2^31-32]");
    if (!d_mask) return fail(TRIE_EINVAL, "d_mask is NULL");
    if (reinterpret_cast<uintptr_t>(d_mask) & 3u) return fail(TRIE_EINVAL, "d_mask must be 4-byte aligned");
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    std::shared_ptr<tmk::DevVocab> voc;
    if ((rc = get_vocab(vocab_bytes, vocab_offsets, V, dev, &voc)) != TRIE_OK) return rc;
    std::lock_guard<std::mutex> lk(f->mu);
    if (f->d_classes && f->device != dev)
        return fail(TRIE_EINVAL, "format was uploaded to device " + std::to_string(f->device) + ", called on device " +
                                     std::to_string(dev));
    if (!f->d_classes) {
        void *p = nullptr;
        cudaError_t e = cudaMalloc(&p, sizeof(uint32_t) * std::max<size_t>(f->classes.size(), 1));
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(TRIE_ENOMEM, std::string("cudaMalloc for the format: ") + cudaGetErrorString(e));
        }
        if (!f->classes.empty() &&
            (e = cudaMemcpy(p, f->classes.data(), sizeof(uint32_t) * f->classes.size(), cudaMemcpyHostToDevice)) !=
                cudaSuccess) {
            cudaFree(p);
            return fail_cuda(e, "uploading the format");
        }
        f->d_classes = static_cast<uint32_t *>(p);
        f->device = dev;
    }
    cudaError_t e = tmk::launch_fmt_compile(f->d_classes, f->L, *voc, d_mask, num_sms(dev), stream);
    if (e != cudaSuccess) return fail_cuda(e, "format mask launch");
    f->vocab = voc;
    f->mask = d_mask;
    f->mask_V = V;
    return TRIE_OK;
}

int fmt_advance(fmt_t f, int32_t *d_states, const int32_t *d_tokens, int32_t B, int32_t *d_err,
                cudaStream_t stream) {
    if (!f) return fail(TRIE_EINVAL, "handle is NULL");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_states || !d_tokens)) return fail(TRIE_EINVAL, "d_states / d_tokens is NULL");
    std::shared_ptr<tmk::DevVocab> voc;
    {
        std::lock_guard<std::mutex> lk(f->mu);
        voc = f->vocab;
    }
    if (!voc) return fail(TRIE_ESTATE, "fmt_advance before fmt_compile_masks on this handle");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != f->device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e = tmk::launch_fmt_advance(f->d_classes, f->L, *voc, d_states, d_states, d_tokens, B, d_err, stream);
    if (e != cudaSuccess) return fail_cuda(e, "format advance launch");
    return TRIE_OK;
}

int fmt_apply_mask(fmt_t f, void *d_logits, int dtype, const int32_t *d_states, int32_t B, int32_t V,
                   cudaStream_t stream) {
    if (!f) return fail(TRIE_EINVAL, "handle is NULL");
    if (dtype != TRIE_DTYPE_F32 && dtype != TRIE_DTYPE_BF16) return fail(TRIE_EINVAL, "unknown dtype");
    if (B < 0) return fail(TRIE_EINVAL, "B must be >= 0");
    if (B > 0 && (!d_logits || !d_states)) return fail(TRIE_EINVAL, "d_logits / d_states is NULL");
    uint32_t *mask;
    int32_t mV;
    {
        std::lock_guard<std::mutex> lk(f->mu);
        mask = f->mask;
        mV = f->mask_V;
    }
    if (!mask) return fail(TRIE_ESTATE, "fmt_apply_mask before fmt_compile_masks on this handle");
    if (V != mV) return fail(TRIE_EINVAL, "V differs from the compiled mask's V");
    if (reinterpret_cast<uintptr_t>(d_logits) & uintptr_t(dtype == TRIE_DTYPE_F32 ? 3 : 1))
        return fail(TRIE_EINVAL, "d_logits is not aligned to its element size");
    if (B == 0) return TRIE_OK;
    int dev, rc;
    if ((rc = current_device(&dev)) != TRIE_OK) return rc;
    if (dev != f->device) return fail(TRIE_EINVAL, "handle belongs to another device");
    cudaError_t e = tmk::launch_apply(d_logits, dtype, mask, d_states, B, V, f->L + 1, num_sms(dev), stream);
    if (e != cudaSuccess) return fail_cuda(e, "format apply launch");
    return TRIE_OK;
}

int fmt_destroy(fmt_t f) {
    if (!f) return TRIE_OK;
    if (f->d_classes) {
        DeviceGuard g(f->device);
        cudaFree(f->d_classes);  // waits for work that may still read it
    }
    delete f;
    return TRIE_OK;
}

int trie_destroy(trie_t h) {
    if (!h) return TRIE_OK;
    if (h->lazy.base) {
        DeviceGuard g(h->lazy.device);
        pool_free(h->lazy.base);
    }
    if (h->dev.base || h->lists.base) {
        DeviceGuard g(h->dev.device);
        // after the work on the device that may still read these
        if (h->lists.toks_separate) pool_free(h->lists.toks);
        if (h->lists.base) {
            cudaDeviceSynchronize();  // no queued work still uses the block
            give_spare_block(h->dev.device, h->lists.base, h->lists.base_bytes, nullptr, 0);
        }
        pool_free(h->dev.hits_base);
        pool_free(h->dev.seg_epoch);
        pool_free(h->dev.base);
        if (h->lists.done) cudaEventDestroy(h->lists.done);
    }
    delete h;
    return TRIE_OK;
}

// Handles released by trie_destroy_async whose host arrays may still be read
// by queued work: each waits for its event, and every release (and every
// build) frees those whose event has completed.
static std::mutex g_retired_mu;
static std::vector<std::pair<cudaEvent_t, trie_t>> &g_retired =
    *new std::vector<std::pair<cudaEvent_t, trie_t>>();

static void sweep_retired() {
    std::vector<trie_t> done;
    {
        std::lock_guard<std::mutex> lk(g_retired_mu);
        size_t keep = 0;
        for (size_t i = 0; i < g_retired.size(); i++) {
            const cudaError_t q = cudaEventQuery(g_retired[i].first);
            if (q == cudaErrorNotReady) {
                g_retired[keep++] = g_retired[i];
                continue;
            }
            cudaGetLastError();
            cudaEventDestroy(g_retired[i].first);
            done.push_back(g_retired[i].second);
        }
        g_retired.resize(keep);
    }
    for (trie_t h : done) delete h;
}

static void retire_handle(trie_t h, cudaEvent_t ev) {
    {
        std::lock_guard<std::mutex> lk(g_retired_mu);
        g_retired.emplace_back(ev, h);
    }
    sweep_retired();
}

int trie_destroy_async(trie_t h, cudaStream_t stream) {
    if (!h) return TRIE_OK;
    int rc = TRIE_OK;
    auto free_on = [&](void *p) {
        if (!p) return;
        cudaError_t e = cudaFreeAsync(p, stream);
        if (e != cudaSuccess) {
            cudaGetLastError();
            rc = fail_cuda(e, "stream-ordered free of the handle's device memory");
        }
    };
    // the vocabularies are released here, on the calling thread (the last
    // reference frees device memory, which a stream callback must not do)
    std::shared_ptr<tmk::DevVocab> v1 = std::move(h->vocab), v2 = std::move(h->trans_vocab),
                                   v3 = std::move(h->lazy.vocab);
    int dev = h->dev.base || h->lists.base || h->lists.toks ? h->dev.device : h->lazy.device;
    if (h->lazy.base) {
        DeviceGuard g(h->lazy.device);
        free_on(h->lazy.base);
    }
    if (h->dev.base || h->lists.base || h->lists.toks) {
        DeviceGuard g(h->dev.device);
        if (h->lists.toks_separate) free_on(h->lists.toks);
        if (h->lists.base) {  // kept for a later handle once the queued work is done
            cudaEvent_t ev = nullptr;
            if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) == cudaSuccess &&
                cudaEventRecord(ev, stream) == cudaSuccess) {
                give_spare_block(h->dev.device, h->lists.base, h->lists.base_bytes, ev, stream);
            } else {
                cudaGetLastError();
                if (ev) cudaEventDestroy(ev);
                free_on(h->lists.base);
            }
        }
        free_on(h->dev.hits_base);
        free_on(h->dev.seg_epoch);
        free_on(h->dev.base);
        // the event may still be pending: CUDA defers its destruction
        if (h->lists.done) cudaEventDestroy(h->lists.done);
    }
    if (dev < 0) {
        delete h;
        return rc;
    }
    // the host arrays (which an upload kernel may still be reading) go once
    // the work queued on the stream so far has run: an event marks that
    // point and a later call frees the handle once the event has completed
    // (no stream callback, which would hold up the stream's later work)
    DeviceGuard g(dev);
    cudaEvent_t ev = nullptr;
    cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventRecord(ev, stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        if (ev) cudaEventDestroy(ev);
        cudaStreamSynchronize(stream);
        cudaGetLastError();
        delete h;
        if (rc == TRIE_OK) rc = fail_cuda(e, "queueing the release of the handle's host memory");
        return rc;
    }
    retire_handle(h, ev);
    return rc;
}

}  // extern "C"
