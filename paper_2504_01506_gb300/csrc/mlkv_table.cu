// C ABI of the store (declared in include/mlkv_gpu.h): argument checks, the
// table's memory, the order of kernels of each call, the ordering of calls
// across streams under a staleness bound (bulk-synchronous, stale-synchronous
// or asynchronous, MLKV Section 3.3.1), status and timing.
#include <algorithm>
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <unordered_map>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "mlkv_internal.cuh"

// A named NVTX range around each call of the C ABI, for timeline tools (nsys,
// ncu --nvtx): it marks when the host issued the call's work, and the
// kernels launched inside it.  NVTX is header-only; with no tool attached a
// range costs a few nanoseconds.  -DMLKV_NVTX=0 leaves it out.
#ifndef MLKV_NVTX
#define MLKV_NVTX 1
#endif
#if MLKV_NVTX
#include <nvtx3/nvToolsExt.h>
namespace {
struct CallRange {
    explicit CallRange(const char* name) { nvtxRangePushA(name); }
    ~CallRange() { nvtxRangePop(); }
    CallRange(const CallRange&) = delete;
    CallRange& operator=(const CallRange&) = delete;
};
}  // namespace
#define MLKV_RANGE(name) CallRange mlkv_call_range_(name)
#else
#define MLKV_RANGE(name) ((void)0)
#endif

using namespace mlkv;

namespace {

int set_error(mlkv_table* t, int code, const char* fmt, ...) {
    if (t) {
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(t->last_error, sizeof(t->last_error), fmt, ap);
        va_end(ap);
    }
    return code;
}

int cuda_error(mlkv_table* t, cudaError_t e, const char* where) {
    return set_error(t, MLKV_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

#define CK(t, call)                                          \
    do {                                                     \
        cudaError_t e_ = (call);                             \
        if (e_ != cudaSuccess) return cuda_error((t), e_, #call); \
    } while (0)

int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// Host-side fault injection (mlkv_debug_fail): a countdown per kind; the call
// that takes it from 1 to 0 fails without calling CUDA at all, so no GPU ever
// sees a fault, and the error paths (MLKV_ERR_NOMEM, MLKV_ERR_CUDA, the
// clean-up of a half-opened table) run as they would for a real failure.
std::atomic<int64_t> g_fail_alloc{0};
std::atomic<int64_t> g_fail_copy{0};
std::atomic<int64_t> g_fail_wait{0};

bool injected(std::atomic<int64_t>& countdown) {
    int64_t v = countdown.load();
    while (v > 0)
        if (countdown.compare_exchange_weak(v, v - 1)) return v == 1;
    return false;
}

// Every device and pinned allocation and every host <-> device copy of the
// library goes through these.
template <class T>
cudaError_t dev_alloc(T** p, size_t bytes) {
    if (injected(g_fail_alloc)) {
        *p = nullptr;
        return cudaErrorMemoryAllocation;
    }
    return cudaMalloc((void**)p, bytes);
}

template <class T>
cudaError_t pinned_alloc(T** p, size_t bytes, unsigned flags) {
    if (injected(g_fail_alloc)) {
        *p = nullptr;
        return cudaErrorMemoryAllocation;
    }
    return cudaHostAlloc((void**)p, bytes, flags);
}

cudaError_t copy_async(void* dst, const void* src, size_t bytes, cudaMemcpyKind kind, cudaStream_t st) {
    if (injected(g_fail_copy)) return cudaErrorInvalidValue;
    return cudaMemcpyAsync(dst, src, bytes, kind, st);
}

// The host tier is pinned host memory from the driver's virtual-memory API
// (cuMemCreate on the host NUMA node nearest the GPU), mapped for the device
// alone.  The GPU then reaches it through its own page tables, in 2 MB pages.
// Host memory that the OS manages (mmap + cudaHostRegister) is reached through
// the CPU's page tables instead, which the OS keeps rewriting (huge pages
// split, NUMA scans); random rows over tens of GB of it moved an order of
// magnitude slower.  The CPU never touches the tier: rows are initialised,
// fetched, written back and exported by kernels.  The entry points come from
// the runtime, so the library does not link the driver library itself.
struct VmmApi {
    PFN_cuMemCreate_v10020 create = nullptr;
    PFN_cuMemRelease_v10020 release = nullptr;
    PFN_cuMemAddressReserve_v10020 reserve = nullptr;
    PFN_cuMemAddressFree_v10020 addr_free = nullptr;
    PFN_cuMemMap_v10020 map = nullptr;
    PFN_cuMemUnmap_v10020 unmap = nullptr;
    PFN_cuMemSetAccess_v10020 set_access = nullptr;
    PFN_cuMemGetAllocationGranularity_v10020 granularity = nullptr;
    bool ok = false;
};

const VmmApi& vmm_api() {
    static const VmmApi api = [] {
        VmmApi a;
        auto get = [](const char* name, void** fn) {
            cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
            return cudaGetDriverEntryPointByVersion(name, fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
                   q == cudaDriverEntryPointSuccess && *fn;
        };
        a.ok = get("cuMemCreate", (void**)&a.create) && get("cuMemRelease", (void**)&a.release) &&
               get("cuMemAddressReserve", (void**)&a.reserve) && get("cuMemAddressFree", (void**)&a.addr_free) &&
               get("cuMemMap", (void**)&a.map) && get("cuMemUnmap", (void**)&a.unmap) &&
               get("cuMemSetAccess", (void**)&a.set_access) &&
               get("cuMemGetAllocationGranularity", (void**)&a.granularity);
        return a;
    }();
    return api;
}

void host_tier_free(Tier& tr) {
    const VmmApi& v = vmm_api();
    if (v.ok && tr.host_dev) {
        const CUdeviceptr va = (CUdeviceptr)tr.host_dev;
        for (int64_t i = 0; i < tr.host_mapped; ++i) {
            v.unmap(va + (size_t)i * tr.host_chunk, tr.host_chunk);
            v.release((CUmemGenericAllocationHandle)tr.host_handles[i]);
        }
        v.addr_free(va, tr.host_bytes);
    }
    delete[] tr.host_handles;
    tr.host_handles = nullptr;
    tr.host_dev = nullptr;
    tr.host_mapped = 0;
}

// Reserves, creates and maps `bytes` (rounded up to whole chunks) of pinned host
// memory readable and writable by the table's device.
int host_tier_alloc(mlkv_table* t, size_t bytes) {
    Tier& tr = t->tier;
    const VmmApi& v = vmm_api();
    if (!v.ok) return set_error(t, MLKV_ERR_CUDA, "driver virtual-memory entry points unavailable");
    int numa = -1;
    if (cudaDeviceGetAttribute(&numa, cudaDevAttrHostNumaId, t->device) != cudaSuccess) {
        cudaGetLastError();
        numa = -1;
    }
    CUmemAllocationProp prop;
    std::memset(&prop, 0, sizeof(prop));
    prop.type = CU_MEM_ALLOCATION_TYPE_PINNED;
    prop.location.type = numa >= 0 ? CU_MEM_LOCATION_TYPE_HOST_NUMA : CU_MEM_LOCATION_TYPE_HOST;
    prop.location.id = numa >= 0 ? numa : 0;
    size_t gran = 0;
    if (v.granularity(&gran, &prop, CU_MEM_ALLOC_GRANULARITY_RECOMMENDED) != CUDA_SUCCESS || gran == 0)
        return set_error(t, MLKV_ERR_CUDA, "host-tier allocation granularity");
    tr.host_chunk = (size_t)round_up((int64_t)std::min<size_t>(bytes, (size_t)1 << 30), (int64_t)gran);
    const int64_t n = (int64_t)((bytes + tr.host_chunk - 1) / tr.host_chunk);
    tr.host_bytes = (size_t)n * tr.host_chunk;
    tr.host_handles = new (std::nothrow) unsigned long long[n];
    if (!tr.host_handles) return MLKV_ERR_NOMEM;
    CUdeviceptr va = 0;
    if (v.reserve(&va, tr.host_bytes, gran, 0, 0) != CUDA_SUCCESS) {
        tr.host_bytes = 0;
        return set_error(t, MLKV_ERR_NOMEM, "host-tier address reservation of %zu bytes", (size_t)n * tr.host_chunk);
    }
    tr.host_dev = (float*)va;
    for (int64_t i = 0; i < n; ++i) {
        CUmemGenericAllocationHandle h;
        if (injected(g_fail_alloc) || v.create(&h, tr.host_chunk, &prop, 0) != CUDA_SUCCESS)
            return set_error(t, MLKV_ERR_NOMEM, "host tier: %lld of %lld chunks of %zu bytes", (long long)i,
                             (long long)n, tr.host_chunk);
        if (v.map(va + (size_t)i * tr.host_chunk, tr.host_chunk, 0, h, 0) != CUDA_SUCCESS) {
            v.release(h);
            return set_error(t, MLKV_ERR_CUDA, "host tier: mapping chunk %lld", (long long)i);
        }
        tr.host_handles[i] = (unsigned long long)h;
        tr.host_mapped = i + 1;
    }
    CUmemAccessDesc acc;
    std::memset(&acc, 0, sizeof(acc));
    acc.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    acc.location.id = t->device;
    acc.flags = CU_MEM_ACCESS_FLAGS_PROT_READWRITE;
    if (v.set_access(va, tr.host_bytes, &acc, 1) != CUDA_SUCCESS)
        return set_error(t, MLKV_ERR_CUDA, "host tier: device access");
    return MLKV_OK;
}

int next_pow2_int(int x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

// Row-kernel geometry for vector width V (4 needs dim % 4 == 0).
bool make_geom(int d, int V, RowGeom& g) {
    if (V == 4 && d % 4) return false;
    g.d = d;
    g.V = V;
    g.NV = (d + V - 1) / V;
    g.G = next_pow2_int(g.NV) < 32 ? next_pow2_int(g.NV) : 32;
    g.KV = (g.NV + g.G - 1) / g.G;
    if (g.KV > 8) return false;
    g.KV = g.KV <= 1 ? 1 : g.KV <= 2 ? 2 : g.KV <= 4 ? 4 : 8;
    g.dpad = (int)round_up(d, 8);
    g.stride = 2 * g.dpad;
    return true;
}

int bit_width_u64(uint64_t x) {
    int b = 0;
    while (x) {
        ++b;
        x >>= 1;
    }
    return b;
}

constexpr int kScanTile = 4096;

int64_t tiles_of(int64_t n) { return (n + kScanTile - 1) / kScanTile; }

// A call's counters.  In stale-synchronous mode the scope also records, when
// the call has enqueued its work, the event the next apply waits for (any
// call but an apply) or the apply's own event.
struct CallScope {
    CallCounters* cur;
    CallCounters* nxt;
    mlkv_table* t = nullptr;
    cudaStream_t st = nullptr;
    bool apply = false;
    ~CallScope() {
        if (!t) return;
        if (apply) {
            ++t->n_applies;
            cudaEventRecord(t->ev_apply[t->n_applies % t->ring], st);
        } else {
            cudaEventRecord(t->ev_other, st);
            t->other_recorded = 1;
        }
    }
};

bool capturing(cudaStream_t st) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return cs == cudaStreamCaptureStatusActive;
}

// A call's counters: one of two copies, taken in turn; each call zeroes the
// other copy for the next one in its first kernel, and its last kernel to read
// them zeroes its own copy when done (release_counters), so no memset is
// enqueued and a call's copy is zero when it starts even where the host no
// longer knows which copy is next: a captured graph replays a fixed sequence
// of calls, which may be odd in number, without passing through the host.
// (find and export use no counters; every other call's last kernel releases
// them.)
//
// Stale-synchronous mode (staleness_bound s >= 1, Gets and applies on two
// streams): a Get waits for every apply issued more than s applies before it,
// so it may run beside the last s (asynchronous mode, s = INT64_MAX: a Get
// waits for no apply); any other call waits for every apply; an
// apply waits for the call before it on the other stream (the Get whose keys
// it updates) and for the apply before it.  Applies count their own counters,
// so a Get and an apply in flight together never share them.
CallScope begin_call(mlkv_table* t, cudaStream_t st, bool get = false) {
    const int p = t->parity;
    t->parity ^= 1;
    t->last_stream = st;
    if (t->stale > 0 && !(get && t->stale == INT64_MAX)) {
        const int64_t j = get ? t->n_applies - t->stale : t->n_applies;
        if (j >= 1) cudaStreamWaitEvent(st, t->ev_apply[j % t->ring], 0);
    }
    CallScope cs{&t->dstate->cc[p], &t->dstate->cc[p ^ 1]};
    if (t->stale > 0) {
        cs.t = t;
        cs.st = st;
    }
    return cs;
}

CallScope begin_apply(mlkv_table* t, cudaStream_t st) {
    const int p = t->parity_apply;
    t->parity_apply ^= 1;
    t->last_apply_stream = st;
    if (t->stale > 0) {
        if (t->other_recorded) cudaStreamWaitEvent(st, t->ev_other, 0);
        if (t->n_applies >= 1) cudaStreamWaitEvent(st, t->ev_apply[t->n_applies % t->ring], 0);
    }
    CallScope cs{&t->dstate->cca[p], &t->dstate->cca[p ^ 1]};
    if (t->stale > 0) {
        cs.t = t;
        cs.st = st;
        cs.apply = true;
    }
    return cs;
}

// Common argument checks.  Returns MLKV_OK, an error, or -1 for "n == 0: done".
int check_call(mlkv_table* t, const void* keys, int64_t n, const void* buf, bool need_buf, void* stream = nullptr) {
    if (!t) return MLKV_ERR_INVALID;
    if (t->stale > 0 && stream && capturing((cudaStream_t)stream))
        return set_error(t, MLKV_ERR_UNSUPPORTED, "calls of a stale-synchronous table cannot be captured into a graph");
    if (n < 0 || n > t->cfg.max_batch)
        return set_error(t, MLKV_ERR_INVALID, "n = %lld outside [0, max_batch = %lld]", (long long)n,
                         (long long)t->cfg.max_batch);
    if (n > 0 && (!keys || (need_buf && !buf))) return set_error(t, MLKV_ERR_INVALID, "null pointer");
    const uint32_t sticky = *(volatile uint32_t*)t->status_host;
    if (sticky) {
        uint32_t chk[3] = {0, 0, 0};
        if (MLKV_CHECK) cudaMemcpy(chk, t->dstate->chk, sizeof(chk), cudaMemcpyDeviceToHost);
        if (chk[0])  // a bounds-checked build found an index out of range
            return set_error(t, (int)sticky, "sticky device status %u (%s) from an earlier call; check site %u, "
                             "index %u >= bound %u", sticky, mlkv_status_string((int)sticky), chk[0], chk[1], chk[2]);
        return set_error(t, (int)sticky, "sticky device status %u (%s) from an earlier call", sticky,
                         mlkv_status_string((int)sticky));
    }
    return n == 0 ? -1 : MLKV_OK;
}

// Chooses the float4 kernels when every row buffer of the call is 16-byte aligned.
int choose_geom(mlkv_table* t, const void* a, const void* b) {
    const bool al = ((uintptr_t)a % 16 == 0) && ((uintptr_t)b % 16 == 0);
    RowGeom g;
    if (al && make_geom(t->cfg.dim, 4, g)) {
        t->geom = g;
        return MLKV_OK;
    }
    if (make_geom(t->cfg.dim, 1, g)) {
        t->geom = g;
        return MLKV_OK;
    }
    return set_error(t, MLKV_ERR_INVALID, "dim %d needs 16-byte aligned row buffers", t->cfg.dim);
}

}  // namespace

namespace mlkv {

bool take_injected_wait() { return injected(g_fail_wait); }

void timer_before(mlkv_table* t, int kid, cudaStream_t st) {
    KernelTimer& tm = t->timer;
    if (!kid || kid != tm.kernel_id || tm.n_events >= KernelTimer::kMax) return;
    if (!tm.ev) {
        tm.ev = new cudaEvent_t[2 * KernelTimer::kMax];
        for (int i = 0; i < 2 * KernelTimer::kMax; ++i) cudaEventCreate(&tm.ev[i]);
    }
    cudaEventRecord(tm.ev[2 * tm.n_events], st);
}

void timer_after(mlkv_table* t, int kid, cudaStream_t st) {
    KernelTimer& tm = t->timer;
    if (!kid || kid != tm.kernel_id || tm.n_events >= KernelTimer::kMax || !tm.ev) return;
    cudaEventRecord(tm.ev[2 * tm.n_events + 1], st);
    tm.n_events++;
}

int persistent_blocks(mlkv_table* t, const void* kernel, int threads) {
    static std::mutex mu;
    static std::unordered_map<const void*, int> cache;
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(kernel);
    int per_sm;
    if (it != cache.end()) {
        per_sm = it->second;
    } else {
        per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, 0) != cudaSuccess ||
            per_sm < 1)
            per_sm = 1;
        cache[kernel] = per_sm;
    }
    return per_sm * t->num_sms;
}

}  // namespace mlkv

extern "C" {

const char* mlkv_status_string(int s) {
    switch (s) {
        case MLKV_OK: return "ok";
        case MLKV_ERR_INVALID: return "invalid argument";
        case MLKV_ERR_UNSUPPORTED: return "unsupported configuration";
        case MLKV_ERR_CUDA: return "CUDA error";
        case MLKV_ERR_NOMEM: return "out of memory";
        case MLKV_ERR_FULL: return "table full";
        case MLKV_ERR_PROBE_LIMIT: return "probe limit exceeded";
        case MLKV_ERR_NOT_FOUND: return "key not found";
        case MLKV_ERR_TIMEOUT: return "bounded wait in a kernel ran out";
        default: return "unknown status";
    }
}

int mlkv_close(mlkv_table* t) {
    MLKV_RANGE("mlkv_close");
    if (!t) return MLKV_OK;
    cudaDeviceSynchronize();
    if (t->timer.ev) {
        for (int i = 0; i < 2 * KernelTimer::kMax; ++i) cudaEventDestroy(t->timer.ev[i]);
        delete[] t->timer.ev;
    }
    if (t->ev_apply) {
        for (int64_t i = 0; i < t->ring; ++i)
            if (t->ev_apply[i]) cudaEventDestroy(t->ev_apply[i]);
        delete[] t->ev_apply;
    }
    if (t->ev_other) cudaEventDestroy(t->ev_other);
    for (int i = 0; i < 2; ++i) {
        if (t->branch[i]) cudaStreamDestroy(t->branch[i]);
        if (t->ev_join[i]) cudaEventDestroy(t->ev_join[i]);
    }
    if (t->ev_fork) cudaEventDestroy(t->ev_fork);
    if (t->tiered) {
        Tier& tr = t->tier;
        if (tr.la_stream) cudaStreamDestroy(tr.la_stream);
        if (tr.ev_main) cudaEventDestroy(tr.ev_main);
        if (tr.ev_la) cudaEventDestroy(tr.ev_la);
        host_tier_free(tr);
        cudaFree(tr.cache);
        cudaFree(tr.row_loc);
        cudaFree(tr.line_row);
        cudaFree(tr.line_stamp);
        cudaFree(tr.ctr);
        cudaFree(tr.fetch);
        cudaFree(tr.n_fetch);
        cudaFree(tr.la_rows);
        cudaFree(tr.la_fetch);
        cudaFree(tr.la_n_fetch);
    } else {
        cudaFree(t->slots);
    }
    cudaFree(t->index);
    cudaFree(t->dstate);
    cudaFree(t->arena);
    for (int i = 0; i < 2; ++i) {
        cudaFree(t->stage_keys[i]);
        cudaFree(t->stage_vals[i]);
    }
    if (t->status_host) cudaFreeHost(t->status_host);
    delete t;
    return MLKV_OK;
}

int mlkv_open(const mlkv_config* cfg, mlkv_table** out) {
    MLKV_RANGE("mlkv_open");
    if (!cfg || !out) return MLKV_ERR_INVALID;
    *out = nullptr;
    const mlkv_config c = *cfg;
    if (c.dim < 1 || c.dim > MLKV_MAX_DIM || (c.dim > 256 && c.dim % 4)) return MLKV_ERR_INVALID;
    if (c.capacity < 1 || c.capacity >= (1ll << 31) - 2) return MLKV_ERR_INVALID;
    if (c.max_batch < 1 || c.max_batch >= (1ll << 30)) return MLKV_ERR_INVALID;
    if (c.reserved != 0 || (c.flags & ~MLKV_IDENTITY_HASH)) return MLKV_ERR_INVALID;
    if (!(c.init_hi >= c.init_lo)) return MLKV_ERR_INVALID;
    // stale-synchronous and asynchronous modes (MLKV Section 3.3.1): HBM-resident tables
    if (c.staleness_bound < 0) return MLKV_ERR_INVALID;
    if (c.staleness_bound != 0 && c.hbm_cache_rows > 0) return MLKV_ERR_UNSUPPORTED;
    // a tier needs room for two batches' rows at once (a call and a look-ahead in flight)
    if (c.hbm_cache_rows < 0 || c.hbm_cache_rows >= (1ll << 31) - 2) return MLKV_ERR_INVALID;
    if (c.hbm_cache_rows > 0 && c.hbm_cache_rows < 2 * c.max_batch + 64) return MLKV_ERR_INVALID;

    mlkv_table* t = new (std::nothrow) mlkv_table();
    if (!t) return MLKV_ERR_NOMEM;
    std::memset(t, 0, sizeof(*t));
    t->cfg = c;
    auto fail = [&](int code) {
        mlkv_close(t);
        return code;
    };
    if (cudaGetDevice(&t->device) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    if (cudaDeviceGetAttribute(&t->num_sms, cudaDevAttrMultiProcessorCount, t->device) != cudaSuccess)
        return fail(MLKV_ERR_CUDA);
    if (!make_geom(c.dim, c.dim % 4 == 0 ? 4 : 1, t->geom)) return fail(MLKV_ERR_INVALID);

    const int64_t stride = t->geom.stride;
    t->tiered = c.hbm_cache_rows > 0;
    if (!t->tiered) {
        if (dev_alloc(&t->slots, (size_t)c.capacity * stride * sizeof(float)) != cudaSuccess)
            return fail(MLKV_ERR_NOMEM);
    } else {
        Tier& tr = t->tier;
        const int64_t C = c.hbm_cache_rows;
        int rc = host_tier_alloc(t, (size_t)c.capacity * stride * sizeof(float));
        if (rc != MLKV_OK) return fail(rc);
        if (dev_alloc(&tr.cache, (size_t)C * stride * sizeof(float)) != cudaSuccess) return fail(MLKV_ERR_NOMEM);
        if (dev_alloc(&tr.row_loc, (size_t)c.capacity * 4) != cudaSuccess ||
            dev_alloc(&tr.line_row, (size_t)C * 4) != cudaSuccess ||
            dev_alloc(&tr.line_stamp, (size_t)C * 4) != cudaSuccess ||
            dev_alloc(&tr.ctr, 4 * sizeof(unsigned long long)) != cudaSuccess ||
            dev_alloc(&tr.fetch, (size_t)c.max_batch * sizeof(uint2)) != cudaSuccess ||
            dev_alloc(&tr.n_fetch, 4) != cudaSuccess ||
            dev_alloc(&tr.la_rows, (size_t)c.max_batch * 4) != cudaSuccess ||
            dev_alloc(&tr.la_fetch, (size_t)c.max_batch * sizeof(uint2)) != cudaSuccess ||
            dev_alloc(&tr.la_n_fetch, 4) != cudaSuccess)
            return fail(MLKV_ERR_NOMEM);
        if (launch_tier_init(t, 0) != cudaSuccess ||  // row r starts in host slot r
            cudaMemset(tr.line_row, 0xFF, (size_t)C * 4) != cudaSuccess ||
            cudaMemset(tr.line_stamp, 0xFF, (size_t)C * 4) != cudaSuccess ||  // never handed out
            cudaMemset(tr.ctr, 0, 4 * sizeof(unsigned long long)) != cudaSuccess)
            return fail(MLKV_ERR_CUDA);
        if (cudaStreamCreateWithFlags(&tr.la_stream, cudaStreamNonBlocking) != cudaSuccess ||
            cudaEventCreateWithFlags(&tr.ev_main, cudaEventDisableTiming) != cudaSuccess ||
            cudaEventCreateWithFlags(&tr.ev_la, cudaEventDisableTiming) != cudaSuccess)
            return fail(MLKV_ERR_CUDA);
        tr.epoch = 1;
        t->slots = tr.cache;
    }
    // The bound kept: s up to kMaxStaleness, a tighter bound above it (which
    // meets the one asked for), none at INT64_MAX.  A Get waits for the apply
    // issued s applies back, so the ring holds the last s + 1 applies' events
    // (the last one's alone with no bound).
    t->stale = c.staleness_bound == INT64_MAX ? INT64_MAX : std::min<int64_t>(c.staleness_bound, kMaxStaleness);
    t->ring = t->stale == INT64_MAX ? 1 : t->stale + 1;
    if (t->stale > 0) {
        t->ev_apply = new (std::nothrow) cudaEvent_t[t->ring]();
        if (!t->ev_apply) return fail(MLKV_ERR_NOMEM);
        for (int64_t i = 0; i < t->ring; ++i)
            if (cudaEventCreateWithFlags(&t->ev_apply[i], cudaEventDisableTiming) != cudaSuccess)
                return fail(MLKV_ERR_CUDA);
        if (cudaEventCreateWithFlags(&t->ev_other, cudaEventDisableTiming) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    }
    for (int i = 0; i < 2; ++i)
        if (cudaStreamCreateWithFlags(&t->branch[i], cudaStreamNonBlocking) != cudaSuccess ||
            cudaEventCreateWithFlags(&t->ev_join[i], cudaEventDisableTiming) != cudaSuccess)
            return fail(MLKV_ERR_CUDA);
    if (cudaEventCreateWithFlags(&t->ev_fork, cudaEventDisableTiming) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    int64_t nslots = 64;
    while (nslots < 2 * c.capacity) nslots <<= 1;
    if (dev_alloc(&t->index, (size_t)nslots * sizeof(Slot)) != cudaSuccess) return fail(MLKV_ERR_NOMEM);
    if (cudaMemset(t->index, 0xFF, (size_t)nslots * sizeof(Slot)) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    t->index_mask = (unsigned long long)(nslots - 1);
    t->bits_rows = bit_width_u64((uint64_t)c.capacity);
    t->bits_lines = t->tiered ? bit_width_u64((uint64_t)c.hbm_cache_rows) : t->bits_rows;
    t->sort_bits = t->bits_rows;

    if (dev_alloc(&t->dstate, sizeof(DevState)) != cudaSuccess) return fail(MLKV_ERR_NOMEM);
    if (cudaMemset(t->dstate, 0, sizeof(DevState)) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    if (pinned_alloc(&t->status_host, sizeof(uint32_t), cudaHostAllocMapped) != cudaSuccess)
        return fail(MLKV_ERR_NOMEM);
    *t->status_host = 0;
    if (cudaHostGetDevicePointer((void**)&t->status_dev_alias, t->status_host, 0) != cudaSuccess)
        return fail(MLKV_ERR_CUDA);

    // Scratch arena, carved in 256-byte aligned pieces.
    const int64_t B = c.max_batch;
    Scratch& s = t->s;
    s.max_long = long_runs_bound(B);
    s.max_items = long_items_bound(B);
    s.tile_sums_len = std::max<int64_t>(tiles_of(B) + 1, t->num_sms);
    // the sort's tiles: 4096 lookups, 1024 in batches under kSortSmallBatch
    const int64_t sort_tiles = std::max<int64_t>(
        tiles_of(B), (std::min<int64_t>(B, (int64_t)kSortSmallBatch - 1) + kSortTileSmall - 1) / kSortTileSmall);
    struct Piece {
        void** ptr;
        int64_t bytes;
    };
    Piece pieces[] = {
        {(void**)&s.row_of_pos, B * 4},     {(void**)&s.slot_of_pos, B * 4},
        {(void**)&s.memo_key, B * 8},       {(void**)&s.memo_row, B * 4},
        {(void**)&s.miss_pos, B * 4},       {(void**)&s.miss_slot, B * 4},
        {(void**)&s.first_flag, B * 4},     {(void**)&s.rank, B * 4},
        {(void**)&s.sk[0], B * 4},          {(void**)&s.sk[1], B * 4},
        {(void**)&s.sv[0], B * 4},          {(void**)&s.sv[1], B * 4},
        {(void**)&s.tile_sums, s.tile_sums_len * 4},
        {(void**)&s.sort_counts, s.sort_counts_bytes = 512 * sort_tiles * 4},
        {(void**)&s.sort_counts2, 512 * sort_tiles * 4},
        {(void**)&s.sort_offsets, 512 * sort_tiles * 4},
        {(void**)&s.sort_dtot, kSortMaxPasses * 512 * 4},
        {(void**)&s.seg_start, (B + 1) * 4},  {(void**)&s.long_s, s.max_long * 4},
        {(void**)&s.long_e, s.max_long * 4},   {(void**)&s.long_row, s.max_long * 4},
        {(void**)&s.long_base, s.max_long * 4}, {(void**)&s.item_s, s.max_items * 4},
        {(void**)&s.item_e, s.max_items * 4},   {(void**)&s.run_row, B * 4},
        {(void**)&s.big_runs, s.max_long * 4},
        {(void**)&s.short_runs, B * 16},
        {(void**)&s.single_runs, B * 8},
        {(void**)&s.small_runs, B * 16},
        {(void**)&s.small_p3, B * 4},
        {(void**)&s.run_p0, B * 4},
        {(void**)&s.partial, s.max_items * 2 * t->geom.dpad * 4},
    };
    int64_t total = 0;
    for (auto& p : pieces) total += round_up(p.bytes, 256);
    if (dev_alloc(&t->arena, (size_t)total) != cudaSuccess) return fail(MLKV_ERR_NOMEM);
    if (cudaMemset(t->arena, 0, (size_t)total) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    t->arena_bytes = total;
    char* base = (char*)t->arena;
    for (auto& p : pieces) {
        *p.ptr = base;
        base += round_up(p.bytes, 256);
    }
    // no position has a remembered row yet
    if (cudaMemset(s.memo_row, 0xFF, (size_t)B * 4) != cudaSuccess) return fail(MLKV_ERR_CUDA);
    if (cudaDeviceSynchronize() != cudaSuccess) return fail(MLKV_ERR_CUDA);
    *out = t;
    return MLKV_OK;
}

}  // extern "C"

namespace {

// On a tiered table every call first waits for a look-ahead in flight, except
// an apply_grad, which may run beside it (see mlkv_lookahead).
int wait_lookahead(mlkv_table* t, cudaStream_t st) {
    if (t->tiered && capturing(st))
        return set_error(t, MLKV_ERR_UNSUPPORTED, "a tiered table's calls cannot be captured into a graph");
    if (t->tiered && t->tier.la_pending) {
        CK(t, cudaStreamWaitEvent(st, t->tier.ev_la, 0));
        t->tier.la_pending = 0;
    }
    return MLKV_OK;
}

// Rows of the lookups -> cache lines (fetching the missing rows); the row
// kernels that follow use the cache as their slot array.
int tier_map(mlkv_table* t, uint32_t epoch, int strict, int64_t n, cudaStream_t st) {
    CK(t, launch_tier_resolve(t, tier_args(t, epoch, epoch, strict), t->s.row_of_pos, n, t->tier.fetch,
                              t->tier.n_fetch, true, st));
    return MLKV_OK;
}

}  // namespace

extern "C" {

int mlkv_get(mlkv_table* t, const int64_t* d_keys, int64_t n, float* d_out, void* stream) {
    MLKV_RANGE("mlkv_get");
    int rc = check_call(t, d_keys, n, d_out, true, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if ((rc = choose_geom(t, d_out, d_out))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    if (t->tiered) {
        if ((rc = wait_lookahead(t, st))) return rc;
        CallScope cs = begin_call(t, st);
        const uint32_t e = ++t->tier.epoch;
        const bool ins = t->cfg.insert_on_miss != 0;
        CK(t, launch_probe(t, d_keys, n, ins, MemoUse::Save, false, !ins, st, cs.cur, cs.nxt));
        if (ins) CK(t, launch_resolve_misses(t, d_keys, n, MissMode::Init, nullptr, st, cs.cur, true));
        if ((rc = tier_map(t, e, 0, n, st))) return rc;
        CK(t, launch_gather_lines(t, t->s.row_of_pos, n, d_out, st));
        return MLKV_OK;
    }
    CallScope cs = begin_call(t, st, true);
    CK(t, launch_get(t, d_keys, n, d_out, st, cs.cur, cs.nxt));
    if (t->cfg.insert_on_miss) CK(t, launch_resolve_misses(t, d_keys, n, MissMode::Get, d_out, st, cs.cur, true));
    return MLKV_OK;
}

int mlkv_insert(mlkv_table* t, const int64_t* d_keys, int64_t n, void* stream) {
    MLKV_RANGE("mlkv_insert");
    int rc = check_call(t, d_keys, n, nullptr, false, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if ((rc = choose_geom(t, t->slots, t->slots))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    if ((rc = wait_lookahead(t, st))) return rc;
    CallScope cs = begin_call(t, st);
    CK(t, launch_probe(t, d_keys, n, true, MemoUse::None, false, false, st, cs.cur, cs.nxt));
    CK(t, launch_resolve_misses(t, d_keys, n, MissMode::Init, nullptr, st, cs.cur, true));
    return MLKV_OK;
}

// Put, and import (the state too): upsert, the last occurrence of a key wins.
static int put_rows(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_vals, const float* d_state,
                    void* stream) {
    int rc = check_call(t, d_keys, n, d_vals, true, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if ((rc = choose_geom(t, d_vals, d_state ? d_state : d_vals))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    if ((rc = wait_lookahead(t, st))) return rc;
    CallScope cs = begin_call(t, st);
    CK(t, launch_probe(t, d_keys, n, true, MemoUse::None, true, false, st, cs.cur, cs.nxt));
    CK(t, launch_resolve_misses(t, d_keys, n, MissMode::Put, nullptr, st, cs.cur, true));
    if (t->tiered && (rc = tier_map(t, ++t->tier.epoch, 0, n, st))) return rc;
    CK(t, launch_put_scatter(t, d_vals, d_state, n, st));
    return MLKV_OK;
}

int mlkv_put(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_vals, void* stream) {
    MLKV_RANGE("mlkv_put");
    return put_rows(t, d_keys, n, d_vals, nullptr, stream);
}

int mlkv_import(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_rows, const float* d_state,
                void* stream) {
    MLKV_RANGE("mlkv_import");
    return put_rows(t, d_keys, n, d_rows, d_state, stream);
}

int mlkv_dump_keys(mlkv_table* t, int64_t* d_keys_out, int64_t n_rows, void* stream) {
    MLKV_RANGE("mlkv_dump_keys");
    if (!t || n_rows < 0 || (n_rows > 0 && !d_keys_out)) return MLKV_ERR_INVALID;
    if (n_rows == 0) return MLKV_OK;
    cudaStream_t st = (cudaStream_t)stream;
    int rc;
    if ((rc = wait_lookahead(t, st))) return rc;
    CK(t, launch_dump_keys(t, d_keys_out, n_rows, st));
    return MLKV_OK;
}

int mlkv_apply_grad(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_grads, void* stream) {
    MLKV_RANGE("mlkv_apply_grad");
    int rc = check_call(t, d_keys, n, d_grads, true, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if ((rc = choose_geom(t, d_grads, d_grads))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    // A tiered apply issued while a look-ahead is in flight runs beside it: it
    // may only use cache lines of the preceding Get (no insert, no fetch).
    if (t->tiered && capturing(st))
        return set_error(t, MLKV_ERR_UNSUPPORTED, "a tiered table's calls cannot be captured into a graph");
    const bool beside = t->tiered && t->tier.la_pending;
    CallScope cs = begin_apply(t, st);
    // stale-synchronous: a Get may be inserting beside this apply, and its memo
    // may be the next Get's; the apply inserts nothing and probes every key
    const bool ins = t->cfg.insert_on_miss != 0 && !beside && t->stale == 0;
    const MemoUse memo = t->stale ? MemoUse::None : MemoUse::Read;
    // On an HBM-resident table the probe also counts the sort's first pass (the
    // tiered apply sorts cache lines, known only after the probe).
    const FirstCounts fc = first_counts(t, n);
    CK(t, launch_probe(t, d_keys, n, ins, memo, false, !ins, st, cs.cur, cs.nxt, nullptr,
                       t->tiered ? nullptr : &fc));
    if (ins)
        CK(t, launch_resolve_misses(t, d_keys, n, MissMode::Init, nullptr, st, cs.cur, false,
                                    t->tiered ? nullptr : &fc));
    if (t->tiered) {
        const uint32_t e = beside ? t->tier.epoch : ++t->tier.epoch;
        if ((rc = tier_map(t, e, beside ? 1 : 0, n, st))) return rc;
        t->sort_bits = t->bits_lines;
    }
    const uint32_t *srow, *spos;
    const uint32_t sent = (uint32_t)((1ull << t->sort_bits) - 1);  // the sort's key of a lookup without a row
    cudaError_t err = launch_sort_rows(t, n, st, &srow, &spos, !t->tiered);
    if (err == cudaSuccess) err = launch_reduce_apply(t, d_grads, srow, spos, n, sent, st, cs.cur);
    t->sort_bits = t->bits_rows;
    if (err != cudaSuccess) return cuda_error(t, err, "apply_grad launches");
    return MLKV_OK;
}

int mlkv_lookahead(mlkv_table* t, const int64_t* d_keys, int64_t n, void* stream) {
    MLKV_RANGE("mlkv_lookahead");
    int rc = check_call(t, d_keys, n, nullptr, false, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if (!t->tiered) return MLKV_OK;  // every row is resident already
    cudaStream_t st = (cudaStream_t)stream;
    if (capturing(st))
        return set_error(t, MLKV_ERR_UNSUPPORTED, "a tiered table's calls cannot be captured into a graph");
    Tier& tr = t->tier;
    // the look-ahead starts after everything the caller issued before it, and
    // runs on the table's side stream; it is stamped with the next call's epoch
    // and never takes lines stamped by the current one
    CK(t, cudaEventRecord(tr.ev_main, st));
    CK(t, cudaStreamWaitEvent(tr.la_stream, tr.ev_main, 0));
    const uint32_t e = tr.epoch + 1;
    CK(t, launch_probe(t, d_keys, n, false, MemoUse::None, false, false, tr.la_stream, nullptr, nullptr, tr.la_rows));
    CK(t, launch_tier_resolve(t, tier_args(t, e, tr.epoch, 0), tr.la_rows, n, tr.la_fetch, tr.la_n_fetch, false,
                              tr.la_stream));
    CK(t, cudaEventRecord(tr.ev_la, tr.la_stream));
    tr.la_pending = 1;
    return MLKV_OK;
}

int mlkv_find(mlkv_table* t, const int64_t* d_keys, int64_t n, int64_t* d_rows, void* stream) {
    MLKV_RANGE("mlkv_find");
    int rc = check_call(t, d_keys, n, d_rows, true, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    cudaStream_t st = (cudaStream_t)stream;
    if ((rc = wait_lookahead(t, st))) return rc;
    CallScope cs = begin_call(t, st);
    CK(t, launch_find(t, d_keys, n, d_rows, st, cs.nxt));
    return MLKV_OK;
}

int mlkv_export(mlkv_table* t, const int64_t* d_keys, int64_t n, float* d_rows, float* d_state,
                void* stream) {
    MLKV_RANGE("mlkv_export");
    int rc = check_call(t, d_keys, n, d_rows ? (void*)d_rows : (void*)d_state, true, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if ((rc = choose_geom(t, d_rows ? d_rows : d_state, d_state ? d_state : d_rows))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    if ((rc = wait_lookahead(t, st))) return rc;
    CallScope cs = begin_call(t, st);
    CK(t, launch_export(t, d_keys, n, d_rows, d_state, st, cs.nxt));
    return MLKV_OK;
}

int mlkv_dedup(mlkv_table* t, const int64_t* d_keys, int64_t n, int64_t* d_unique_keys,
               int32_t* d_counts, int64_t* d_num_unique, void* stream) {
    MLKV_RANGE("mlkv_dedup");
    if (t && n == 0) {  // nothing to sort: report zero distinct keys
        int rc = check_call(t, d_keys, n, nullptr, false, stream);
        if (rc > 0) return rc;
        if (d_num_unique)
            CK(t, cudaMemsetAsync(d_num_unique, 0, sizeof(int64_t), (cudaStream_t)stream));
        return MLKV_OK;
    }
    int rc = check_call(t, d_keys, n, d_unique_keys, true, stream);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    if (!d_counts || !d_num_unique) return set_error(t, MLKV_ERR_INVALID, "null pointer");
    cudaStream_t st = (cudaStream_t)stream;
    if ((rc = wait_lookahead(t, st))) return rc;
    CallScope cs = begin_call(t, st);
    CK(t, launch_probe(t, d_keys, n, false, MemoUse::None, false, false, st, cs.cur, cs.nxt));
    const uint32_t *srow, *spos;
    CK(t, launch_sort_rows(t, n, st, &srow, &spos));
    CK(t, launch_segments(t, srow, spos, n, st, cs.cur));
    CK(t, launch_dedup_out(t, d_keys, spos, n, d_unique_keys, d_counts, d_num_unique, st, cs.cur));
    return MLKV_OK;
}

// The staging set of a host-buffer call: the applies of a stale-synchronous
// table have their own, since a Get may still be reading its keys beside them.
static int ensure_staging(mlkv_table* t, bool apply, int& set) {
    set = apply && t->stale > 0 ? 1 : 0;
    if (t->stage_keys[set]) return MLKV_OK;
    const size_t kb = (size_t)t->cfg.max_batch * sizeof(int64_t);
    const size_t vb = (size_t)t->cfg.max_batch * t->cfg.dim * sizeof(float);
    if (dev_alloc(&t->stage_keys[set], kb) != cudaSuccess) return set_error(t, MLKV_ERR_NOMEM, "staging keys");
    if (dev_alloc(&t->stage_vals[set], vb) != cudaSuccess) {
        cudaFree(t->stage_keys[set]);
        t->stage_keys[set] = nullptr;
        return set_error(t, MLKV_ERR_NOMEM, "staging values");
    }
    return MLKV_OK;
}

int mlkv_get_host(mlkv_table* t, const int64_t* h_keys, int64_t n, float* h_out, void* stream) {
    MLKV_RANGE("mlkv_get_host");
    int rc = check_call(t, h_keys, n, h_out, true);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    int set;
    if ((rc = ensure_staging(t, false, set))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    CK(t, copy_async(t->stage_keys[set], h_keys, (size_t)n * 8, cudaMemcpyHostToDevice, st));
    if ((rc = mlkv_get(t, t->stage_keys[set], n, t->stage_vals[set], stream))) return rc;
    CK(t, copy_async(h_out, t->stage_vals[set], (size_t)n * t->cfg.dim * 4, cudaMemcpyDeviceToHost, st));
    return MLKV_OK;
}

int mlkv_apply_grad_host(mlkv_table* t, const int64_t* h_keys, int64_t n, const float* h_grads,
                         void* stream) {
    MLKV_RANGE("mlkv_apply_grad_host");
    int rc = check_call(t, h_keys, n, h_grads, true);
    if (rc) return rc < 0 ? MLKV_OK : rc;
    int set;
    if ((rc = ensure_staging(t, true, set))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    CK(t, copy_async(t->stage_keys[set], h_keys, (size_t)n * 8, cudaMemcpyHostToDevice, st));
    CK(t, copy_async(t->stage_vals[set], h_grads, (size_t)n * t->cfg.dim * 4, cudaMemcpyHostToDevice, st));
    return mlkv_apply_grad(t, t->stage_keys[set], n, t->stage_vals[set], stream);
}

int mlkv_sync(mlkv_table* t) {
    MLKV_RANGE("mlkv_sync");
    if (!t) return MLKV_ERR_INVALID;
    CK(t, cudaStreamSynchronize(t->last_stream));
    if (t->last_apply_stream != t->last_stream) CK(t, cudaStreamSynchronize(t->last_apply_stream));
    if (t->tiered) CK(t, cudaStreamSynchronize(t->tier.la_stream));
    uint32_t st = 0;
    CK(t, cudaMemcpy(&st, &t->dstate->status, sizeof(st), cudaMemcpyDeviceToHost));
    if (st) {
        uint32_t chk[3] = {0, 0, 0};
        CK(t, cudaMemcpy(chk, t->dstate->chk, sizeof(chk), cudaMemcpyDeviceToHost));
        if (chk[0])  // a bounds-checked build found an index out of range
            set_error(t, (int)st, "device status %u (%s): check site %u, index %u >= bound %u", st,
                      mlkv_status_string((int)st), chk[0], chk[1], chk[2]);
        else
            set_error(t, (int)st, "device status %u (%s)", st, mlkv_status_string((int)st));
    }
    return (int)st;
}

int mlkv_clear_status(mlkv_table* t) {
    MLKV_RANGE("mlkv_clear_status");
    if (!t) return MLKV_ERR_INVALID;
    CK(t, cudaDeviceSynchronize());
    CK(t, cudaMemset(&t->dstate->status, 0, sizeof(uint32_t)));
    CK(t, cudaMemset(t->dstate->chk, 0, sizeof(t->dstate->chk)));
    // a call that a device error cut short may have left keys half inserted:
    // their slots and the first-occurrence flags go back to idle
    CK(t, cudaMemset(t->s.first_flag, 0, (size_t)t->cfg.max_batch * 4));
    CK(t, launch_reset_pending(t, 0));
    // ... and its counters, which its last kernel did not release
    CK(t, cudaMemset(t->dstate->cc, 0, sizeof(t->dstate->cc)));
    CK(t, cudaMemset(t->dstate->cca, 0, sizeof(t->dstate->cca)));
    // ... and the sort's counts and digit totals, zero between sorts
    CK(t, cudaMemset(t->s.sort_counts, 0, t->s.sort_counts_bytes));
    CK(t, cudaMemset(t->s.sort_counts2, 0, t->s.sort_counts_bytes));
    CK(t, cudaMemset(t->s.sort_dtot, 0, kSortMaxPasses * 512 * 4));
    CK(t, cudaDeviceSynchronize());
    *(volatile uint32_t*)t->status_host = 0;
    t->last_error[0] = 0;
    return MLKV_OK;
}

int64_t mlkv_size(mlkv_table* t) {
    if (!t) return -1;
    if (cudaStreamSynchronize(t->last_stream) != cudaSuccess) return -1;
    if (t->last_apply_stream != t->last_stream && cudaStreamSynchronize(t->last_apply_stream) != cudaSuccess)
        return -1;
    if (t->tiered && cudaStreamSynchronize(t->tier.la_stream) != cudaSuccess) return -1;
    unsigned long long nr = 0;
    if (cudaMemcpy(&nr, &t->dstate->next_row, sizeof(nr), cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
    return (int64_t)nr;
}

int64_t mlkv_last_unique(mlkv_table* t) {
    if (!t) return -1;
    if (cudaStreamSynchronize(t->last_stream) != cudaSuccess) return -1;
    if (t->last_apply_stream != t->last_stream && cudaStreamSynchronize(t->last_apply_stream) != cudaSuccess)
        return -1;
    uint32_t u = 0;
    if (cudaMemcpy(&u, &t->dstate->last_unique, sizeof(u), cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
    return (int64_t)u;
}

int64_t mlkv_launch_count(mlkv_table* t) { return t ? t->launches : -1; }

int mlkv_tier_stats(mlkv_table* t, int64_t* rows_fetched, int64_t* rows_written_back, int64_t* sweep_lines) {
    if (!t || !rows_fetched || !rows_written_back || !sweep_lines) return MLKV_ERR_INVALID;
    *rows_fetched = 0;
    *rows_written_back = 0;
    *sweep_lines = 0;
    if (!t->tiered) return MLKV_OK;
    CK(t, cudaDeviceSynchronize());
    unsigned long long c[4];
    CK(t, cudaMemcpy(c, t->tier.ctr, sizeof(c), cudaMemcpyDeviceToHost));
    *rows_fetched = (int64_t)c[2];
    *rows_written_back = (int64_t)c[3];
    *sweep_lines = (int64_t)c[1];
    return MLKV_OK;
}

int mlkv_time_kernel(mlkv_table* t, int32_t kernel_id) {
    if (!t) return MLKV_ERR_INVALID;
    t->timer.kernel_id = kernel_id;
    t->timer.n_events = 0;
    return MLKV_OK;
}

int mlkv_kernel_time(mlkv_table* t, double* total_ms, int64_t* launches) {
    if (!t || !total_ms || !launches) return MLKV_ERR_INVALID;
    double sum = 0;
    const int n = t->timer.n_events;
    for (int i = 0; i < n; ++i) {
        CK(t, cudaEventSynchronize(t->timer.ev[2 * i + 1]));
        float ms = 0;
        CK(t, cudaEventElapsedTime(&ms, t->timer.ev[2 * i], t->timer.ev[2 * i + 1]));
        sum += ms;
    }
    *total_ms = sum;
    *launches = n;
    t->timer.n_events = 0;
    return MLKV_OK;
}

const char* mlkv_last_error(mlkv_table* t) { return t ? t->last_error : "null table"; }

int mlkv_debug_fail(int32_t kind, int64_t nth) {
    if (nth < 0) return MLKV_ERR_INVALID;
    switch (kind) {
        case MLKV_FAULT_ALLOC: g_fail_alloc.store(nth); return MLKV_OK;
        case MLKV_FAULT_COPY: g_fail_copy.store(nth); return MLKV_OK;
        case MLKV_FAULT_WAIT: g_fail_wait.store(nth); return MLKV_OK;
        default: return MLKV_ERR_INVALID;
    }
}

}  // extern "C"
