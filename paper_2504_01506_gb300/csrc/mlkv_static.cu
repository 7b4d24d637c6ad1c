// Dedup of a batch of raw 64-bit keys that allocates no memory: its working
// arrays live in one file-scope __device__ array of fixed size.  For callers
// that must not allocate device memory when they need the dedup: plugins
// inside an engine that reserved the device's memory up front and owns every
// allocation, and latency-bound loops that ban cudaMalloc / cudaFree because
// those may synchronise the device.  It needs no table.
//
// Work: a stable LSD radix sort of the keys (8 passes of 8 bits: histogram
// per 4096-key tile, one-block scan of the [digit][tile] counts, stable
// scatter), then one block marks run heads and writes each distinct key with
// the length of its run.
#include <mutex>

#include "mlkv_internal.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kItems = 16;
constexpr int kTile = kThreads * kItems;  // 4096
constexpr int kWarps = kThreads / 32;
constexpr int kRadix = 256;
constexpr int kMaxTiles = MLKV_STATIC_MAX_KEYS / kTile;

// Layout of the static scratch (bytes): two key buffers, the tile histograms,
// the run starts.  Every call overwrites all of it that it reads, so nothing
// has to start at zero.
constexpr size_t kKeysBytes = sizeof(unsigned long long) * MLKV_STATIC_MAX_KEYS;
constexpr size_t kHistOff = 2 * kKeysBytes;
constexpr size_t kHistBytes = sizeof(uint32_t) * kRadix * kMaxTiles;
constexpr size_t kSegOff = kHistOff + kHistBytes;
constexpr size_t kScratchBytes = kSegOff + sizeof(uint32_t) * (MLKV_STATIC_MAX_KEYS + 1);

static __device__ __align__(256) unsigned char g_dedup_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// The device address of g_dedup_scratch on the current device, looked up once
// per device (the host-side symbol is not a device address).
int scratch_address(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MLKV_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return MLKV_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_dedup_scratch) != cudaSuccess || !p) return MLKV_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return MLKV_OK;
}

__global__ void __launch_bounds__(kThreads) k_st_hist(const unsigned long long* __restrict__ keys, uint32_t n,
                                                      uint32_t* __restrict__ hist, uint32_t ntiles, int shift) {
    __shared__ uint32_t cnt[kRadix];
    cnt[threadIdx.x] = 0;
    __syncthreads();
    const uint32_t base = blockIdx.x * kTile;
    for (int k = 0; k < kItems; ++k) {
        const uint32_t i = base + k * kThreads + threadIdx.x;
        if (i < n) atomicAdd(&cnt[(uint32_t)(keys[i] >> shift) & (kRadix - 1)], 1u);
    }
    __syncthreads();
    hist[threadIdx.x * ntiles + blockIdx.x] = cnt[threadIdx.x];
}

// One block: exclusive scan of len <= kRadix * kMaxTiles counts, in place.
__global__ void __launch_bounds__(kThreads) k_st_scan(uint32_t* hist, uint32_t len) {
    __shared__ uint32_t warp_sums[kWarps];
    constexpr int per = kRadix * kMaxTiles / kThreads;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    uint32_t v[per];
    uint32_t local = 0;
    for (int k = 0; k < per; ++k) {
        const uint32_t i = threadIdx.x * per + k;
        v[k] = i < len ? hist[i] : 0u;
        local += v[k];
    }
    uint32_t x = local;
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[w] = x;
    __syncthreads();
    uint32_t before = 0;
    for (int i = 0; i < w; ++i) before += warp_sums[i];
    uint32_t run = before + x - local;
    for (int k = 0; k < per; ++k) {
        const uint32_t i = threadIdx.x * per + k;
        if (i < len) hist[i] = run;
        run += v[k];
    }
}

__global__ void __launch_bounds__(kThreads) k_st_scatter(const unsigned long long* __restrict__ kin,
                                                         unsigned long long* __restrict__ kout, uint32_t n,
                                                         const uint32_t* __restrict__ hist, uint32_t ntiles,
                                                         int shift) {
    __shared__ uint32_t wcnt[kWarps][kRadix];
    __shared__ uint32_t gbase[kRadix];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < kWarps * kRadix; i += kThreads) (&wcnt[0][0])[i] = 0;
    gbase[threadIdx.x] = hist[threadIdx.x * ntiles + blockIdx.x];
    __syncthreads();
    const uint32_t base = blockIdx.x * kTile + w * (kItems * 32);
    uint32_t lt;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(lt));
    unsigned long long key[kItems];
    uint32_t rnk[kItems];
    for (int r = 0; r < kItems; ++r) {
        const uint32_t i = base + r * 32 + lane;
        const bool valid = i < n;
        const unsigned long long k = valid ? kin[i] : 0ull;
        const uint32_t dig = (uint32_t)(k >> shift) & (kRadix - 1);
        const uint32_t peers = __match_any_sync(0xffffffffu, valid ? dig : 0xFFFFFFFFu);
        uint32_t before = 0;
        if (valid) before = wcnt[w][dig];
        __syncwarp();
        if (valid && lane == __ffs(peers) - 1) wcnt[w][dig] = before + __popc(peers);
        __syncwarp();
        key[r] = k;
        rnk[r] = valid ? before + __popc(peers & lt) : 0xFFFFFFFFu;
    }
    __syncthreads();
    {
        uint32_t run = 0;
        for (int ww = 0; ww < kWarps; ++ww) {
            const uint32_t c = wcnt[ww][threadIdx.x];
            wcnt[ww][threadIdx.x] = run;
            run += c;
        }
    }
    __syncthreads();
    for (int r = 0; r < kItems; ++r) {
        if (rnk[r] == 0xFFFFFFFFu) continue;
        const uint32_t dig = (uint32_t)(key[r] >> shift) & (kRadix - 1);
        kout[gbase[dig] + wcnt[w][dig] + rnk[r]] = key[r];
    }
}

// One block of 1024 threads: run heads of the sorted keys, their ranks, and
// (distinct key, run length) per run.
__global__ void __launch_bounds__(1024) k_st_runs(const unsigned long long* __restrict__ sorted, uint32_t n,
                                                  uint32_t* __restrict__ seg_start, int64_t* __restrict__ uniq,
                                                  int32_t* __restrict__ counts, int64_t* __restrict__ num) {
    __shared__ uint32_t warp_sums[32];
    __shared__ uint32_t total_s;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const uint32_t per = (n + 1023) / 1024;
    const uint32_t first = threadIdx.x * per;
    uint32_t cnt = 0;
    for (uint32_t k = 0; k < per; ++k) {
        const uint32_t p = first + k;
        cnt += (p < n && (p == 0 || sorted[p] != sorted[p - 1])) ? 1u : 0u;
    }
    uint32_t x = cnt;
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[w] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t s = 0;
        for (int i = 0; i < 32; ++i) {
            const uint32_t c = warp_sums[i];
            warp_sums[i] = s;
            s += c;
        }
        total_s = s;
    }
    __syncthreads();
    uint32_t run = warp_sums[w] + x - cnt;
    for (uint32_t k = 0; k < per; ++k) {
        const uint32_t p = first + k;
        if (p < n && (p == 0 || sorted[p] != sorted[p - 1])) seg_start[run++] = p;
    }
    __syncthreads();
    const uint32_t U = total_s;
    for (uint32_t u = threadIdx.x; u < U; u += blockDim.x) {
        const uint32_t s = seg_start[u];
        const uint32_t e = u + 1 < U ? seg_start[u + 1] : n;
        uniq[u] = (int64_t)sorted[s];
        counts[u] = (int32_t)(e - s);
    }
    if (threadIdx.x == 0) *num = (int64_t)U;
}

}  // namespace

extern "C" int mlkv_dedup_keys_static(const int64_t* d_keys, int64_t n, int64_t* d_unique_keys,
                                      int32_t* d_counts, int64_t* d_num_unique, void* stream) {
    if (n < 0 || n > MLKV_STATIC_MAX_KEYS || !d_num_unique) return MLKV_ERR_INVALID;
    if (n > 0 && (!d_keys || !d_unique_keys || !d_counts)) return MLKV_ERR_INVALID;
    void* scratch = nullptr;
    const int rc = scratch_address(&scratch);
    if (rc != MLKV_OK) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    if (n == 0)
        return cudaMemsetAsync(d_num_unique, 0, sizeof(int64_t), st) == cudaSuccess ? MLKV_OK : MLKV_ERR_CUDA;
    unsigned char* base = static_cast<unsigned char*>(scratch);
    unsigned long long* buf[2] = {reinterpret_cast<unsigned long long*>(base),
                                  reinterpret_cast<unsigned long long*>(base + kKeysBytes)};
    uint32_t* hist = reinterpret_cast<uint32_t*>(base + kHistOff);
    uint32_t* seg = reinterpret_cast<uint32_t*>(base + kSegOff);
    const uint32_t un = (uint32_t)n;
    const uint32_t ntiles = (un + kTile - 1) / kTile;
    const unsigned long long* kin = reinterpret_cast<const unsigned long long*>(d_keys);
    for (int pass = 0; pass < 8; ++pass) {
        const int shift = 8 * pass;
        unsigned long long* kout = buf[pass & 1];
        k_st_hist<<<ntiles, kThreads, 0, st>>>(kin, un, hist, ntiles, shift);
        k_st_scan<<<1, kThreads, 0, st>>>(hist, kRadix * ntiles);
        k_st_scatter<<<ntiles, kThreads, 0, st>>>(kin, kout, un, hist, ntiles, shift);
        kin = kout;
    }
    k_st_runs<<<1, 1024, 0, st>>>(kin, un, seg, d_unique_keys, d_counts, d_num_unique);
    return cudaGetLastError() == cudaSuccess ? MLKV_OK : MLKV_ERR_CUDA;
}
