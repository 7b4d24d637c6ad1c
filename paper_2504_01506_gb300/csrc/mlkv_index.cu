// Hash index kernels: probe / insert-on-miss, the fused Get (probe + row
// gather), deterministic row-id hand-out for new keys, Put, find and export.
//
// Index: open addressing with linear probing over 16-byte slots (two per
// 32-byte sector), at most half full.  A key is published by one 64-bit
// compare-and-swap on an empty slot whose row field already reads
// ROW_PENDING, so a reader never pairs a key with a stale row.
//
// New keys get dense row ids in first-occurrence order (the numbering the
// Get / Put upsert of MLKV Section 3.1 leaves open): while probing, every
// lookup of a new key lowers the slot's `aux` to its batch position with
// atomicMin; the lookup whose position survives is the first occurrence; an
// exclusive scan over first-occurrence flags gives each new key its rank, and
// row = rows handed out so far + rank.
#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

// Device-scope relaxed loads: they see slots published by compare-and-swap in
// the same kernel and still hit in L2 (the coherence point of GPU accesses);
// a volatile load would be a system-scope access.
__device__ __forceinline__ ulonglong2 ld_slot_relaxed(const Slot* s) {
    ulonglong2 v;
    asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];" : "=l"(v.x), "=l"(v.y) : "l"(s) : "memory");
    return v;
}

__device__ __forceinline__ uint32_t ld_u32_relaxed(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Probes `key`.  Returns its row, ROW_ABSENT, or (INSERT only) ROW_PENDING
// with `slot_out` = the slot that now holds the key and the slot's aux
// lowered to `pos`.
template <bool INSERT>
__device__ __forceinline__ uint32_t probe_key(const IndexArgs& ia, unsigned long long key,
                                              uint32_t pos, uint32_t& slot_out) {
    if (key == EMPTY_KEY) {
        record_error(ia.err, MLKV_ERR_INVALID);
        return ROW_ABSENT;
    }
    unsigned long long s = (ia.identity_hash ? key : hash_key(key)) & ia.mask;
    for (int i = 0; i < PROBE_LIMIT; ++i) {
        ulonglong2 v = INSERT ? ld_slot_relaxed(ia.index + s)
                              : __ldg(reinterpret_cast<const ulonglong2*>(ia.index + s));
        if (v.x == key) {
            uint32_t row = (uint32_t)v.y;
            slot_out = (uint32_t)s;
            if (row != ROW_PENDING || !INSERT) return row == ROW_PENDING ? ROW_ABSENT : row;
            atomicMin(&ia.index[s].aux, pos);
            return ROW_PENDING;
        }
        if (v.x == EMPTY_KEY) {
            if (!INSERT) return ROW_ABSENT;
            unsigned long long old = atomicCAS(&ia.index[s].key, EMPTY_KEY, key);
            if (old == EMPTY_KEY || old == key) {
                slot_out = (uint32_t)s;
                uint32_t row = ld_u32_relaxed(&ia.index[s].row);
                if (row != ROW_PENDING) return row;
                atomicMin(&ia.index[s].aux, pos);
                return ROW_PENDING;
            }
            // another key took this slot first: keep probing
        }
        s = (s + 1) & ia.mask;
    }
    record_error(ia.err, MLKV_ERR_PROBE_LIMIT);
    return ROW_ABSENT;
}

// Appends (pos, slot) to the miss list with one atomic per converged group of
// lanes.  The list holds at most one entry per lookup (n): an entry past that
// could only come from a counter left set, and is not written.
__device__ __forceinline__ void append_miss(CallCounters* cur, uint32_t* miss_pos,
                                            uint32_t* miss_slot, uint32_t pos, uint32_t slot, uint32_t n) {
    const unsigned m = __activemask();
    const int lane = threadIdx.x & 31;
    const int leader = __ffs(m) - 1;
    uint32_t base = 0;
    if (lane == leader) base = atomicAdd(&cur->n_miss, (uint32_t)__popc(m));
    base = __shfl_sync(m, base, leader);
    const uint32_t i = base + __popc(m & lanemask_lt());
    if (i < n) {
        miss_pos[i] = pos;
        miss_slot[i] = slot;
    }
}

__device__ __forceinline__ void zero_counters(CallCounters* nxt) {
    if (nxt && blockIdx.x == 0 && threadIdx.x < sizeof(CallCounters) / 4)
        reinterpret_cast<uint32_t*>(nxt)[threadIdx.x] = 0u;
}

struct RowArgs {
    float* slots;
    int stride;
    int dpad;
    int d;
    int NV;
    int G;
};

RowArgs row_args(mlkv_table* t) {
    return RowArgs{t->slots, t->geom.stride, t->geom.dpad, t->geom.d, t->geom.NV, t->geom.G};
}

IndexArgs index_args(mlkv_table* t) {
    return IndexArgs{t->index, t->index_mask, (t->cfg.flags & MLKV_IDENTITY_HASH) ? 1u : 0u,
                     ErrSink{&t->dstate->status, t->status_dev_alias}};
}

// ---------------------------------------------------------------------------
// row_of_pos[p] (and the slot) for every position.  Each thread takes
// kProbeKeys lookups spaced a block apart, so that their loads are in flight
// together (the probe is latency-bound: a key load, then a random slot load).
// With CT > 0 (the gradient apply on an HBM-resident table) a block of CT
// threads covers one tile of the sort (CT * kProbeKeys lookups: 1024 threads
// for 4096-lookup tiles, 256 for 1024) and also counts the first sort pass's
// digits of its rows (see FirstCounts).
constexpr int kProbeKeys = 4;

template <bool INSERT, int CT>
__global__ void __launch_bounds__(CT ? CT : 256) k_probe(IndexArgs ia, const int64_t* __restrict__ keys,
                                               uint32_t n, uint32_t* __restrict__ row_of_pos,
                                               uint32_t* __restrict__ slot_of_pos,
                                               uint32_t* miss_pos, uint32_t* miss_slot,
                                               CallCounters* cur, CallCounters* nxt,
                                               int report_absent, Memo memo, int memo_use, FirstCounts fc) {
    constexpr bool COUNT = CT > 0;
    static_assert(!COUNT || kProbeKeys * CT == kSortTile || kProbeKeys * CT == kSortTileSmall,
                  "a counting block covers one sort tile");
    pdl_enter();
    zero_counters(nxt);
    __shared__ uint32_t hist[COUNT ? kSortMaxRadix : 1];
    if (COUNT) {
        for (int d = threadIdx.x; d < fc.radix; d += blockDim.x) hist[d] = 0u;
        __syncthreads();
    }
    const uint32_t base = blockIdx.x * (blockDim.x * kProbeKeys) + threadIdx.x;
    unsigned long long k[kProbeKeys];
    uint32_t known[kProbeKeys];
#pragma unroll
    for (int j = 0; j < kProbeKeys; ++j) {
        const uint32_t p = base + j * blockDim.x;
        k[j] = p < n ? (unsigned long long)__ldg(keys + p) : 0ull;
        known[j] = ROW_PENDING;
        if (memo_use == (int)MemoUse::Read && p < n) {
            const uint32_t r = memo.row[p];  // loaded beside the key it belongs to
            if ((unsigned long long)memo.key[p] == k[j]) known[j] = r;
        }
    }
#pragma unroll
    for (int j = 0; j < kProbeKeys; ++j) {
        const uint32_t p = base + j * blockDim.x;
        if (p >= n) continue;
        uint32_t row = known[j];
        if (row >= ROW_ABSENT) {  // not the row the last Get found for this key here: probe
            uint32_t slot = 0;
            row = probe_key<INSERT>(ia, k[j], p, slot);
            if (!INSERT && report_absent && row == ROW_ABSENT) record_error(ia.err, MLKV_ERR_NOT_FOUND);
            if (slot_of_pos) slot_of_pos[p] = slot;
            if (INSERT && row == ROW_PENDING) append_miss(cur, miss_pos, miss_slot, p, slot, n);
            if (memo_use == (int)MemoUse::Save) {
                memo.key[p] = (int64_t)k[j];
                memo.row[p] = row;
            }
        }
        row_of_pos[p] = row;
        // a lookup of a new key is counted by the miss kernel, once it has its row
        if (COUNT && row != ROW_PENDING)
            atomicAdd(&hist[(row >= ROW_ABSENT ? fc.sent : row) & (uint32_t)(fc.radix - 1)], 1u);
    }
    if (COUNT) {
        __syncthreads();
        for (int d = threadIdx.x; d < fc.radix; d += blockDim.x) {
            const uint32_t c = hist[d];
            fc.counts[(size_t)d * fc.ntiles + blockIdx.x] = c;
            if (c) atomicAdd(fc.dtot + d, c);
        }
    }
}

// Group-cooperative copy of one row (or NaN) into dst.
template <int V, int KV>
__device__ __forceinline__ void copy_row(const float* __restrict__ src, float* __restrict__ dst,
                                         int NV, int G, int glane, bool absent) {
    using VT = typename Vec<V>::T;
    const VT* s = reinterpret_cast<const VT*>(src);
    VT* o = reinterpret_cast<VT*>(dst);
#pragma unroll
    for (int k = 0; k < KV; ++k) {
        const int j = glane + G * k;
        if (j < NV) __stcs(o + j, absent ? Vec<V>::nan() : __ldg(s + j));
    }
}

// The fused Get: each warp probes 32 consecutive lookups (one per lane), then
// its lane groups gather the 32 rows with vector loads, streaming the output.
// Lookups of new keys are left to the miss path.
// Tuning (set at build time): minimum resident blocks per SM for the Get
// kernel's register allocation, and rows each lane group has in flight.
#ifndef MLKV_GET_MIN_BLOCKS
#define MLKV_GET_MIN_BLOCKS 8
#endif
#ifndef MLKV_GET_ROWS_IN_FLIGHT
#define MLKV_GET_ROWS_IN_FLIGHT 1
#endif

template <int V, int KV, bool INSERT>
__global__ void __launch_bounds__(256, MLKV_GET_MIN_BLOCKS) k_get(IndexArgs ia, RowArgs ra,
                                             const int64_t* __restrict__ keys, uint32_t n,
                                             float* __restrict__ out, uint32_t* miss_pos,
                                             uint32_t* miss_slot, CallCounters* cur,
                                             CallCounters* nxt, Memo memo) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    zero_counters(nxt);
    const int lane = threadIdx.x & 31;
    const uint32_t base = (blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5)) * 32u;
    if (base >= n) return;  // warp-uniform
    const uint32_t p = base + lane;
    uint32_t row = ROW_PENDING;  // lanes past the end skip the gather
    if (p < n) {
        uint32_t slot = 0;
        const int64_t key = keys[p];
        row = probe_key<INSERT>(ia, (unsigned long long)key, p, slot);
        if (INSERT && row == ROW_PENDING) append_miss(cur, miss_pos, miss_slot, p, slot, n);
        if (!INSERT && row == ROW_ABSENT) record_error(ia.err, MLKV_ERR_NOT_FOUND);
        memo.key[p] = key;
        memo.row[p] = row;
    }
    const int G = ra.G, R = 32 / G, glane = lane & (G - 1), gid = lane / G;
    constexpr int UNR = KV >= MLKV_GET_ROWS_IN_FLIGHT ? 1 : MLKV_GET_ROWS_IN_FLIGHT / KV;
    for (int it0 = 0; it0 < G; it0 += UNR) {
        VT v[UNR][KV];
        uint32_t rr[UNR];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            const int q = (it0 + u) * R + gid;
            const uint32_t r = __shfl_sync(0xffffffffu, row, q & 31);
            rr[u] = (it0 + u < G) ? r : ROW_PENDING;
            if (rr[u] < ROW_ABSENT) {
                const VT* src = reinterpret_cast<const VT*>(ra.slots + (size_t)rr[u] * ra.stride);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (j < ra.NV) v[u][k] = __ldg(src + j);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            if (rr[u] == ROW_PENDING) continue;
            const int q = (it0 + u) * R + gid;
            VT* dst = reinterpret_cast<VT*>(out + (size_t)(base + q) * ra.d);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int j = glane + G * k;
                if (j < ra.NV) __stcs(dst + j, rr[u] == ROW_ABSENT ? Vec<V>::nan() : v[u][k]);
            }
        }
    }
}

// The Get with its rows moved by the SM's asynchronous copies, for calls of
// fewer than kBulkMaxBatch lookups (rows of at most kBulkRowBytes, 16-byte
// aligned buffers).  Each warp probes kBulkRows consecutive lookups as k_get
// does, then copies their rows into its shared-memory stage with cp.async (16
// bytes a lane, L2 only; no registers hold rows in flight, so all of them are
// in flight at once), and writes the stage to the output with one bulk store:
// the output rows are contiguous.  The store runs on while the warp probes its
// next lookups; the stage is reused once the store has read it.  Rows of new
// keys are left to the miss path, which writes their output rows after this
// kernel.  Measured against k_get: faster where a call is too small to fill
// the GPU with k_get's warps (latency-bound: 200k lookups, 45 -> 37 us),
// slower on millions of lookups (194 -> 205 us), where k_get's 64 warps a SM
// beat the few warps the stages leave room for.
#ifndef MLKV_GET_BULK
#define MLKV_GET_BULK 1
#endif
#ifndef MLKV_GET_BULK_MAX_BATCH
#define MLKV_GET_BULK_MAX_BATCH (1u << 19)
#endif
constexpr uint32_t kBulkMaxBatch = MLKV_GET_BULK_MAX_BATCH;
constexpr int kBulkThreads = 128;  // 4 warps
constexpr uint32_t kBulkRowBytes = 512;
#ifndef MLKV_GET_BULK_ROWS
#define MLKV_GET_BULK_ROWS 8
#endif
constexpr uint32_t kBulkRows = MLKV_GET_BULK_ROWS;  // lookups a warp takes at a time (its stage: their rows)

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gmem_src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Bulk copy of `bytes` (a multiple of 16; both addresses 16-byte aligned) from
// shared memory to global memory, as one bulk group.
__device__ __forceinline__ void bulk_store(void* gdst, const void* ssrc, uint32_t bytes) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(ssrc);
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n\tcp.async.bulk.commit_group;"
                 ::"l"(gdst), "r"(s), "r"(bytes) : "memory");
}

template <bool INSERT>
__global__ void __launch_bounds__(kBulkThreads) k_get_bulk(IndexArgs ia, RowArgs ra, const int64_t* __restrict__ keys,
                                                           uint32_t n, float* __restrict__ out, uint32_t* miss_pos,
                                                           uint32_t* miss_slot, CallCounters* cur, CallCounters* nxt,
                                                           Memo memo) {
    pdl_enter();
    zero_counters(nxt);
    extern __shared__ __align__(128) unsigned char smem[];
    constexpr int kWarps = kBulkThreads / 32;
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const uint32_t nvec = (uint32_t)ra.d >> 2;  // 16-byte vectors per row
    const uint32_t rowbytes = nvec * 16u;
    float4* stage = reinterpret_cast<float4*>(smem + (size_t)wib * kBulkRows * rowbytes);
    uint32_t* srow = reinterpret_cast<uint32_t*>(smem + (size_t)kWarps * kBulkRows * rowbytes) + wib * 32;
    const float4 nan4 = Vec<4>::nan();
    const uint32_t nwarps = gridDim.x * kWarps;
    bool stored = false;  // a bulk store of this warp's stage is in flight
    for (uint32_t base = (blockIdx.x * kWarps + wib) * kBulkRows; base < n; base += nwarps * kBulkRows) {
        const uint32_t p = base + lane;
        uint32_t row = ROW_PENDING;
        if (lane < (int)kBulkRows && p < n) {
            uint32_t slot = 0;
            const int64_t key = keys[p];
            row = probe_key<INSERT>(ia, (unsigned long long)key, p, slot);
            if (INSERT && row == ROW_PENDING) append_miss(cur, miss_pos, miss_slot, p, slot, n);
            if (!INSERT && row == ROW_ABSENT) record_error(ia.err, MLKV_ERR_NOT_FOUND);
            memo.key[p] = key;
            memo.row[p] = row;
        }
        const uint32_t cnt = min(kBulkRows, n - base);
        if (stored && lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        __syncwarp();
        srow[lane] = row;
        __syncwarp();
        for (uint32_t i = lane; i < cnt * nvec; i += 32) {
            const uint32_t q = i / nvec, c = i - q * nvec;
            const uint32_t r = srow[q];
            if (r < ROW_ABSENT)
                cp_async16(stage + i, reinterpret_cast<const float4*>(ra.slots + (size_t)r * ra.stride) + c);
            else if (r == ROW_ABSENT)
                stage[i] = nan4;  // a new key's row (ROW_PENDING) is written by the miss path later
        }
        cp_async_wait_all();
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the stage, for the bulk store
        __syncwarp();
        if (lane == 0) bulk_store(out + (size_t)base * ra.d, stage, cnt * rowbytes);
        stored = true;
    }
    if (stored && lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ---------------------------------------------------------------------------
// The miss path: new keys of a call get rows.  One kernel, one block per SM.
// In steady-state training nothing misses and every block returns at once; a
// call with misses runs four phases separated by grid barriers:
//   1. flag the first occurrence of each new key (the lookup whose position
//      survived in the slot's aux);
//   2. rank the flags: an exclusive scan over the call's positions, block b
//      owning positions [b * per, (b + 1) * per);
//   3. each first occurrence takes row = rows handed out so far + rank and
//      writes its init row (not for Put) and state_init;
//   4. every missed lookup reads its key's row (a Get gathers it into its
//      output), flags and the slot's aux go back to idle, the row counter
//      advances.
// Data written by other blocks within the kernel is read from L2 (ld.cg).
constexpr int kMissThreads = 512;
constexpr int kMissWarps = kMissThreads / 32;
constexpr uint32_t kBarrierSpins = 1u << 21;  // with its L2 load and 100 ns sleep, 1-2 s a barrier

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Every block of the grid arrives at `ctr` (zero at the call's start) and waits
// until all have.  Only blocks of this one grid wait here, and the kernel lets
// the next kernel launch only after its last barrier, so every block of the
// grid (one per SM) can become resident.  The wait is bounded: a spin that runs
// out records MLKV_ERR_TIMEOUT and the block returns (false).
// (`extra` is 0; mlkv_debug_fail's wait injection makes it 1, a count that
// no grid reaches, so that the wait runs out.)
__device__ bool grid_barrier(uint32_t* ctr, uint32_t extra, const ErrSink& err) {
    __shared__ int ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        ok = 1;
        __threadfence();
        atomicAdd(ctr, 1u);
        uint32_t spins = 0;
        while (ld_acquire_u32(ctr) < gridDim.x + extra) {
            if (++spins > kBarrierSpins) {
                record_error(err, MLKV_ERR_TIMEOUT);
                ok = 0;
                break;
            }
            __nanosleep(100);
        }
        __threadfence();
    }
    __syncthreads();
    return ok != 0;
}

// Sum over the block of one value per thread.
__device__ __forceinline__ uint32_t miss_block_sum(uint32_t v) {
    __shared__ uint32_t part[kMissWarps];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) part[w] = v;
    __syncthreads();
    uint32_t t = 0;
#pragma unroll
    for (int k = 0; k < kMissWarps; ++k) t += part[k];
    return t;
}

// Exclusive scan over the block of one value per thread; *total = the sum.
__device__ __forceinline__ uint32_t miss_block_scan(uint32_t v, uint32_t& total) {
    __shared__ uint32_t part[kMissWarps];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();
    if (lane == 31) part[w] = x;
    __syncthreads();
    uint32_t before = 0;
    total = 0;
#pragma unroll
    for (int k = 0; k < kMissWarps; ++k) {
        if (k < w) before += part[k];
        total += part[k];
    }
    return before + x - v;
}

template <int V, int KV>
__global__ void __launch_bounds__(kMissThreads) k_miss(IndexArgs ia, RowArgs ra, const int64_t* __restrict__ keys,
                                                       uint32_t n, const uint32_t* __restrict__ miss_pos,
                                                       const uint32_t* __restrict__ miss_slot,
                                                       uint32_t* __restrict__ flag, uint32_t* __restrict__ rank,
                                                       uint32_t* __restrict__ block_sums,
                                                       uint32_t* __restrict__ row_of_pos, float* __restrict__ out,
                                                       CallCounters* cur, DevState* ds,
                                                       unsigned long long capacity, int init_row,
                                                       unsigned long long seed, float lo, float span,
                                                       float state_init, uint32_t bar_extra, int release,
                                                       FirstCounts fc) {
    // waits for the kernel before it, like every kernel; lets the next one
    // launch only once the grid barriers are behind it (see grid_barrier)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const uint32_t m = min(cur->n_miss, n);  // never more misses than lookups
    if (m == 0) {
        if (release) release_counters(cur, gridDim.x);
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        return;
    }
    using VT = typename Vec<V>::T;
    const uint32_t nthreads = gridDim.x * blockDim.x;
    const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
    const int G = ra.G, glane = threadIdx.x & (G - 1);
    const uint32_t group = tid / G, ngroups = nthreads / G;
    // A block whose wait ran out returns at once; the first sort pass's counts
    // (an apply's) still get its share of the missed lookups, which keep no row
    // (the phase-4 share, so that every lookup is counted once).
    auto give_up = [&]() {
        if (fc.counts && glane == 0)
            for (uint32_t i = group; i < m; i += ngroups) {
                const uint32_t p = miss_pos[i];
                const uint32_t dig = fc.sent & (uint32_t)(fc.radix - 1);
                atomicAdd(&fc.counts[(size_t)dig * fc.ntiles + (p >> fc.tile_shift)], 1u);
                atomicAdd(fc.dtot + dig, 1u);
            }
    };
    // 1. first occurrences
    for (uint32_t i = tid; i < m; i += nthreads) {
        const uint32_t p = miss_pos[i];
        if (ia.index[miss_slot[i]].aux == p) flag[p] = 1u;
    }
    if (!grid_barrier(&cur->bar[0], bar_extra, ia.err)) return give_up();
    // 2. ranks: the first occurrences at earlier positions
    const uint32_t per = (n + gridDim.x - 1) / gridDim.x;
    const uint32_t p_lo = min(n, blockIdx.x * per), p_hi = min(n, p_lo + per);
    uint32_t cnt = 0;
    for (uint32_t p = p_lo + threadIdx.x; p < p_hi; p += blockDim.x) cnt += __ldcg(flag + p);
    const uint32_t mine = miss_block_sum(cnt);
    if (threadIdx.x == 0) block_sums[blockIdx.x] = mine;
    if (!grid_barrier(&cur->bar[1], bar_extra, ia.err)) return give_up();
    uint32_t b_before = 0;
    for (uint32_t b = threadIdx.x; b < blockIdx.x; b += blockDim.x) b_before += __ldcg(block_sums + b);
    uint32_t run = miss_block_sum(b_before);
    for (uint32_t p0 = p_lo; p0 < p_hi; p0 += blockDim.x) {  // uniform
        const uint32_t p = p0 + threadIdx.x;
        const uint32_t f = p < p_hi ? __ldcg(flag + p) : 0u;
        uint32_t tot;
        const uint32_t ex = miss_block_scan(f, tot);
        if (f) rank[p] = run + ex;
        run += tot;
    }
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) cur->n_new = run;  // every first occurrence
    if (!grid_barrier(&cur->bar[2], bar_extra, ia.err)) return give_up();
    // 3. rows of the first occurrences
    const unsigned long long next = ds->next_row;
    for (uint32_t i = group; i < m; i += ngroups) {
        const uint32_t p = miss_pos[i], s = miss_slot[i];
        if (ia.index[s].aux != p) continue;
        const unsigned long long r = next + __ldcg(rank + p);
        if (r >= capacity) {
            if (glane == 0) record_error(ia.err, MLKV_ERR_FULL);
            continue;
        }
        const unsigned long long key = (unsigned long long)keys[p];
        float* w = ra.slots + (size_t)r * ra.stride;
        VT* wv = reinterpret_cast<VT*>(w);
        VT* gv = reinterpret_cast<VT*>(w + ra.dpad);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j >= ra.NV) continue;
            if (init_row) {
                float e[V];
#pragma unroll
                for (int c = 0; c < V; ++c) e[c] = init_element(seed, key, (uint32_t)(j * V + c), lo, span);
                wv[j] = Vec<V>::from(e);
            }
            gv[j] = Vec<V>::splat(state_init);
        }
        if (glane == 0) ia.index[s].row = (uint32_t)r;
    }
    if (!grid_barrier(&cur->bar[3], bar_extra, ia.err)) return give_up();
    // 4. every missed lookup takes its key's row
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        const unsigned long long nr = next + __ldcg(&cur->n_new);
        ds->next_row = nr < capacity ? nr : capacity;
    }
    for (uint32_t i = group; i < m; i += ngroups) {
        const uint32_t p = miss_pos[i], s = miss_slot[i];
        const uint32_t r0 = ld_u32_relaxed(&ia.index[s].row);
        const uint32_t r = r0 == ROW_PENDING ? ROW_ABSENT : r0;
        if (glane == 0) {
            if (row_of_pos) row_of_pos[p] = r;
            flag[p] = 0u;
            ia.index[s].aux = AUX_IDLE;
            if (fc.counts) {  // the first sort pass's count of this lookup's digit in its tile
                const uint32_t dig = (r >= ROW_ABSENT ? fc.sent : r) & (uint32_t)(fc.radix - 1);
                atomicAdd(&fc.counts[(size_t)dig * fc.ntiles + (p >> fc.tile_shift)], 1u);
                atomicAdd(fc.dtot + dig, 1u);
            }
        }
        if (out)
            copy_row<V, KV>(ra.slots + (size_t)(r == ROW_ABSENT ? 0 : r) * ra.stride,
                            out + (size_t)p * ra.d, ra.NV, G, glane, r == ROW_ABSENT);
    }
    if (release) release_counters(cur, gridDim.x);
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Put 1/2: the last occurrence of each key wins: aux = min over its
// occurrences of (0xFFFFFFFE - p).
__global__ void k_put_mark(Slot* __restrict__ index, const uint32_t* __restrict__ row_of_pos,
                           const uint32_t* __restrict__ slot_of_pos, uint32_t n) {
    pdl_enter();
    const uint32_t p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n || row_of_pos[p] >= ROW_ABSENT) return;
    atomicMin(&index[slot_of_pos[p]].aux, 0xFFFFFFFEu - p);
}

// Put 2/2: the winning occurrence writes the row and puts aux back to idle.
template <int V, int KV>
__global__ void __launch_bounds__(256) k_put_scatter(Slot* __restrict__ index, RowArgs ra,
                                                     const uint32_t* __restrict__ row_of_pos,
                                                     const uint32_t* __restrict__ slot_of_pos,
                                                     const float* __restrict__ vals,
                                                     const float* __restrict__ state, uint32_t n) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    const int lane = threadIdx.x & 31, G = ra.G, R = 32 / G, glane = lane & (G - 1), gid = lane / G;
    const uint32_t warp = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const uint32_t nwarps = gridDim.x * (blockDim.x >> 5);
    for (uint32_t b = warp * R; b < n; b += nwarps * R) {  // warp-uniform
        const uint32_t p = b + gid;
        bool win = false;
        uint32_t r = 0, s = 0;
        if (p < n) {
            r = row_of_pos[p];
            s = slot_of_pos[p];
            win = r < ROW_ABSENT && index[s].aux == 0xFFFFFFFEu - p;
        }
        __syncwarp();
        if (win) {
            const VT* src = reinterpret_cast<const VT*>(vals + (size_t)p * ra.d);
            VT* dst = reinterpret_cast<VT*>(ra.slots + (size_t)r * ra.stride);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int j = glane + G * k;
                if (j < ra.NV) dst[j] = __ldg(src + j);
            }
            if (state) {  // import: the state too
                const VT* ssrc = reinterpret_cast<const VT*>(state + (size_t)p * ra.d);
                VT* sdst = reinterpret_cast<VT*>(ra.slots + (size_t)r * ra.stride + ra.dpad);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (j < ra.NV) sdst[j] = __ldg(ssrc + j);
                }
            }
            if (glane == 0) index[s].aux = AUX_IDLE;
        }
    }
}

__global__ void __launch_bounds__(256) k_find(IndexArgs ia, const int64_t* __restrict__ keys,
                                              uint32_t n, int64_t* __restrict__ rows,
                                              CallCounters* nxt) {
    pdl_enter();
    zero_counters(nxt);
    const uint32_t p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n) return;
    uint32_t slot = 0;
    const uint32_t r = probe_key<false>(ia, (unsigned long long)keys[p], p, slot);
    rows[p] = r >= ROW_ABSENT ? -1 : (int64_t)r;
}

// Export: like Get without insertion, copying row and/or state.
// With a tier, a row is read from its cache line when it has one, else from
// its host slot.
struct ExportTier {
    const uint32_t* row_loc;
    const float* cache;
    const float* host;
};

template <int V, int KV>
__global__ void __launch_bounds__(256) k_export(IndexArgs ia, RowArgs ra,
                                                const int64_t* __restrict__ keys, uint32_t n,
                                                float* __restrict__ rows_out,
                                                float* __restrict__ state_out, CallCounters* nxt,
                                                ExportTier et) {
    pdl_enter();
    zero_counters(nxt);
    const int lane = threadIdx.x & 31;
    const uint32_t base = (blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5)) * 32u;
    if (base >= n) return;
    const uint32_t p = base + lane;
    uint32_t row = ROW_PENDING;
    if (p < n) {
        uint32_t slot = 0;
        row = probe_key<false>(ia, (unsigned long long)keys[p], p, slot);
    }
    const int G = ra.G, R = 32 / G, glane = lane & (G - 1), gid = lane / G;
    for (int it = 0; it < G; ++it) {
        const int q = it * R + gid;
        const uint32_t r = __shfl_sync(0xffffffffu, row, q);
        if (r == ROW_PENDING) continue;
        const float* src = ra.slots + (size_t)(r == ROW_ABSENT ? 0 : r) * ra.stride;
        if (et.row_loc && r != ROW_ABSENT) {
            const uint32_t l = et.row_loc[r];
            src = l < LOC_HOST ? et.cache + (size_t)l * ra.stride : et.host + (size_t)(l & ~LOC_HOST) * ra.stride;
        }
        if (rows_out) copy_row<V, KV>(src, rows_out + (size_t)(base + q) * ra.d, ra.NV, G, glane, r == ROW_ABSENT);
        if (state_out)
            copy_row<V, KV>(src + ra.dpad, state_out + (size_t)(base + q) * ra.d, ra.NV, G, glane, r == ROW_ABSENT);
    }
}

// Dispatch over (V, KV) for the row kernels.
template <template <int, int> class F, typename... A>
cudaError_t dispatch_row(const RowGeom& g, A&&... a) {
    if (g.V == 4) {
        switch (g.KV) {
            case 1: return F<4, 1>::run(a...);
            case 2: return F<4, 2>::run(a...);
            case 4: return F<4, 4>::run(a...);
            default: return F<4, 8>::run(a...);
        }
    }
    switch (g.KV) {
        case 1: return F<1, 1>::run(a...);
        case 2: return F<1, 2>::run(a...);
        case 4: return F<1, 4>::run(a...);
        default: return F<1, 8>::run(a...);
    }
}

inline unsigned grid_for(int64_t items, int per_block) {
    return (unsigned)((items + per_block - 1) / per_block);
}

inline unsigned capped_grid(mlkv_table* t, int64_t items, int per_block, int per_sm) {
    int64_t g = (items + per_block - 1) / per_block;
    int64_t cap = (int64_t)t->num_sms * per_sm;
    if (g > cap) g = cap;
    return (unsigned)(g < 1 ? 1 : g);
}

// Blocks per SM and shared memory of k_get_bulk for rows of `rowbytes`.
template <bool INSERT>
int bulk_grid(mlkv_table* t, size_t smem, int64_t n) {
    static int configured[2] = {0, 0};
    static int per_sm_cache[kBulkRowBytes / 16 + 1] = {0};
    const int kind = INSERT ? 1 : 0;
    if (!configured[kind]) {
        cudaFuncSetAttribute(k_get_bulk<INSERT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(4 * kBulkRows * kBulkRowBytes + 4 * 32 * 4));
        configured[kind] = 1;
    }
    const size_t idx = (smem - 4 * 32 * 4) / (4 * kBulkRows * 16);
    int per_sm = idx < sizeof(per_sm_cache) / sizeof(int) ? per_sm_cache[idx] : 0;
    if (per_sm == 0) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_get_bulk<INSERT>, kBulkThreads, smem) !=
                cudaSuccess || per_sm < 1)
            per_sm = 1;
        if (idx < sizeof(per_sm_cache) / sizeof(int)) per_sm_cache[idx] = per_sm;
    }
    int64_t g = (n + 4 * kBulkRows - 1) / (4 * kBulkRows);
    const int64_t cap = (int64_t)per_sm * t->num_sms;
    return (int)(g < cap ? g : cap);
}

template <int V, int KV>
struct GetRun {
    static cudaError_t run(mlkv_table* t, const int64_t* keys, int64_t n, float* out,
                           cudaStream_t st, CallCounters* cur, CallCounters* nxt) {
        const uint32_t rowbytes = (uint32_t)t->geom.d * 4;
        if (MLKV_GET_BULK && V == 4 && rowbytes <= kBulkRowBytes && (uint64_t)n < kBulkMaxBatch) {
            const size_t smem = (size_t)4 * kBulkRows * rowbytes + 4 * 32 * 4;
            if (t->cfg.insert_on_miss)
                MLKV_LAUNCH(t, MLKV_K_GET_GATHER, k_get_bulk<true>, bulk_grid<true>(t, smem, n), kBulkThreads, smem,
                            st, index_args(t), row_args(t), keys, (uint32_t)n, out, t->s.miss_pos, t->s.miss_slot,
                            cur, nxt, Memo{t->s.memo_key, t->s.memo_row});
            else
                MLKV_LAUNCH(t, MLKV_K_GET_GATHER, k_get_bulk<false>, bulk_grid<false>(t, smem, n), kBulkThreads,
                            smem, st, index_args(t), row_args(t), keys, (uint32_t)n, out, t->s.miss_pos,
                            t->s.miss_slot, cur, nxt, Memo{t->s.memo_key, t->s.memo_row});
            return cudaGetLastError();
        }
        const unsigned grid = grid_for(n, 256);  // 8 warps x 32 lookups per block
        if (t->cfg.insert_on_miss)
            MLKV_LAUNCH(t, MLKV_K_GET_GATHER, (k_get<V, KV, true>), grid, 256, 0, st, index_args(t),
                        row_args(t), keys, (uint32_t)n, out, t->s.miss_pos, t->s.miss_slot, cur, nxt,
                        Memo{t->s.memo_key, t->s.memo_row});
        else
            MLKV_LAUNCH(t, MLKV_K_GET_GATHER, (k_get<V, KV, false>), grid, 256, 0, st, index_args(t),
                        row_args(t), keys, (uint32_t)n, out, t->s.miss_pos, t->s.miss_slot, cur, nxt,
                        Memo{t->s.memo_key, t->s.memo_row});
        return cudaGetLastError();
    }
};

template <int V, int KV>
struct MissRun {
    static cudaError_t run(mlkv_table* t, const int64_t* keys, int64_t n, MissMode mode, float* out,
                           cudaStream_t st, CallCounters* cur, bool release, const FirstCounts* fc) {
        const float span = t->cfg.init_hi - t->cfg.init_lo;
        RowArgs init_ra = row_args(t);  // new rows live in the host tier when tiered
        if (t->tiered) init_ra.slots = t->tier.host_dev;
        MLKV_LAUNCH(t, 0, (k_miss<V, KV>), t->num_sms, kMissThreads, 0, st, index_args(t), init_ra, keys,
                    (uint32_t)n, t->s.miss_pos, t->s.miss_slot, t->s.first_flag, t->s.rank, t->s.tile_sums,
                    mode == MissMode::Get ? nullptr : t->s.row_of_pos, mode == MissMode::Get ? out : nullptr, cur,
                    t->dstate, (unsigned long long)t->cfg.capacity, mode == MissMode::Put ? 0 : 1,
                    (unsigned long long)t->cfg.seed, t->cfg.init_lo, span, t->cfg.state_init,
                    take_injected_wait() ? 1u : 0u, release ? 1 : 0, fc ? *fc : FirstCounts{});
        return cudaGetLastError();
    }
};

template <int V, int KV>
struct PutRun {
    static cudaError_t run(mlkv_table* t, const float* vals, const float* state, int64_t n, cudaStream_t st) {
        MLKV_LAUNCH(t, 0, k_put_mark, grid_for(n, 256), 256, 0, st, t->index, t->s.row_of_pos,
                    t->s.slot_of_pos, (uint32_t)n);
        const unsigned g = capped_grid(t, n * (int64_t)t->geom.G, 256, 8);
        MLKV_LAUNCH(t, MLKV_K_PUT_SCATTER, (k_put_scatter<V, KV>), g, 256, 0, st, t->index, row_args(t),
                    t->s.row_of_pos, t->s.slot_of_pos, vals, state, (uint32_t)n);
        return cudaGetLastError();
    }
};

// The key of every row below n_rows, at its row: a checkpoint's keys in row
// order (rows are dense, handed out in first-occurrence order).
__global__ void __launch_bounds__(256) k_dump_keys(const Slot* __restrict__ index, unsigned long long nslots,
                                                   int64_t* __restrict__ out, uint32_t n_rows) {
    pdl_enter();
    for (unsigned long long s = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x; s < nslots;
         s += (unsigned long long)gridDim.x * blockDim.x) {
        const unsigned long long key = index[s].key;
        const uint32_t row = index[s].row;
        if (key != EMPTY_KEY && row < n_rows) out[row] = (int64_t)key;
    }
}

template <int V, int KV>
struct ExportRun {
    static cudaError_t run(mlkv_table* t, const int64_t* keys, int64_t n, float* rows, float* state,
                           cudaStream_t st, CallCounters* nxt) {
        ExportTier et{nullptr, nullptr, nullptr};
        if (t->tiered) et = ExportTier{t->tier.row_loc, t->tier.cache, t->tier.host_dev};
        MLKV_LAUNCH(t, 0, (k_export<V, KV>), grid_for(n, 256), 256, 0, st, index_args(t),
                    row_args(t), keys, (uint32_t)n, rows, state, nxt, et);
        return cudaGetLastError();
    }
};

}  // namespace

cudaError_t launch_probe(mlkv_table* t, const int64_t* keys, int64_t n, bool insert, MemoUse memo,
                         bool want_slot, bool report_absent, cudaStream_t st, CallCounters* cur,
                         CallCounters* nxt, uint32_t* rows_out, const FirstCounts* fc) {
    uint32_t* slot_of_pos = want_slot ? t->s.slot_of_pos : nullptr;
    uint32_t* rows = rows_out ? rows_out : t->s.row_of_pos;
    if (want_slot && memo == MemoUse::Read) memo = MemoUse::None;  // the memo holds no slots
    const Memo m{t->s.memo_key, t->s.memo_row};
    const int ra = report_absent ? 1 : 0;
    if (fc) {  // one block per sort tile, counting the first pass
        const unsigned g = grid_for(n, 1 << fc->tile_shift);
        if (fc->tile_shift == 12) {
            if (insert)
                MLKV_LAUNCH(t, MLKV_K_PROBE, (k_probe<true, 1024>), g, 1024, 0, st, index_args(t), keys,
                            (uint32_t)n, rows, slot_of_pos, t->s.miss_pos, t->s.miss_slot, cur, nxt, 0, m,
                            (int)memo, *fc);
            else
                MLKV_LAUNCH(t, MLKV_K_PROBE, (k_probe<false, 1024>), g, 1024, 0, st, index_args(t), keys,
                            (uint32_t)n, rows, slot_of_pos, t->s.miss_pos, t->s.miss_slot, cur, nxt, ra, m,
                            (int)memo, *fc);
        } else {  // the small tiles: kSortTileSmall / kProbeKeys threads
            constexpr int CT = kSortTileSmall / kProbeKeys;
            if (insert)
                MLKV_LAUNCH(t, MLKV_K_PROBE, (k_probe<true, CT>), g, CT, 0, st, index_args(t), keys,
                            (uint32_t)n, rows, slot_of_pos, t->s.miss_pos, t->s.miss_slot, cur, nxt, 0, m,
                            (int)memo, *fc);
            else
                MLKV_LAUNCH(t, MLKV_K_PROBE, (k_probe<false, CT>), g, CT, 0, st, index_args(t), keys,
                            (uint32_t)n, rows, slot_of_pos, t->s.miss_pos, t->s.miss_slot, cur, nxt, ra, m,
                            (int)memo, *fc);
        }
        return cudaGetLastError();
    }
    const FirstCounts none{};
    const unsigned g = grid_for(n, 256 * kProbeKeys);
    if (insert)
        MLKV_LAUNCH(t, MLKV_K_PROBE, (k_probe<true, 0>), g, 256, 0, st, index_args(t), keys,
                    (uint32_t)n, rows, slot_of_pos, t->s.miss_pos, t->s.miss_slot, cur, nxt, 0, m, (int)memo, none);
    else
        MLKV_LAUNCH(t, MLKV_K_PROBE, (k_probe<false, 0>), g, 256, 0, st, index_args(t), keys,
                    (uint32_t)n, rows, slot_of_pos, t->s.miss_pos, t->s.miss_slot, cur, nxt, ra, m, (int)memo, none);
    return cudaGetLastError();
}

cudaError_t launch_get(mlkv_table* t, const int64_t* keys, int64_t n, float* out, cudaStream_t st,
                       CallCounters* cur, CallCounters* nxt) {
    return dispatch_row<GetRun>(t->geom, t, keys, n, out, st, cur, nxt);
}

cudaError_t launch_resolve_misses(mlkv_table* t, const int64_t* keys, int64_t n, MissMode mode,
                                  float* out, cudaStream_t st, CallCounters* cur, bool release,
                                  const FirstCounts* fc) {
    return dispatch_row<MissRun>(t->geom, t, keys, n, mode, out, st, cur, release, fc);
}

cudaError_t launch_put_scatter(mlkv_table* t, const float* vals, const float* state, int64_t n, cudaStream_t st) {
    return dispatch_row<PutRun>(t->geom, t, vals, state, n, st);
}

// Slots of keys that never got a row (an insert cut short by a device error)
// go back to idle, so that a later call inserts them afresh.
__global__ void __launch_bounds__(256) k_reset_pending(Slot* __restrict__ index, unsigned long long nslots) {
    for (unsigned long long s = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x; s < nslots;
         s += (unsigned long long)gridDim.x * blockDim.x)
        if (index[s].key != EMPTY_KEY && index[s].row == ROW_PENDING) index[s].aux = AUX_IDLE;
}

cudaError_t launch_reset_pending(mlkv_table* t, cudaStream_t st) {
    k_reset_pending<<<(unsigned)t->num_sms * 8, 256, 0, st>>>(t->index, t->index_mask + 1);
    return cudaGetLastError();
}

cudaError_t launch_dump_keys(mlkv_table* t, int64_t* out, int64_t n_rows, cudaStream_t st) {
    const unsigned long long nslots = t->index_mask + 1;
    MLKV_LAUNCH(t, 0, k_dump_keys, (unsigned)t->num_sms * 8, 256, 0, st, t->index, nslots, out, (uint32_t)n_rows);
    return cudaGetLastError();
}

cudaError_t launch_find(mlkv_table* t, const int64_t* keys, int64_t n, int64_t* rows,
                        cudaStream_t st, CallCounters* nxt) {
    MLKV_LAUNCH(t, 0, k_find, grid_for(n, 256), 256, 0, st, index_args(t), keys, (uint32_t)n, rows, nxt);
    return cudaGetLastError();
}

cudaError_t launch_export(mlkv_table* t, const int64_t* keys, int64_t n, float* rows, float* state,
                          cudaStream_t st, CallCounters* nxt) {
    return dispatch_row<ExportRun>(t->geom, t, keys, n, rows, state, st, nxt);
}

}  // namespace mlkv
