// Dedup of a gradient batch: a stable LSD radix sort of (row id, position)
// pairs, then the segment starts of the sorted row ids.
//
// The sort key is the 32-bit row id, not the 64-bit key: rows are dense in
// [0, capacity), so 3 passes of 9 bits cover 10^8 rows (against 5+ passes for
// 40-bit keys), and the sorted order visits rows in memory order.  An absent
// lookup is given the all-ones digit pattern and sorts last.
//
// The sort follows the single-pass ("Onesweep") scheme of Adinets & Merrill
// (2022): one kernel reads the keys once and counts the digits of every pass;
// then each pass is one kernel in which a block ranks its 4096-element tile
// (stable: warp match over rounds of 32 in order), publishes its per-digit
// count, and finds the count of all earlier tiles by looking back over their
// published values (decoupled look-back).  Tiles are taken in launch order
// from an atomic ticket, so every tile looked at is held by a running block;
// each poll loop is bounded and reports MLKV_ERR_TIMEOUT if it runs out.
#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

constexpr int kThreads = 256;
constexpr int kItems = 16;
constexpr int kTile = kThreads * kItems;  // 4096
constexpr int kWarps = kThreads / 32;

__device__ __forceinline__ int spad(int i) { return i + (i >> 5); }

// Exclusive scan of one value per thread over a 256-thread block.
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t& total) {
    __shared__ uint32_t warp_sums[kWarps];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[w] = x;
    __syncthreads();
    if (w == 0) {
        uint32_t s = lane < kWarps ? warp_sums[lane] : 0u;
#pragma unroll
        for (int o = 1; o < kWarps; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        if (lane < kWarps) warp_sums[lane] = s;
    }
    __syncthreads();
    const uint32_t wprefix = w ? warp_sums[w - 1] : 0u;
    total = warp_sums[kWarps - 1];
    __syncthreads();
    return wprefix + x - v;
}

// Sum of tile_sums[0..b) by the whole block.
__device__ __forceinline__ uint32_t tiles_before(const uint32_t* __restrict__ tile_sums, uint32_t b) {
    uint32_t s = 0;
    for (uint32_t i = threadIdx.x; i < b; i += kThreads) s += tile_sums[i];
    uint32_t total;
    block_exclusive_scan(s, total);
    return total;
}

// --- generic exclusive scan -------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_scan_reduce(const uint32_t* __restrict__ in, uint32_t n,
                                                          uint32_t* __restrict__ tile_sums,
                                                          const uint32_t* enable) {
    if (enable && *enable == 0u) return;
    const uint32_t base = blockIdx.x * kTile;
    uint32_t s = 0;
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
        const uint32_t i = base + k * kThreads + threadIdx.x;
        if (i < n) s += in[i];
    }
    uint32_t total;
    block_exclusive_scan(s, total);
    if (threadIdx.x == 0) tile_sums[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kThreads) k_scan_down(const uint32_t* in, uint32_t* out, uint32_t n,
                                                        const uint32_t* __restrict__ tile_sums,
                                                        uint32_t* total_out, const uint32_t* enable) {
    if (enable && *enable == 0u) return;
    __shared__ uint32_t tile[kTile + kTile / 32];
    const uint32_t base = blockIdx.x * kTile;
    const uint32_t prefix = tiles_before(tile_sums, blockIdx.x);
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
        const int i = k * kThreads + threadIdx.x;
        tile[spad(i)] = (base + i < n) ? in[base + i] : 0u;
    }
    __syncthreads();
    uint32_t local = 0;
#pragma unroll
    for (int k = 0; k < kItems; ++k) local += tile[spad(threadIdx.x * kItems + k)];
    uint32_t block_total;
    uint32_t run = block_exclusive_scan(local, block_total) + prefix;
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
        const int i = spad(threadIdx.x * kItems + k);
        const uint32_t v = tile[i];
        tile[i] = run;
        run += v;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
        const int i = k * kThreads + threadIdx.x;
        if (base + i < n) out[base + i] = tile[spad(i)];
    }
    if (total_out && blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) *total_out = prefix + block_total;
}

// --- radix sort ---------------------------------------------------------------
// Pass 0 reads the probe's row ids (sentinels mapped to `sent`) and uses the
// lookup position as the value.
__device__ __forceinline__ uint32_t sort_key(uint32_t r, uint32_t sent, bool first) {
    return first ? (r >= ROW_ABSENT ? sent : r) : r;
}

constexpr int kMaxRadix = 1 << kSortMaxDigitBits;
constexpr uint32_t kFlagAgg = 1u << 30, kFlagIncl = 2u << 30, kValMask = (1u << 30) - 1;
constexpr int kPollIters = 1 << 22;

// Look-back words are read and published with device-scope relaxed accesses
// (value and flag share one 32-bit word, so no further ordering is needed).
__device__ __forceinline__ uint32_t ld_word(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_word(uint32_t* p, uint32_t v) {
    asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}

// Digit counts of every pass in one read; the last block to finish turns
// them into exclusive prefix sums (per pass) and clears the look-back words.
__global__ void __launch_bounds__(kThreads) k_sort_count(const uint32_t* __restrict__ keys, uint32_t n,
                                                         uint32_t sent, int passes, int D, uint32_t* ghist,
                                                         uint32_t* status, uint32_t status_len,
                                                         uint32_t* done_ctr) {
    __shared__ uint32_t cnt[kSortMaxPasses][kMaxRadix];
    __shared__ bool last;
    const int radix = 1 << D;
    for (int i = threadIdx.x; i < kSortMaxPasses * kMaxRadix; i += kThreads) (&cnt[0][0])[i] = 0;
    for (uint32_t i = blockIdx.x * kThreads + threadIdx.x; i < status_len; i += gridDim.x * kThreads) status[i] = 0;
    __syncthreads();
    for (uint32_t i = blockIdx.x * kThreads + threadIdx.x; i < n; i += gridDim.x * kThreads) {
        const uint32_t k = sort_key(keys[i], sent, true);
        for (int p = 0; p < passes; ++p) atomicAdd(&cnt[p][(k >> (p * D)) & (radix - 1)], 1u);
    }
    __syncthreads();
    for (int p = 0; p < passes; ++p)
        for (int d = threadIdx.x; d < radix; d += kThreads)
            if (cnt[p][d]) atomicAdd(&ghist[p * kMaxRadix + d], cnt[p][d]);
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last = atomicAdd(done_ctr, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int p = 0; p < passes; ++p) {
        // radix <= 512: two counts per thread, block scan of the pair sums
        const int d0 = threadIdx.x * 2;
        const uint32_t a = d0 < radix ? __ldcg(&ghist[p * kMaxRadix + d0]) : 0u;
        const uint32_t b = d0 + 1 < radix ? __ldcg(&ghist[p * kMaxRadix + d0 + 1]) : 0u;
        uint32_t total;
        const uint32_t excl = block_exclusive_scan(a + b, total);
        if (d0 < radix) ghist[p * kMaxRadix + d0] = excl;
        if (d0 + 1 < radix) ghist[p * kMaxRadix + d0 + 1] = excl + a;
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kThreads) k_sort_scatter(const uint32_t* __restrict__ kin,
                                                           const uint32_t* __restrict__ vin,
                                                           uint32_t* __restrict__ kout,
                                                           uint32_t* __restrict__ vout, uint32_t n,
                                                           const uint32_t* __restrict__ gstart,
                                                           uint32_t* status, uint32_t* tile_ctr, int shift,
                                                           int radix, uint32_t sent, int first, ErrSink err) {
    __shared__ uint32_t wcnt[kWarps][kMaxRadix];
    __shared__ uint32_t gbase[kMaxRadix];
    __shared__ uint32_t tile_s;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    if (threadIdx.x == 0) tile_s = atomicAdd(tile_ctr, 1u);
    for (int i = threadIdx.x; i < kWarps * kMaxRadix; i += kThreads) (&wcnt[0][0])[i] = 0;
    __syncthreads();
    const uint32_t tile = tile_s;
    const uint32_t base = tile * kTile + w * (kItems * 32);
    const uint32_t lt = lanemask_lt();
    uint32_t key[kItems], val[kItems], rnk[kItems];
#pragma unroll
    for (int r = 0; r < kItems; ++r) {
        const uint32_t i = base + r * 32 + lane;
        const bool valid = i < n;
        const uint32_t k = valid ? sort_key(kin[i], sent, first) : 0u;
        const uint32_t v = valid ? (first ? i : vin[i]) : 0u;
        const uint32_t dig = (k >> shift) & (radix - 1);
        const uint32_t peers = __match_any_sync(0xffffffffu, valid ? dig : 0xFFFFFFFFu);
        uint32_t before = 0;
        if (valid) before = wcnt[w][dig];
        __syncwarp();
        if (valid && lane == __ffs(peers) - 1) wcnt[w][dig] = before + __popc(peers);
        __syncwarp();
        key[r] = k;
        val[r] = v;
        rnk[r] = valid ? before + __popc(peers & lt) : 0xFFFFFFFFu;
    }
    __syncthreads();
    // per digit: exclusive prefix over the warps, the tile's count, then the
    // look-back for the count of all earlier tiles
    for (int d = threadIdx.x; d < radix; d += kThreads) {
        uint32_t run = 0;
#pragma unroll
        for (int ww = 0; ww < kWarps; ++ww) {
            const uint32_t c = wcnt[ww][d];
            wcnt[ww][d] = run;
            run += c;
        }
        uint32_t* my = status + (size_t)tile * radix + d;
        if (tile == 0) {
            st_word(my, kFlagIncl | run);
            gbase[d] = gstart[d];
            continue;
        }
        st_word(my, kFlagAgg | run);
        uint32_t excl = 0;
        for (int t = (int)tile - 1; t >= 0; --t) {
            const uint32_t* q = status + (size_t)t * radix + d;
            uint32_t v = ld_word(q);
            for (int it = 0; it < kPollIters && (v & ~kValMask) == 0; ++it) v = ld_word(q);
            if ((v & ~kValMask) == 0) {
                record_error(err, MLKV_ERR_TIMEOUT);
                break;
            }
            excl += v & kValMask;
            if (v & kFlagIncl) break;
        }
        st_word(my, kFlagIncl | (excl + run));
        gbase[d] = gstart[d] + excl;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kItems; ++r) {
        if (rnk[r] == 0xFFFFFFFFu) continue;
        const uint32_t dig = (key[r] >> shift) & (radix - 1);
        const uint32_t dst = gbase[dig] + wcnt[w][dig] + rnk[r];
        kout[dst] = key[r];
        vout[dst] = val[r];
    }
}

// --- segments -------------------------------------------------------------------
__device__ __forceinline__ bool is_head(const uint32_t* srow, uint32_t p, uint32_t n, uint32_t sent) {
    if (p >= n) return false;
    const uint32_t r = srow[p];
    return r != sent && (p == 0 || srow[p - 1] != r);
}

__global__ void __launch_bounds__(kThreads) k_seg_reduce(const uint32_t* __restrict__ srow, uint32_t n,
                                                         uint32_t sent, uint32_t* __restrict__ tile_sums) {
    const uint32_t base = blockIdx.x * kTile;
    uint32_t s = 0;
#pragma unroll 4
    for (int k = 0; k < kItems; ++k) s += is_head(srow, base + k * kThreads + threadIdx.x, n, sent);
    uint32_t total;
    block_exclusive_scan(s, total);
    if (threadIdx.x == 0) tile_sums[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kThreads) k_seg_down(const uint32_t* __restrict__ srow,
                                                       const uint32_t* __restrict__ spos, uint32_t n,
                                                       uint32_t sent, const uint32_t* __restrict__ tile_sums,
                                                       uint32_t* __restrict__ seg_start,
                                                       uint32_t* __restrict__ run_row,
                                                       uint32_t* __restrict__ run_p0, CallCounters* cur,
                                                       DevState* ds) {
    const uint32_t base = blockIdx.x * kTile;
    const uint32_t prefix = tiles_before(tile_sums, blockIdx.x);
    // thread t owns items base + t*16 .. +15 (consecutive, for an in-order compaction)
    const uint32_t first = base + threadIdx.x * kItems;
    uint32_t flags = 0, cnt = 0;
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
        const uint32_t p = first + k;
        if (is_head(srow, p, n, sent)) {
            flags |= 1u << k;
            ++cnt;
        }
        if (p < n && srow[p] != sent && (p + 1 == n || srow[p + 1] == sent)) cur->n_valid = p + 1;
    }
    uint32_t block_total;
    uint32_t run = block_exclusive_scan(cnt, block_total) + prefix;
#pragma unroll
    for (int k = 0; k < kItems; ++k)
        if (flags & (1u << k)) {
            const uint32_t p = first + k;
            seg_start[run] = p;
            run_row[run] = srow[p];
            run_p0[run] = spos[p];
            ++run;
        }
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) {
        cur->n_unique = prefix + block_total;
        ds->last_unique = prefix + block_total;
    }
}

__global__ void k_dedup_out(const int64_t* __restrict__ keys, const uint32_t* __restrict__ spos,
                            const uint32_t* __restrict__ seg_start, const CallCounters* cur,
                            int64_t* __restrict__ uniq, int32_t* __restrict__ counts, int64_t* num) {
    const uint32_t U = cur->n_unique, nv = cur->n_valid;
    if (blockIdx.x == 0 && threadIdx.x == 0) *num = (int64_t)U;
    for (uint32_t u = blockIdx.x * blockDim.x + threadIdx.x; u < U; u += gridDim.x * blockDim.x) {
        const uint32_t s = seg_start[u];
        const uint32_t e = u + 1 < U ? seg_start[u + 1] : nv;
        uniq[u] = keys[spos[s]];
        counts[u] = (int32_t)(e - s);
    }
}

inline unsigned tiles(int64_t n) { return (unsigned)((n + kTile - 1) / kTile); }

}  // namespace

cudaError_t launch_exclusive_scan(mlkv_table* t, const uint32_t* in, uint32_t* out, int64_t n,
                                  uint32_t* total, const uint32_t* enable, cudaStream_t st) {
    const unsigned nt = tiles(n);
    MLKV_LAUNCH(t, 0, k_scan_reduce, nt, kThreads, 0, st, in, (uint32_t)n, t->s.tile_sums, enable);
    MLKV_LAUNCH(t, 0, k_scan_down, nt, kThreads, 0, st, in, out, (uint32_t)n, t->s.tile_sums, total, enable);
    return cudaGetLastError();
}

cudaError_t launch_sort_rows(mlkv_table* t, int64_t n, cudaStream_t st, const uint32_t** srow,
                             const uint32_t** spos) {
    const int bits = t->sort_bits;
    const int passes = (bits + kSortMaxDigitBits - 1) / kSortMaxDigitBits;
    const int D = (bits + passes - 1) / passes;
    const int radix = 1 << D;
    const uint32_t sent = (uint32_t)((1ull << bits) - 1);
    const unsigned nt = tiles(n);
    // digit counts, tile tickets and the completion counter start at zero
    cudaError_t e = cudaMemsetAsync(t->s.sort_ghist, 0, t->s.sort_ghist_bytes, st);
    if (e != cudaSuccess) return e;
    uint32_t* ghist = t->s.sort_ghist;
    uint32_t* tile_ctr = ghist + kSortMaxPasses * kMaxRadix;
    uint32_t* done_ctr = tile_ctr + kSortMaxPasses;
    const uint32_t status_len = (uint32_t)((int64_t)passes * nt * radix);
    int64_t cg = nt;
    if (cg > (int64_t)t->num_sms * 4) cg = (int64_t)t->num_sms * 4;
    MLKV_LAUNCH(t, 0, k_sort_count, (unsigned)cg, kThreads, 0, st, t->s.row_of_pos, (uint32_t)n, sent, passes,
                D, ghist, t->s.sort_status, status_len, done_ctr);
    const ErrSink err{&t->dstate->status, t->status_dev_alias};
    const uint32_t* kin = t->s.row_of_pos;
    const uint32_t* vin = nullptr;
    int out = 0;
    for (int p = 0; p < passes; ++p) {
        MLKV_LAUNCH(t, MLKV_K_SORT_SCATTER, k_sort_scatter, nt, kThreads, 0, st, kin, vin, t->s.sk[out],
                    t->s.sv[out], (uint32_t)n, ghist + p * kMaxRadix,
                    t->s.sort_status + (size_t)p * nt * radix, tile_ctr + p, p * D, radix, sent, p == 0, err);
        kin = t->s.sk[out];
        vin = t->s.sv[out];
        out ^= 1;
    }
    *srow = kin;
    *spos = vin;
    return cudaGetLastError();
}

cudaError_t launch_segments(mlkv_table* t, const uint32_t* srow, const uint32_t* spos, int64_t n,
                            cudaStream_t st, CallCounters* cur) {
    const uint32_t sent = (uint32_t)((1ull << t->sort_bits) - 1);
    const unsigned nt = tiles(n);
    MLKV_LAUNCH(t, MLKV_K_SEGMENTS, k_seg_reduce, nt, kThreads, 0, st, srow, (uint32_t)n, sent, t->s.tile_sums);
    MLKV_LAUNCH(t, MLKV_K_SEGMENTS, k_seg_down, nt, kThreads, 0, st, srow, spos, (uint32_t)n, sent,
                t->s.tile_sums, t->s.seg_start, t->s.run_row, t->s.run_p0, cur, t->dstate);
    return cudaGetLastError();
}

cudaError_t launch_dedup_out(mlkv_table* t, const int64_t* keys, const uint32_t* spos, int64_t n,
                             int64_t* uniq, int32_t* counts, int64_t* num, cudaStream_t st,
                             CallCounters* cur) {
    int64_t g = (n + 255) / 256;
    if (g > (int64_t)t->num_sms * 8) g = (int64_t)t->num_sms * 8;
    if (g < 1) g = 1;
    MLKV_LAUNCH(t, 0, k_dedup_out, (unsigned)g, 256, 0, st, keys, spos, t->s.seg_start, cur, uniq, counts, num);
    return cudaGetLastError();
}

}  // namespace mlkv
