// Segmented gradient reduction fused with the sparse Adagrad read-modify-write.
//
// After the sort, the lookups of one row form a run (segment) of consecutive
// sorted positions, in occurrence order (the sort is stable).  For every run
// the sum g of its gradient rows is formed and one Adagrad step is applied to
// the row and its state, each read once and written once:
//     G += g*g ;  w -= lr * g / (sqrt(G) + eps)          (element-wise)
// This is the per-key Rmw of MLKV Section 3.2 step 8, with the gradient of the
// embedding map E (Section 2.1) summed over the key's lookups.
//
//  k_heads        a warp per window of 32 sorted positions finds the runs
//                 that start there (a row id unlike its left neighbour) and
//                 their lengths; runs of one lookup, of 2 .. kSmallRun lookups
//                 (with their positions) and the other runs of <=
//                 MLKV_SEQ_SEGMENT_MAX lookups go to three lists (one atomic
//                 per block and list; any order: every run is summed on its
//                 own), longer ones are measured (a warp-wide search for their
//                 end) and listed for k_long_*.
//  k_single       one lane group per run of one lookup: row, state and the
//                 gradient row loaded together, then the Adagrad step.
//  k_small        one lane group per run of 2 .. kSmallRun lookups, whose
//                 positions k_heads wrote into the run's record: row, state and
//                 every gradient row in one round trip, the occurrence-order
//                 sum, then the Adagrad step.
//  k_short        one lane group per run of kSmallRun + 1 ..
//                 MLKV_SEQ_SEGMENT_MAX lookups: the row, the state, the first
//                 gradient row and the run's other positions are loaded
//                 together, the rest summed in occurrence order, then the
//                 Adagrad step.
//  k_long_sum     one lane group per chunk of 64 lookups (16 in calls of
//                 fewer than 2^19 lookups) of a long run
//                 (Zipf-hot keys reach 10^4-10^5 lookups): the chunk's sum,
//                 compensated, to scratch as a (sum, compensation) pair.
//  k_long_combine per long run: the chunk pairs added in a fixed order with
//                 compensation (split over a whole block's lane groups for the
//                 runs of many chunks, one lane group for the others), the sum
//                 rounded once, and the row updated.
// Long runs are summed with compensation because the Adagrad step is
// ill-conditioned where a summed gradient element lands near eps (with zero
// state, u = lr * g / (|g| + eps) changes fast in g there): a plain fp32 sum
// of 10^2-10^4 terms can then move the update by more than 1e-5, while the
// compensated sum stays within about one rounding of the exact sum.
// Each is tuned for requests in flight (resident warps against rows in flight
// per warp): the access pattern is random 512-byte rows, which HBM serves near
// its copy bandwidth only with many requests in flight.  Results do not depend
// on scheduling.
#include <algorithm>

#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

// Long runs are summed in chunks: of kChunkLarge lookups in calls of at least
// MLKV_SMALL_BATCH lookups, of kChunkSmall in smaller ones (few long runs:
// more chunks to sum in parallel).  Set at build time.
#ifndef MLKV_SMALL_BATCH
#define MLKV_SMALL_BATCH (1u << 19)
#endif
#ifndef MLKV_CHUNK_SMALL
#define MLKV_CHUNK_SMALL 16
#endif
constexpr uint32_t kChunkLarge = 64, kChunkSmall = MLKV_CHUNK_SMALL, kSmallBatch = MLKV_SMALL_BATCH;
// Long runs of more than `big` chunk sums (the hottest rows) are combined by a
// whole block of k_long_combine (MLKV_COMBINE_THREADS); the rest by one lane
// group each.
// In calls of at least kSmallBatch lookups, big = kBigRunLarge (many long
// runs: lane groups keep the SMs busy); below, kBigRunSmall (few long runs:
// blocks sum their chunks in parallel).
constexpr uint32_t kBigRunLarge = 32, kBigRunSmall = 4;

// Tuning (set at build time): gradient rows in flight per lane group, and the
// minimum resident blocks per SM the register allocation must allow.
#ifndef MLKV_REDUCE_ROWS_IN_FLIGHT
#define MLKV_REDUCE_ROWS_IN_FLIGHT 8
#endif
#ifndef MLKV_SHORT_MIN_BLOCKS
#define MLKV_SHORT_MIN_BLOCKS 2
#endif
// k_short: runs a lane group claims at a time.
#ifndef MLKV_SHORT_GRAB
#define MLKV_SHORT_GRAB 4
#endif
// k_single: runs of one lookup in flight per lane group, and blocks per SM.
#ifndef MLKV_SINGLES
#define MLKV_SINGLES 1
#endif
#ifndef MLKV_SINGLE_MIN_BLOCKS
#define MLKV_SINGLE_MIN_BLOCKS 6
#endif
// The apply's reduce kernels on three streams (0: one after the other).
#ifndef MLKV_REDUCE_BRANCHES
#define MLKV_REDUCE_BRANCHES 1
#endif
// Narrow rows (a row on at most 16 lanes: dim <= 64): runs of one lookup two
// at a time per lane group on at most 3 blocks per SM, runs of 5-32 lookups
// with 4 gradient rows in flight at 3 blocks per SM (more warps); 0: the
// wide rows' kernels for every dim.
#ifndef MLKV_NARROW_ROWS
#define MLKV_NARROW_ROWS 1
#endif
// k_single on at most this many blocks per SM (0: as many as fit).
#ifndef MLKV_SINGLE_PER_SM
#define MLKV_SINGLE_PER_SM 0
#endif
// Launch order of the reduce kernels.  MLKV_SHORT_FIRST: the runs of 5-32 launched before those of 2-4 (0: never,
// 1: always, 2: in calls of fewer than kSmallBatch lookups).
#ifndef MLKV_SHORT_FIRST
#define MLKV_SHORT_FIRST 2
#endif
// k_long_combine's block (a big run's chunks are split over its lane groups):
// 256 threads fit the slots that retiring blocks of the other reduce kernels
// free, where a 1024-thread block waited for a whole SM to drain (DLRM: the
// combine started 70 us after its chunk sums were done).
#ifndef MLKV_COMBINE_THREADS
#define MLKV_COMBINE_THREADS 256
#endif
// k_small: blocks per SM the register allocation must allow.
#ifndef MLKV_SMALL_MIN_BLOCKS
#define MLKV_SMALL_MIN_BLOCKS 4
#endif
constexpr uint32_t NONE = 0xFFFFFFFFu;  // no position (a small run's record past its end)
#ifndef MLKV_LONG_ROWS_IN_FLIGHT
#define MLKV_LONG_ROWS_IN_FLIGHT 8
#endif
#ifndef MLKV_LONG_MIN_BLOCKS
#define MLKV_LONG_MIN_BLOCKS 2
#endif

struct RowArgs {
    float* slots;
    int stride;
    int dpad;
    int NV;
    int G;
    int d;
    uint32_t nrows;  // rows of the slot array (bounds-checked build)
};

// Sites of the bounds-checked build (in_bounds).
enum CheckSite : uint32_t {
    kChkSingleRow = 1, kChkSinglePos, kChkSmallRow, kChkSmallPos, kChkShortRun, kChkShortRow, kChkShortPos,
    kChkLongItem, kChkLongPos, kChkCombineRun, kChkCombineRow, kChkHeadsPos, kChkListEntry
};

struct RunArgs {
    const float* grads;
    const uint32_t* srow;  // sorted row ids; lookups without a row hold `sent` and come last
    const uint32_t* spos;  // their lookup positions
    uint32_t n;
    uint32_t sent;
    CallCounters* cur;
    uint4* runs;           // [max_batch] short runs of 2 or more lookups: (first sorted position, one
                           //   past the last, row, first lookup position)
    uint2* singles;        // [max_batch] runs of one lookup: (row, lookup position)
    uint4* smalls;         // [max_batch] runs of 2 .. kSmallRun lookups: (row, p0, p1, p2), positions in
                           //   occurrence order, NONE past the run's end
    uint32_t* small_p3;    // [max_batch] their fourth position (or NONE)
    uint32_t* long_s;      // [max_long] first sorted position
    uint32_t* long_e;      // [max_long] one past the last
    uint32_t* long_row;    // [max_long]
    uint32_t* long_base;   // [max_long] first chunk item
    uint32_t* item_s;      // [max_items] first sorted position of each chunk
    uint32_t* item_e;      // [max_items] one past its last
    uint32_t* big_runs;    // [max_long] long runs of more than `big` chunks
    float* partial;        // [max_items][dpad]
    uint32_t max_long;
    uint32_t max_items;
    uint32_t chunk;        // lookups per chunk of a long run (kChunkLarge or kChunkSmall)
    uint32_t big;          // long runs of more chunks than this are combined by a whole block
    ErrSink err;
    float lr, eps;
    uint32_t release;      // non-zero in the apply's last kernels: the blocks of all of them (release_counters)
};

__device__ __forceinline__ unsigned group_mask(int G, int gid) {
    return G == 32 ? 0xffffffffu : (((1u << G) - 1u) << (gid * G));
}

// acc += the gradient rows of sorted positions s .. s+len-1, in that order.
// The group loads up to G positions at a time (one per lane) and hands them
// round with group shuffles.  With PRE the first G positions were loaded by
// the caller (pl_first, one per lane).  With COMP every addition is
// compensated (comp_add): acc + cmp is then the sum to about twice fp32's
// precision; without it cmp is not touched.
template <int V, int KV, int ROWS = MLKV_REDUCE_ROWS_IN_FLIGHT, bool PRE = false, bool COMP = false>
__device__ __forceinline__ void sum_rows(typename Vec<V>::T (&acc)[KV], typename Vec<V>::T (&cmp)[KV],
                                         const float* __restrict__ grads,
                                         const uint32_t* __restrict__ spos, uint32_t s, uint32_t len, int d,
                                         int NV, int G, int glane, unsigned gmask, const ErrSink& err,
                                         uint32_t site, uint32_t n, uint32_t pl_first = 0u) {
    using VT = typename Vec<V>::T;
    constexpr int UNR = KV >= ROWS ? 1 : ROWS / KV;
    for (uint32_t base = 0; base < len; base += G) {
        const uint32_t cnt = min((uint32_t)G, len - base);
        if (MLKV_CHECK && !in_bounds(err, site, s + base + cnt - 1, n)) return;
        const uint32_t pl = (PRE && base == 0) ? pl_first
                            : (uint32_t)glane < cnt ? __ldg(spos + s + base + glane) : 0u;
        for (uint32_t x = 0; x < cnt; x += UNR) {
            VT g[UNR][KV];
#pragma unroll
            for (int u = 0; u < UNR; ++u) {
                uint32_t p = __shfl_sync(gmask, pl, (int)(x + u) & (G - 1), G);
                if (MLKV_CHECK && x + u < cnt && !in_bounds(err, site, p, n)) p = 0;
                const VT* src = reinterpret_cast<const VT*>(grads + (size_t)p * d);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (x + u < cnt && j < NV) g[u][k] = __ldcs(src + j);
                }
            }
#pragma unroll
            for (int u = 0; u < UNR; ++u)
#pragma unroll
                for (int k = 0; k < KV; ++k)
                    if (x + u < cnt && glane + G * k < NV) {
                        if (COMP) Vec<V>::cadd(acc[k], cmp[k], g[u][k]);
                        else Vec<V>::add(acc[k], g[u][k]);
                    }
        }
    }
}

template <int V, int KV>
__device__ __forceinline__ void load_row_state(const RowArgs& ra, uint32_t row, typename Vec<V>::T (&w)[KV],
                                               typename Vec<V>::T (&G)[KV], int glane) {
    using VT = typename Vec<V>::T;
    const float* slot = ra.slots + (size_t)row * ra.stride;
    const VT* wv = reinterpret_cast<const VT*>(slot);
    const VT* gv = reinterpret_cast<const VT*>(slot + ra.dpad);
#pragma unroll
    for (int k = 0; k < KV; ++k) {
        const int j = glane + ra.G * k;
        if (j < ra.NV) {
            w[k] = wv[j];
            G[k] = gv[j];
        }
    }
}

template <int V, int KV>
__device__ __forceinline__ void adagrad_store(const RowArgs& ra, uint32_t row, typename Vec<V>::T (&w)[KV],
                                              typename Vec<V>::T (&G)[KV], const typename Vec<V>::T (&g)[KV],
                                              int glane, float lr, float eps) {
    using VT = typename Vec<V>::T;
    float* slot = ra.slots + (size_t)row * ra.stride;
    VT* wv = reinterpret_cast<VT*>(slot);
    VT* gv = reinterpret_cast<VT*>(slot + ra.dpad);
#pragma unroll
    for (int k = 0; k < KV; ++k) {
        const int j = glane + ra.G * k;
        if (j < ra.NV) {
            Vec<V>::adagrad(w[k], G[k], g[k], lr, eps);
            wv[j] = w[k];
            gv[j] = G[k];
        }
    }
}

// Where the run of `row` that starts at sorted position s ends: the first
// later position holding another row, or n.  The whole warp searches: 32
// probes at doubling distances, then rounds of 32 evenly spaced probes, each
// round narrowing [lo, hi) (srow[lo] == row; hi == n or srow[hi] != row) 32-fold.
__device__ __forceinline__ uint32_t run_end(const uint32_t* __restrict__ srow, uint32_t n, uint32_t s,
                                            uint32_t row, int lane) {
    uint32_t lo = s, hi = n;
    {
        const unsigned long long q = (unsigned long long)s + (64ull << lane);
        const bool eq = q < hi && __ldg(srow + q) == row;
        const int k = __popc(__ballot_sync(0xffffffffu, eq));  // the equal probes are the first k lanes
        if (k) lo = (uint32_t)((unsigned long long)s + (64ull << (k - 1)));
        const unsigned long long qh = (unsigned long long)s + (64ull << k);
        if (qh < hi) hi = (uint32_t)qh;
    }
    while (hi - lo > 1) {
        const uint32_t step = (hi - lo + 31) / 32;
        const unsigned long long q = (unsigned long long)lo + (unsigned long long)step * (lane + 1);
        const bool eq = q < hi && __ldg(srow + q) == row;
        const uint32_t c = __popc(__ballot_sync(0xffffffffu, eq));
        const unsigned long long nhi = (unsigned long long)lo + (unsigned long long)step * (c + 1);
        lo += step * c;
        if (nhi < hi) hi = (uint32_t)nhi;
    }
    return hi;
}

// The same, for a run of `row` that covers position q0 - 1 (q0 a multiple of
// 32): first the next 1024 positions in one round (32 consecutive per lane,
// 16-byte loads), which ends most runs; beyond that, run_end.
__device__ __forceinline__ uint32_t scan_end(const uint32_t* __restrict__ srow, uint32_t n, uint32_t q0,
                                             uint32_t row, int lane) {
    if (q0 >= n) return n;
    const uint32_t b = q0 + 32u * lane;
    int first = 32;  // first position of this lane's 32 with another row
    if (b + 32 <= n) {
        const uint4* v = reinterpret_cast<const uint4*>(srow + b);
#pragma unroll
        for (int k = 7; k >= 0; --k) {
            const uint4 x = __ldg(v + k);
            if (x.w != row) first = 4 * k + 3;
            if (x.z != row) first = 4 * k + 2;
            if (x.y != row) first = 4 * k + 1;
            if (x.x != row) first = 4 * k;
        }
    } else {
        for (int k = 31; k >= 0; --k)
            if (b + k >= n || __ldg(srow + b + k) != row) first = k;
    }
    const unsigned m = __ballot_sync(0xffffffffu, first < 32);
    if (m) {
        const int l = __ffs(m) - 1;
        return q0 + 32u * l + (uint32_t)__shfl_sync(0xffffffffu, first, l);
    }
    return run_end(srow, n, q0 + 1023u, row, lane);
}

// Chunks of `chunk` lookups of the long runs qs[k] .. qe[k] (k < nq): this
// lane's run's count, and the exclusive prefix over the lanes (the whole warp).
__device__ __forceinline__ uint32_t long_chunks(const uint32_t* qs, const uint32_t* qe, int nq, int lane,
                                                uint32_t chunk, uint32_t& excl) {
    const uint32_t nit = lane < nq ? (qe[lane] - qs[lane] + chunk - 1) / chunk : 0u;
    uint32_t x = nit;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    excl = x - nit;
    return __shfl_sync(0xffffffffu, x, 31);  // all the runs' chunks
}

// Writes the long runs qs[k], qe[k], qr[k] (k < nq: start, end, row) at list
// entries h0.. and their chunks at items ib0.. for k_long_sum / k_long_combine
// (the whole warp).
__device__ __forceinline__ void write_long_runs(const RunArgs& a, const uint32_t* qs, const uint32_t* qe,
                                                const uint32_t* qr, int nq, uint32_t h0, uint32_t ib0,
                                                int lane) {
    uint32_t excl;
    const uint32_t chunk = a.chunk;
    long_chunks(qs, qe, nq, lane, chunk, excl);
    if (lane < nq) {
        a.long_s[h0 + lane] = qs[lane];
        a.long_e[h0 + lane] = qe[lane];
        a.long_row[h0 + lane] = qr[lane];
        a.long_base[h0 + lane] = ib0 + excl;
        if ((qe[lane] - qs[lane] + chunk - 1) / chunk > a.big) a.big_runs[atomicAdd(&a.cur->n_big, 1u)] = h0 + lane;
    }
    for (int k = 0; k < nq; ++k) {
        const uint32_t s = qs[k], e = qe[k];
        const uint32_t m = (e - s + chunk - 1) / chunk;
        const uint32_t ib = ib0 + __shfl_sync(0xffffffffu, excl, k);
        for (uint32_t c = lane; c < m; c += 32) {
            a.item_s[ib + c] = s + c * chunk;
            a.item_e[ib + c] = min(s + (c + 1) * chunk, e);
        }
    }
}

// One short run [s, s + len) of `row`, first lookup p0, by one lane group: the
// row, the state and the first gradient row are loaded together, the rest of
// the gradient rows are added in occurrence order, then the Adagrad step.
template <int V, int KV, int ROWS = MLKV_REDUCE_ROWS_IN_FLIGHT>
__device__ __forceinline__ void short_run(const RowArgs& ra, const RunArgs& a, uint32_t s, uint32_t len,
                                          uint32_t row, uint32_t p0, int glane, unsigned gmask) {
    using VT = typename Vec<V>::T;
    if (MLKV_CHECK && !(in_bounds(a.err, kChkShortRun, s + len, (unsigned long long)a.n + 1) &&
                        in_bounds(a.err, kChkShortRun, 1, len) && in_bounds(a.err, kChkShortRow, row, ra.nrows) &&
                        in_bounds(a.err, kChkShortPos, p0, a.n)))
        return;
    VT w[KV], Gs[KV], acc[KV];
    // the positions of the run's other lookups load beside its row, state and
    // first gradient row, so a run of a few lookups costs two round trips
    const uint32_t rest = len - 1;
    const uint32_t pl0 = (uint32_t)glane < min(rest, (uint32_t)ra.G) ? __ldg(a.spos + s + 1 + glane) : 0u;
    load_row_state<V, KV>(ra, row, w, Gs, glane);
    const VT* g0 = reinterpret_cast<const VT*>(a.grads + (size_t)p0 * ra.d);
#pragma unroll
    for (int k = 0; k < KV; ++k) {
        acc[k] = Vec<V>::zero();
        const int j = glane + ra.G * k;
        if (j < ra.NV) Vec<V>::add(acc[k], __ldcs(g0 + j));  // 0 + g: first term, in order
    }
    if (len > 1)
        sum_rows<V, KV, ROWS, true>(acc, acc, a.grads, a.spos, s + 1, rest, ra.d, ra.NV,
                                                          ra.G, glane, gmask, a.err, kChkShortPos, a.n, pl0);
    adagrad_store<V, KV>(ra, row, w, Gs, acc, glane, a.lr, a.eps);
}

// A warp per window of 32 sorted positions (windows dealt out grid-stride).
// A run starts where a row id differs from its left neighbour; it ends at the
// next change of value in the window (the next run, or the absent lookups
// that sort last) or, for the window's last run, where the next window's row
// ids first differ (past that, it is long and its end is searched for after
// the windows).  Runs of one lookup and the other runs of <=
// MLKV_SEQ_SEGMENT_MAX lookups are staged in the warp's two shared-memory
// lists, long ones in its queue; at the end the block reserves room in the
// two run lists, the long-run list and the chunk list with one atomic each and
// the warps copy their runs out.  (Counters that every warp bumps queue up at
// the end of the kernel.)
#ifndef MLKV_HEADS_MIN_BLOCKS
#define MLKV_HEADS_MIN_BLOCKS 4
#endif
__global__ void __launch_bounds__(256, MLKV_HEADS_MIN_BLOCKS) k_heads(RunArgs a) {
    pdl_enter();
    constexpr int kList = 128, kListS = 64, kQueue = 16;
    __shared__ uint4 lst[8][kListS];  // (start, end, row, first lookup) of short runs
    __shared__ uint2 sgl[8][kList];   // (row, lookup) of runs of one lookup
    __shared__ uint4 sml[8][kListS];  // (row, p0, p1, p2) of small runs
    __shared__ uint32_t sp3[8][kListS];  // ... and their p3
    __shared__ uint32_t qs[8][kQueue], qr[8][kQueue], qe[8][kQueue];  // long runs: start, row, end (0: unknown)
    __shared__ uint32_t wsh[8], wlg[8], wit[8], ws1[8], ws2[8];  // per warp: short runs, long runs, chunks,
                                                                 // runs of one lookup, small runs; then
                                                                 // their bases
    const uint32_t n = a.n, sent = a.sent;
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const uint32_t lt = lanemask_lt();
    const uint32_t warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
    const uint32_t nwin = (n + 31) >> 5;
    int cnt = 0, cnt1 = 0, cnt2 = 0, nq = 0;  // warp-uniform
    // full lists or a full queue go out at once (only batches far above a few
    // runs per window and warp get here)
    auto flush = [&]() {
        __syncwarp();
        uint32_t base = 0, base1 = 0, base2 = 0;
        if (lane == 0 && cnt) base = atomicAdd(&a.cur->n_short, (uint32_t)cnt);
        if (lane == 0 && cnt1) base1 = atomicAdd(&a.cur->n_single, (uint32_t)cnt1);
        if (lane == 0 && cnt2) base2 = atomicAdd(&a.cur->n_small, (uint32_t)cnt2);
        base = __shfl_sync(0xffffffffu, base, 0);
        base1 = __shfl_sync(0xffffffffu, base1, 0);
        base2 = __shfl_sync(0xffffffffu, base2, 0);
        for (int k = lane; k < cnt; k += 32) a.runs[base + k] = lst[wib][k];
        for (int k = lane; k < cnt1; k += 32) a.singles[base1 + k] = sgl[wib][k];
        for (int k = lane; k < cnt2; k += 32) {
            a.smalls[base2 + k] = sml[wib][k];
            a.small_p3[base2 + k] = sp3[wib][k];
        }
        cnt = 0;
        cnt1 = 0;
        cnt2 = 0;
        __syncwarp();
    };
    auto measure = [&]() {  // fills in the unknown ends of the queued long runs
        __syncwarp();
        for (int k = 0; k < nq; ++k) {
            // an unknown end lies past the window after the run's first one
            if (qe[wib][k] == 0u) {
                const uint32_t e = scan_end(a.srow, n, (qs[wib][k] & ~31u) + 64u, qr[wib][k], lane);
                __syncwarp();
                if (lane == 0) qe[wib][k] = e;
                __syncwarp();
            }
        }
    };
    auto emit_long = [&](uint32_t h0, uint32_t ib0) {
        if (nq) write_long_runs(a, qs[wib], qe[wib], qr[wib], nq, h0, ib0, lane);
        nq = 0;
        __syncwarp();
    };
    // a window's row ids, the next window's, the left neighbour and the
    // positions, loaded one window ahead
    auto load = [&](uint32_t w, uint32_t& r, uint32_t& nr, uint32_t& l0, uint32_t& pos) {
        const uint32_t p = (w << 5) + lane;
        r = p < n ? __ldg(a.srow + p) : sent;
        nr = p + 32 < n ? __ldg(a.srow + p + 32) : sent;
        pos = p < n ? __ldg(a.spos + p) : 0u;
        l0 = lane == 0 && p > 0 && p <= n ? __ldg(a.srow + p - 1) : ~r;
    };
    uint32_t xr = sent, xnr = sent, xl0 = 0u, xpos = 0u;
    if (warp < nwin) load(warp, xr, xnr, xl0, xpos);
    for (uint32_t w = warp; w < nwin; w += nwarps) {  // warp-uniform
        const uint32_t p = (w << 5) + lane;
        const uint32_t r = xr, nr = xnr, pos = xpos;
        uint32_t left = __shfl_up_sync(0xffffffffu, r, 1);
        if (lane == 0) left = xl0;
        if (w + nwarps < nwin) load(w + nwarps, xr, xnr, xl0, xpos);
        const unsigned em = __ballot_sync(0xffffffffu, r != left);  // a run, or the absent tail, starts here
        const bool head = r != sent && r != left;
        const unsigned hm = __ballot_sync(0xffffffffu, head);
        if (!hm) continue;
        const uint32_t lrow = __shfl_sync(0xffffffffu, r, 31 - __clz(hm));
        const unsigned diff = __ballot_sync(0xffffffffu, nr != lrow);  // for the window's last run
        const unsigned after = lane == 31 ? 0u : em & (0xFFFFFFFEu << lane);
        uint32_t len = 0;
        bool lng = false;
        if (head) {
            if (after) len = (uint32_t)(__ffs(after) - 1 - lane);
            else if (diff) len = 32 - lane + (__ffs(diff) - 1);
            else lng = true;
            lng = lng || len > MLKV_SEQ_SEGMENT_MAX;
        }
        const bool shrt = head && !lng;  // len >= 1
        const bool smll = shrt && len > 1 && len <= kSmallRun;
        const unsigned sm = __ballot_sync(0xffffffffu, shrt && len > kSmallRun);
        const unsigned s1 = __ballot_sync(0xffffffffu, shrt && len == 1);
        const unsigned s2 = __ballot_sync(0xffffffffu, smll);
        // a small run's other positions: from the lanes after its head, or, where
        // the run goes on into the next window, from the sorted positions
        const uint32_t q1 = __shfl_down_sync(0xffffffffu, pos, 1);
        const uint32_t q2 = __shfl_down_sync(0xffffffffu, pos, 2);
        const uint32_t q3 = __shfl_down_sync(0xffffffffu, pos, 3);
        if (cnt + __popc(sm) > kListS || cnt1 + __popc(s1) > kList || cnt2 + __popc(s2) > kListS) flush();
        if (shrt && len > kSmallRun) lst[wib][cnt + __popc(sm & lt)] = make_uint4(p, p + len, r, pos);
        if (shrt && len == 1) sgl[wib][cnt1 + __popc(s1 & lt)] = make_uint2(r, pos);
        if (smll && MLKV_CHECK && !in_bounds(a.err, kChkHeadsPos, p + len - 1, n)) len = 2;
        if (smll && (!MLKV_CHECK || in_bounds(a.err, kChkHeadsPos, p + len - 1, n))) {
            const uint32_t p1 = lane + 1 < 32 ? q1 : __ldg(a.spos + p + 1);
            const uint32_t p2 = len < 3 ? NONE : lane + 2 < 32 ? q2 : __ldg(a.spos + p + 2);
            const uint32_t p3 = len < 4 ? NONE : lane + 3 < 32 ? q3 : __ldg(a.spos + p + 3);
            const int k = cnt2 + __popc(s2 & lt);
            sml[wib][k] = make_uint4(r, pos, p1, p2);
            sp3[wib][k] = p3;
        }
        cnt += __popc(sm);
        cnt1 += __popc(s1);
        cnt2 += __popc(s2);
        for (unsigned lm = __ballot_sync(0xffffffffu, head && lng); lm; lm &= lm - 1) {
            const int i = __ffs(lm) - 1;
            if (nq == kQueue) {
                measure();
                uint32_t excl, h0 = 0, ib0 = 0;
                const uint32_t items = long_chunks(qs[wib], qe[wib], nq, lane, a.chunk, excl);
                if (lane == 0) {
                    h0 = atomicAdd(&a.cur->n_long, (uint32_t)nq);
                    ib0 = atomicAdd(&a.cur->n_items, items);
                }
                h0 = __shfl_sync(0xffffffffu, h0, 0);
                ib0 = __shfl_sync(0xffffffffu, ib0, 0);
                if (h0 + nq > a.max_long || ib0 + items > a.max_items) {
                    if (lane == 0) record_error(a.err, MLKV_ERR_FULL);
                    nq = 0;
                } else {
                    emit_long(h0, ib0);
                }
            }
            const uint32_t row = __shfl_sync(0xffffffffu, r, i);
            const uint32_t ln = __shfl_sync(0xffffffffu, len, i);  // 0 when the end is past the next window
            if (lane == 0) {
                qs[wib][nq] = (w << 5) + i;
                qr[wib][nq] = row;
                qe[wib][nq] = ln ? (w << 5) + i + ln : 0u;
            }
            ++nq;
        }
    }
    measure();
    uint32_t excl;
    const uint32_t items = long_chunks(qs[wib], qe[wib], nq, lane, a.chunk, excl);
    if (lane == 0) {
        wsh[wib] = (uint32_t)cnt;
        wlg[wib] = (uint32_t)nq;
        wit[wib] = items;
        ws1[wib] = (uint32_t)cnt1;
        ws2[wib] = (uint32_t)cnt2;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t ts = 0, tl = 0, ti = 0, t1 = 0, t2 = 0;
        for (int k = 0; k < 8; ++k) {
            ts += wsh[k];
            tl += wlg[k];
            ti += wit[k];
            t1 += ws1[k];
            t2 += ws2[k];
        }
        uint32_t bs = ts ? atomicAdd(&a.cur->n_short, ts) : 0u;
        uint32_t bl = tl ? atomicAdd(&a.cur->n_long, tl) : 0u;
        uint32_t bi = ti ? atomicAdd(&a.cur->n_items, ti) : 0u;
        uint32_t b1 = t1 ? atomicAdd(&a.cur->n_single, t1) : 0u;
        uint32_t b2 = t2 ? atomicAdd(&a.cur->n_small, t2) : 0u;
        for (int k = 0; k < 8; ++k) {
            const uint32_t c0 = wsh[k], c1 = wlg[k], c2 = wit[k], c3 = ws1[k], c4 = ws2[k];
            wsh[k] = bs;
            wlg[k] = bl;
            wit[k] = bi;
            ws1[k] = b1;
            ws2[k] = b2;
            bs += c0;
            bl += c1;
            bi += c2;
            b1 += c3;
            b2 += c4;
        }
    }
    __syncthreads();
    for (int k = lane; k < cnt; k += 32) a.runs[wsh[wib] + k] = lst[wib][k];
    for (int k = lane; k < cnt1; k += 32) a.singles[ws1[wib] + k] = sgl[wib][k];
    for (int k = lane; k < cnt2; k += 32) {
        a.smalls[ws2[wib] + k] = sml[wib][k];
        a.small_p3[ws2[wib] + k] = sp3[wib][k];
    }
    if (wlg[wib] + nq > a.max_long || wit[wib] + items > a.max_items) {
        if (lane == 0 && nq) record_error(a.err, MLKV_ERR_FULL);
        return;
    }
    emit_long(wlg[wib], wit[wib]);
}

// One lane group per listed run of 2 .. MLKV_SEQ_SEGMENT_MAX lookups.  The
// run's record (bounds, row, first lookup position) is loaded one run ahead;
// its row, state, first gradient row and the positions of its other lookups
// then load together, and the other gradient rows after them.
__device__ __forceinline__ uint4 run_meta(const RunArgs& a, uint32_t u, uint32_t U) {
    return u < U ? __ldg(a.runs + u) : make_uint4(0u, 0u, 0u, 0u);
}

template <int V, int KV, int ROWS = MLKV_REDUCE_ROWS_IN_FLIGHT>
__global__ void __launch_bounds__(256, ROWS >= 8 ? MLKV_SHORT_MIN_BLOCKS : 3) k_short(RowArgs ra, RunArgs a) {
    pdl_enter();
    if (MLKV_CHECK && !in_bounds(a.err, kChkListEntry, a.cur->n_short, (unsigned long long)a.n + 1)) return;
    const uint32_t U = min(a.cur->n_short, a.n);  // a list never holds more runs than lookups
    const int lane = threadIdx.x & 31, G = ra.G, glane = lane & (G - 1), gid = lane / G;
    const unsigned gmask = group_mask(G, gid);
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) / G;
    const uint32_t ngroups = (gridDim.x * blockDim.x) / G;
    // Runs take 5 .. 32 lookups, so fixed shares would leave the kernel to the
    // group with the most lookups: each group claims chunks of `grab` runs, its
    // first chunk by its index, the rest from a counter (one atomic a chunk).
    // With fewer runs than MLKV_SHORT_GRAB per group, one run at a time: every
    // run then starts at once instead of queueing behind others.
    const uint32_t grab = U >= ngroups * (uint32_t)MLKV_SHORT_GRAB ? (uint32_t)MLKV_SHORT_GRAB : 1u;
    uint32_t base = group * grab;
    while (base < U) {  // uniform within the group
        const uint32_t end = min(U, base + grab);
        uint4 next = run_meta(a, base, end);
        for (uint32_t u = base; u < end; ++u) {
            const uint4 m = next;  // (start, end, row, first lookup)
            next = run_meta(a, u + 1, end);
            short_run<V, KV, ROWS>(ra, a, m.x, m.y - m.x, m.z, m.w, glane, gmask);
        }
        uint32_t c = 0;
        if (glane == 0) c = atomicAdd(&a.cur->short_next, grab);
        base = ngroups * grab + __shfl_sync(gmask, c, 0, G);
    }
    if (a.release) release_counters(a.cur, a.release);
}

// One lane group per run of one lookup (most runs of a Zipf batch): its row,
// state and gradient row, SINGLES runs at a time, records loaded one round
// ahead; the sum is the gradient row itself (0 + g), then the Adagrad step.
// With no loop over positions it needs few registers, so more warps (and
// rows) are in flight than in k_short.
template <int V, int KV, int SG = MLKV_SINGLES>
__global__ void __launch_bounds__(256, SG == 1 ? MLKV_SINGLE_MIN_BLOCKS : 4) k_single(RowArgs ra, RunArgs a) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    if (MLKV_CHECK && !in_bounds(a.err, kChkListEntry, a.cur->n_single, (unsigned long long)a.n + 1)) return;
    const uint32_t U = min(a.cur->n_single, a.n);  // a list never holds more runs than lookups
    const int lane = threadIdx.x & 31, G = ra.G, glane = lane & (G - 1);
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) / G;
    const uint32_t ngroups = (gridDim.x * blockDim.x) / G;
    const uint2 none = make_uint2(0xFFFFFFFFu, 0u);
    uint2 next[SG];
#pragma unroll
    for (int j = 0; j < SG; ++j) next[j] = group * SG + j < U ? __ldg(a.singles + group * SG + j) : none;
    for (uint32_t u = group * SG; u < U; u += ngroups * SG) {  // uniform within the group
        uint2 m[SG];
#pragma unroll
        for (int j = 0; j < SG; ++j) {
            m[j] = next[j];
            const uint32_t v = u + ngroups * SG + j;
            next[j] = v < U ? __ldg(a.singles + v) : none;
        }
        VT w[SG][KV], Gs[SG][KV], g[SG][KV];
#pragma unroll
        for (int j = 0; j < SG; ++j) {
            if (m[j].x == 0xFFFFFFFFu) continue;
            if (MLKV_CHECK && !(in_bounds(a.err, kChkSingleRow, m[j].x, ra.nrows) &&
                                in_bounds(a.err, kChkSinglePos, m[j].y, a.n))) {
                m[j].x = 0xFFFFFFFFu;
                continue;
            }
            load_row_state<V, KV>(ra, m[j].x, w[j], Gs[j], glane);
            const VT* src = reinterpret_cast<const VT*>(a.grads + (size_t)m[j].y * ra.d);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int jj = glane + G * k;
                if (jj < ra.NV) g[j][k] = __ldcs(src + jj);
            }
        }
#pragma unroll
        for (int j = 0; j < SG; ++j) {
            if (m[j].x == 0xFFFFFFFFu) continue;
            VT acc[KV];
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                acc[k] = Vec<V>::zero();
                if (glane + G * k < ra.NV) Vec<V>::add(acc[k], g[j][k]);  // 0 + g, as in a longer run
            }
            adagrad_store<V, KV>(ra, m[j].x, w[j], Gs[j], acc, glane, a.lr, a.eps);
        }
    }
    if (a.release) release_counters(a.cur, a.release);
}

// One lane group per run of 2 .. kSmallRun lookups (most runs of more than one
// lookup in a Zipf batch).  k_heads put the run's positions in its record, so
// the row, the state and every gradient row of the run load together, in one
// round trip (records loaded one run ahead); then the sum 0 + g0 + g1 + ... in
// occurrence order and the Adagrad step.  No loop over positions: few
// registers and many warps, as in k_single.
template <int V, int KV>
__global__ void __launch_bounds__(256, KV >= 4 ? 2 : MLKV_SMALL_MIN_BLOCKS) k_small(RowArgs ra, RunArgs a) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    if (MLKV_CHECK && !in_bounds(a.err, kChkListEntry, a.cur->n_small, (unsigned long long)a.n + 1)) return;
    const uint32_t U = min(a.cur->n_small, a.n);  // a list never holds more runs than lookups
    const int lane = threadIdx.x & 31, G = ra.G, glane = lane & (G - 1);
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) / G;
    const uint32_t ngroups = (gridDim.x * blockDim.x) / G;
    uint4 next = group < U ? __ldg(a.smalls + group) : make_uint4(0u, 0u, 0u, 0u);
    uint32_t next3 = group < U ? __ldg(a.small_p3 + group) : NONE;
    for (uint32_t u = group; u < U; u += ngroups) {  // uniform within the group
        const uint4 m = next;  // (row, p0, p1, p2)
        const uint32_t p3 = next3;
        const uint32_t v = u + ngroups;
        next = v < U ? __ldg(a.smalls + v) : make_uint4(0u, 0u, 0u, 0u);
        next3 = v < U ? __ldg(a.small_p3 + v) : NONE;
        VT w[KV], Gs[KV], g[kSmallRun][KV];
        if (MLKV_CHECK && !(in_bounds(a.err, kChkSmallRow, m.x, ra.nrows) && in_bounds(a.err, kChkSmallPos, m.y, a.n) &&
                            in_bounds(a.err, kChkSmallPos, m.z, a.n) &&
                            (m.w == NONE || in_bounds(a.err, kChkSmallPos, m.w, a.n)) &&
                            (p3 == NONE || in_bounds(a.err, kChkSmallPos, p3, a.n))))
            continue;
        load_row_state<V, KV>(ra, m.x, w, Gs, glane);
        const uint32_t ps[kSmallRun] = {m.y, m.z, m.w, p3};
#pragma unroll
        for (int i = 0; i < kSmallRun; ++i) {
            if (ps[i] == NONE) continue;  // uniform within the group
            const VT* src = reinterpret_cast<const VT*>(a.grads + (size_t)ps[i] * ra.d);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int j = glane + G * k;
                if (j < ra.NV) g[i][k] = __ldcs(src + j);
            }
        }
        VT acc[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            acc[k] = Vec<V>::zero();
            if (glane + G * k >= ra.NV) continue;
#pragma unroll
            for (int i = 0; i < kSmallRun; ++i)
                if (ps[i] != NONE) Vec<V>::add(acc[k], g[i][k]);  // 0 + g0 + g1 + ...: occurrence order
        }
        adagrad_store<V, KV>(ra, m.x, w, Gs, acc, glane, a.lr, a.eps);
    }
    if (a.release) release_counters(a.cur, a.release);  // when it is its stream's last kernel
}

template <int V, int KV>
__global__ void __launch_bounds__(256, MLKV_LONG_MIN_BLOCKS) k_long_sum(RowArgs ra, RunArgs a) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    const uint32_t NI = min(a.cur->n_items, a.max_items);
    const int lane = threadIdx.x & 31, G = ra.G, glane = lane & (G - 1), gid = lane / G;
    const unsigned gmask = group_mask(G, gid);
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) / G;
    const uint32_t ngroups = (gridDim.x * blockDim.x) / G;
    for (uint32_t it = group; it < NI; it += ngroups) {
        const uint32_t s = __ldg(a.item_s + it), e = __ldg(a.item_e + it);
        if (MLKV_CHECK && !in_bounds(a.err, kChkLongItem, e, (unsigned long long)a.n + 1)) continue;
        VT acc[KV], cmp[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            acc[k] = Vec<V>::zero();
            cmp[k] = Vec<V>::zero();
        }
        sum_rows<V, KV, MLKV_LONG_ROWS_IN_FLIGHT, false, true>(acc, cmp, a.grads, a.spos, s, e > s ? e - s : 0u,
                                                               ra.d, ra.NV, G, glane, gmask, a.err, kChkLongPos,
                                                               a.n);
        // the chunk's (sum, compensation) pair
        VT* part = reinterpret_cast<VT*>(a.partial + (size_t)it * 2 * ra.dpad);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < ra.NV) {
                __stcg(part + j, acc[k]);
                __stcg(part + ra.dpad / V + j, cmp[k]);
            }
        }
    }
}


// (acc, cmp) += the chunk pairs base + k0 .. base + k1 - 1, in that order, with
// eight vectors per lane in flight: each chunk's sum added with compensation,
// then its own compensation added to cmp.
template <int V, int KV>
__device__ __forceinline__ void sum_partials(typename Vec<V>::T (&acc)[KV], typename Vec<V>::T (&cmp)[KV],
                                             const RowArgs& ra, const float* partial, uint32_t base, uint32_t k0,
                                             uint32_t k1, int glane) {
    using VT = typename Vec<V>::T;
    constexpr int UNR = KV >= 4 ? 1 : 4 / KV;
    const int half = ra.dpad / V;
    for (uint32_t x = k0; x < k1; x += UNR) {
        VT g[UNR][KV], c[UNR][KV];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            const VT* src = reinterpret_cast<const VT*>(partial + (size_t)(base + x + u) * 2 * ra.dpad);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int j = glane + ra.G * k;
                if (x + u < k1 && j < ra.NV) {
                    g[u][k] = __ldcg(src + j);
                    c[u][k] = __ldcg(src + half + j);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u)
#pragma unroll
            for (int k = 0; k < KV; ++k)
                if (x + u < k1 && glane + ra.G * k < ra.NV) {
                    Vec<V>::cadd(acc[k], cmp[k], g[u][k]);
                    Vec<V>::add(cmp[k], c[u][k]);
                }
    }
}

// One launch for every long run.  A run of more than a.big chunk sums (the
// hottest rows) takes a whole block: its lane groups split the sums in a fixed
// way, then group 0 adds the groups' results in order.  Every other long run
// takes one lane group, which adds its sums in order.  Then the Adagrad step.
template <int V, int KV>
__global__ void __launch_bounds__(1024) k_long_combine(RowArgs ra, RunArgs a, DevState* ds) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    extern __shared__ float sh[];  // [groups][2][dpad]: each group's (sum, compensation) pair
    const uint32_t nl = min(a.cur->n_long, a.max_long), nb = a.cur->n_big;
    if (blockIdx.x == 0 && threadIdx.x == 0)
        ds->last_unique = a.cur->n_single + a.cur->n_small + a.cur->n_short + a.cur->n_long;  // one run per row
    const int G = ra.G, glane = threadIdx.x & (G - 1);
    const int group = threadIdx.x / G;
    const int ngroups = blockDim.x / G;
    for (uint32_t i = blockIdx.x; i < nb; i += gridDim.x) {  // block-uniform
        if (MLKV_CHECK && !in_bounds(a.err, kChkCombineRun, i, a.max_long)) break;
        const uint32_t h = a.big_runs[i];
        if (MLKV_CHECK && !in_bounds(a.err, kChkCombineRun, h, nl)) continue;
        const uint32_t base = a.long_base[h];
        const uint32_t m = (a.long_e[h] - a.long_s[h] + a.chunk - 1) / a.chunk;
        if (MLKV_CHECK && !(in_bounds(a.err, kChkCombineRun, base + m, (unsigned long long)a.max_items + 1) &&
                            in_bounds(a.err, kChkCombineRow, a.long_row[h], ra.nrows)))
            continue;
        const uint32_t per = (m + ngroups - 1) / ngroups;
        const uint32_t k0 = min(m, group * per), k1 = min(m, k0 + per);
        VT acc[KV], cmp[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            acc[k] = Vec<V>::zero();
            cmp[k] = Vec<V>::zero();
        }
        sum_partials<V, KV>(acc, cmp, ra, a.partial, base, k0, k1, glane);
        VT* mine = reinterpret_cast<VT*>(sh + (size_t)group * 2 * ra.dpad);
        const int half = ra.dpad / V;
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < ra.NV) {
                mine[j] = acc[k];
                mine[half + j] = cmp[k];
            }
        }
        __syncthreads();
        if (group == 0) {
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                acc[k] = Vec<V>::zero();
                cmp[k] = Vec<V>::zero();
            }
            for (int gi = 0; gi < ngroups; ++gi) {
                const VT* src = reinterpret_cast<const VT*>(sh + (size_t)gi * 2 * ra.dpad);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (j < ra.NV) {
                        Vec<V>::cadd(acc[k], cmp[k], src[j]);
                        Vec<V>::add(cmp[k], src[half + j]);
                    }
                }
            }
#pragma unroll
            for (int k = 0; k < KV; ++k) Vec<V>::add(acc[k], cmp[k]);  // the sum, rounded once
            VT w[KV], Gs[KV];
            const uint32_t row = a.long_row[h];
            load_row_state<V, KV>(ra, row, w, Gs, glane);
            adagrad_store<V, KV>(ra, row, w, Gs, acc, glane, a.lr, a.eps);
        }
        __syncthreads();
    }
    // the other long runs: on the blocks that took no big run (all blocks when
    // the big runs outnumber them)
    const uint32_t b0 = nb < gridDim.x ? nb : 0u;
    const uint32_t gg = (blockIdx.x - b0) * ngroups + group, ngg = (gridDim.x - b0) * ngroups;
    for (uint32_t h = blockIdx.x < b0 ? nl : gg; h < nl; h += ngg) {  // uniform within the group
        const uint32_t m = (a.long_e[h] - a.long_s[h] + a.chunk - 1) / a.chunk;
        if (m > a.big) continue;
        if (MLKV_CHECK && !(in_bounds(a.err, kChkCombineRun, a.long_base[h] + m, (unsigned long long)a.max_items + 1) &&
                            in_bounds(a.err, kChkCombineRow, a.long_row[h], ra.nrows)))
            continue;
        VT acc[KV], cmp[KV], w[KV], Gs[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            acc[k] = Vec<V>::zero();
            cmp[k] = Vec<V>::zero();
        }
        const uint32_t row = a.long_row[h];
        load_row_state<V, KV>(ra, row, w, Gs, glane);
        sum_partials<V, KV>(acc, cmp, ra, a.partial, a.long_base[h], 0u, m, glane);
#pragma unroll
        for (int k = 0; k < KV; ++k) Vec<V>::add(acc[k], cmp[k]);  // the sum, rounded once
        adagrad_store<V, KV>(ra, row, w, Gs, acc, glane, a.lr, a.eps);
    }
    if (a.release) release_counters(a.cur, a.release);
}

template <int V, int KV>
void launch_short(mlkv_table* t, bool narrow, int grid, cudaStream_t st, const RowArgs& ra, const RunArgs& a) {
    if (narrow)
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_SHORT, (k_short<V, KV, 4>), grid, 256, 0, st, ra, a);
    else
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_SHORT, (k_short<V, KV>), grid, 256, 0, st, ra, a);
}

template <int V, int KV>
cudaError_t run_reduce(mlkv_table* t, const float* grads, const uint32_t* srow, const uint32_t* spos,
                       int64_t n, uint32_t sent, cudaStream_t st, CallCounters* cur) {
    RowArgs ra{t->slots, t->geom.stride, t->geom.dpad, t->geom.NV, t->geom.G, t->geom.d,
               (uint32_t)(t->tiered ? t->cfg.hbm_cache_rows : t->cfg.capacity)};
    RunArgs a{grads, srow, spos, (uint32_t)n, sent, cur, t->s.short_runs, t->s.single_runs, t->s.small_runs,
              t->s.small_p3, t->s.long_s, t->s.long_e,
              t->s.long_row, t->s.long_base, t->s.item_s, t->s.item_e, t->s.big_runs, t->s.partial,
              (uint32_t)t->s.max_long,
              (uint32_t)t->s.max_items, n >= kSmallBatch ? kChunkLarge : kChunkSmall,
              n >= kSmallBatch ? kBigRunLarge : kBigRunSmall,
              ErrSink{&t->dstate->status, t->status_dev_alias, t->dstate->chk}, t->cfg.lr, t->cfg.eps};
    // a warp per 32 positions, the windows dealt out grid-stride over at most
    // one wave of blocks
#ifndef MLKV_HEADS_ONE_WAVE
#define MLKV_HEADS_ONE_WAVE 1
#endif
    const int64_t cap = MLKV_HEADS_ONE_WAVE ? persistent_blocks(t, (const void*)k_heads, 256) : (int64_t)t->num_sms * 8;
    int64_t gh = (n + 255) / 256;
    if (gh > cap) gh = cap;
    if (gh < 1) gh = 1;
    MLKV_LAUNCH(t, MLKV_K_SEGMENTS, k_heads, (unsigned)gh, 256, 0, st, a);
    // The runs of one lookup, of 2 .. kSmallRun and of up to
    // MLKV_SEQ_SEGMENT_MAX lookups, and the long runs (chunk sums, then their
    // combine) touch disjoint rows and scratch: they run on three streams at
    // once, each filling the others' tails, and join at the end of the call;
    // the last kernel of each stream releases the counters they read.
    cudaStream_t s1 = st, s2 = st;
    // While a kernel class is being timed (mlkv_time_kernel) the reduce kernels
    // run one after another: on three streams a kernel's events would also
    // span the time it waits for the SMs the others hold.
    const bool branches = MLKV_REDUCE_BRANCHES && t->timer.kernel_id == 0;
    if (branches) {
        cudaError_t e;
        if ((e = cudaEventRecord(t->ev_fork, st)) != cudaSuccess ||
            (e = cudaStreamWaitEvent(t->branch[0], t->ev_fork, 0)) != cudaSuccess ||
            (e = cudaStreamWaitEvent(t->branch[1], t->ev_fork, 0)) != cudaSuccess)
            return e;
        s1 = t->branch[0];
        s2 = t->branch[1];
    }
    const int gl = persistent_blocks(t, (const void*)k_long_sum<V, KV>, 256);
    const int g2 = persistent_blocks(t, (const void*)k_small<V, KV>, 256);
    const bool narrow = MLKV_NARROW_ROWS && t->geom.G <= 16;
    const void* short_k = narrow ? (const void*)k_short<V, KV, 4> : (const void*)k_short<V, KV>;
    const void* single_k = narrow ? (const void*)k_single<V, KV, 2> : (const void*)k_single<V, KV>;
    const int gs = persistent_blocks(t, short_k, 256);
    int g1 = persistent_blocks(t, single_k, 256);
    if (MLKV_SINGLE_PER_SM > 0 && g1 > MLKV_SINGLE_PER_SM * t->num_sms) g1 = MLKV_SINGLE_PER_SM * t->num_sms;
    if (narrow && g1 > 3 * t->num_sms) g1 = 3 * t->num_sms;
    // the combine's block (MLKV_COMBINE_THREADS): the groups' (sum,
    // compensation) pairs must fit the default 48 KB of shared memory
    int big = MLKV_COMBINE_THREADS;
    while (big > 64 && (size_t)(big / t->geom.G) * 2 * t->geom.dpad * sizeof(float) > 48 * 1024) big /= 2;
    const size_t smem = (size_t)(big / t->geom.G) * 2 * t->geom.dpad * sizeof(float);
    // 1024 threads per SM: 4,864 lane groups of 32 for the ordinary long runs
    const int gc = t->num_sms * (1024 / big);
    // The counters are released by the apply's last kernels: the last of each
    // stream (the combine, the last of the runs of 2-4 and of 5-32, the runs
    // of one), or the combine alone when all run in stream order.
    RunArgs last = a;
    const bool short_first = MLKV_SHORT_FIRST == 1 || (MLKV_SHORT_FIRST == 2 && n < (int64_t)kSmallBatch);
    last.release = (uint32_t)(gc + (branches ? g1 + (short_first ? g2 : gs) : 0));
    const RunArgs& tail = branches ? last : a;
    const cudaStream_t s_long = s2, s_single = st;
    MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_LONG, (k_long_sum<V, KV>), gl, 256, 0, s_long, ra, a);
    if (branches)
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_LONG_COMBINE, (k_long_combine<V, KV>), gc, big, smem, s_long, ra, last,
                               t->dstate);
    if (short_first) {
        // the runs of 5-32 (the longest per run of the three) before those of
        // 2-4: in a small batch the runs of 5-32 would otherwise be last to
        // start, after the runs of one had filled the SMs
        launch_short<V, KV>(t, narrow, gs, s1, ra, a);
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_SMALL, (k_small<V, KV>), g2, 256, 0, s1, ra, tail);
    } else {
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_SMALL, (k_small<V, KV>), g2, 256, 0, s1, ra, a);
        launch_short<V, KV>(t, narrow, gs, s1, ra, tail);
    }
    if (narrow)
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_SINGLE, (k_single<V, KV, 2>), g1, 256, 0, s_single, ra, tail);
    else
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_REDUCE_SINGLE, (k_single<V, KV>), g1, 256, 0, s_single, ra, tail);
    if (branches) {
        cudaError_t e;
        if ((e = cudaEventRecord(t->ev_join[0], s1)) != cudaSuccess ||
            (e = cudaEventRecord(t->ev_join[1], s2)) != cudaSuccess ||
            (e = cudaStreamWaitEvent(st, t->ev_join[0], 0)) != cudaSuccess ||
            (e = cudaStreamWaitEvent(st, t->ev_join[1], 0)) != cudaSuccess)
            return e;
    } else {
        MLKV_LAUNCH_PERSISTENT(t, MLKV_K_LONG_COMBINE, (k_long_combine<V, KV>), gc, big, smem, st, ra, last,
                               t->dstate);
    }
    return cudaGetLastError();
}

}  // namespace

int64_t long_runs_bound(int64_t max_batch) { return max_batch / (MLKV_SEQ_SEGMENT_MAX + 1) + 1; }

int64_t long_items_bound(int64_t max_batch) {
    // chunks of kChunkLarge lookups in calls of at least kSmallBatch lookups, of kChunkSmall below
    const int64_t small = std::min<int64_t>(max_batch, (int64_t)kSmallBatch - 1) / kChunkSmall;
    return std::max<int64_t>(max_batch / kChunkLarge, small) + long_runs_bound(max_batch) + 1;
}

cudaError_t launch_reduce_apply(mlkv_table* t, const float* grads, const uint32_t* srow,
                                const uint32_t* spos, int64_t n, uint32_t sent, cudaStream_t st,
                                CallCounters* cur) {
    const RowGeom& g = t->geom;
    if (g.V == 4) {
        switch (g.KV) {
            case 1: return run_reduce<4, 1>(t, grads, srow, spos, n, sent, st, cur);
            case 2: return run_reduce<4, 2>(t, grads, srow, spos, n, sent, st, cur);
            case 4: return run_reduce<4, 4>(t, grads, srow, spos, n, sent, st, cur);
            default: return run_reduce<4, 8>(t, grads, srow, spos, n, sent, st, cur);
        }
    }
    switch (g.KV) {
        case 1: return run_reduce<1, 1>(t, grads, srow, spos, n, sent, st, cur);
        case 2: return run_reduce<1, 2>(t, grads, srow, spos, n, sent, st, cur);
        case 4: return run_reduce<1, 4>(t, grads, srow, spos, n, sent, st, cur);
        default: return run_reduce<1, 8>(t, grads, srow, spos, n, sent, st, cur);
    }
}

}  // namespace mlkv
