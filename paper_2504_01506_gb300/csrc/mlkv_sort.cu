// Dedup of a gradient batch: a stable LSD radix sort of (row id, position)
// pairs, then the segment starts of the sorted row ids.
//
// The sort key is the 32-bit row id, not the 64-bit key: rows are dense in
// [0, capacity), so 3 passes of 9 bits cover 10^8 rows (against 5+ passes for
// 40-bit keys), and the sorted order visits rows in memory order.  An absent
// lookup is given the all-ones digit pattern and sorts last.
//
// Each pass is a reduce-then-scan pass over tiles of 4096 elements (1024 in
// batches of fewer than kSortSmallBatch lookups, which would otherwise cover a
// fraction of the SMs): the digit counts of every tile and the pass's digit
// totals come first; one kernel gives every (tile, digit) the output position
// of its first element (the elements of lower digits plus those of the digit
// in earlier tiles); a second ranks each tile's elements stably (over rounds
// of 32, in order) and scatters them.  The counts of the first pass are made
// by a histogram kernel, or in a gradient apply by the probe and the miss
// kernel (FirstCounts); those of every later pass by the scatter before it,
// which knows the tile each element lands in and adds the element's next digit
// to that tile's count (one add per run of equal targets in a warp), so no
// pass after the first reads its input twice.  No block waits on another, so
// a pass costs the same when the sort shares the GPU with other kernels.  (A
// single-pass decoupled look-back sort was slower here: a batch is about one
// wave of tiles, and the chain of tiles that know their prefix grows one
// window per round trip.)
#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

// the tiles of the segment scan (k_seg_*), and the block of the histogram and
// offsets kernels
constexpr int kThreads = 256;
constexpr int kItems = 16;
constexpr int kTile = kThreads * kItems;  // 4096
constexpr int kWarps = kThreads / 32;

// Exclusive scan of one value per thread over a block of THREADS threads.
template <int THREADS>
__device__ __forceinline__ uint32_t block_exclusive_scan_n(uint32_t v, uint32_t& total) {
    constexpr int kWarps = THREADS / 32;
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

__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t& total) {
    return block_exclusive_scan_n<kThreads>(v, total);
}

// Sum of tile_sums[0..b) by the whole block.
__device__ __forceinline__ uint32_t tiles_before(const uint32_t* __restrict__ tile_sums, uint32_t b) {
    uint32_t s = 0;
    for (uint32_t i = threadIdx.x; i < b; i += kThreads) s += tile_sums[i];
    uint32_t total;
    block_exclusive_scan(s, total);
    return total;
}

// --- radix sort ---------------------------------------------------------------
// Pass 0 reads the probe's row ids (sentinels mapped to `sent`) and uses the
// lookup position as the value.
__device__ __forceinline__ uint32_t sort_key(uint32_t r, uint32_t sent, bool first) {
    return first ? (r >= ROW_ABSENT ? sent : r) : r;
}

constexpr int kMaxRadix = kSortMaxRadix;

#ifndef MLKV_SORT_RANK_BALLOT
#define MLKV_SORT_RANK_BALLOT 1
#endif

// Lanes of the warp whose (valid, digit) equals this lane's: a warp match, or
// one ballot per digit bit.
__device__ __forceinline__ uint32_t digit_peers(uint32_t dig, bool valid, int bits) {
#if MLKV_SORT_RANK_BALLOT
    const uint32_t vm = __ballot_sync(0xffffffffu, valid);
    uint32_t peers = valid ? vm : ~vm;
    for (int b = 0; b < bits; ++b) {
        const bool one = (dig >> b) & 1u;
        const uint32_t m = __ballot_sync(0xffffffffu, one);
        peers &= one ? m : ~m;
    }
    return peers;
#else
    (void)bits;
    return __match_any_sync(0xffffffffu, valid ? dig : 0xFFFFFFFFu);
#endif
}

// Digit counts of one tile, written to column `tile` of counts[d][tile], and
// added to the pass's digit totals dtot[d]: the first pass of a sort whose
// counts the probe did not make.  A thread counts consecutive elements and
// adds a run of equal digits with one atomic.
template <int TILE>
__global__ void __launch_bounds__(TILE >= 1024 ? kThreads : TILE / 4) k_sort_hist(const uint32_t* __restrict__ kin, uint32_t n,
                                                        uint32_t* __restrict__ counts, uint32_t* __restrict__ dtot,
                                                        uint32_t ntiles, int shift, int radix, uint32_t sent,
                                                        int first) {
    constexpr int kHThreads = TILE >= 1024 ? kThreads : TILE / 4;
    constexpr int kItems = TILE / kHThreads;
    static_assert(kItems % 4 == 0, "whole 16-byte loads");
    pdl_enter();
    __shared__ uint32_t hist[kMaxRadix];
    for (int d = threadIdx.x; d < radix; d += kHThreads) hist[d] = 0;
    __syncthreads();
    const uint32_t i0 = blockIdx.x * TILE + threadIdx.x * kItems;
    uint32_t key[kItems];
    if (i0 + kItems <= n) {  // consecutive keys, 16-byte aligned
        const uint4* src = reinterpret_cast<const uint4*>(kin + i0);
#pragma unroll
        for (int q = 0; q < kItems / 4; ++q) {
            const uint4 v = __ldg(src + q);
            key[4 * q] = v.x;
            key[4 * q + 1] = v.y;
            key[4 * q + 2] = v.z;
            key[4 * q + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int r = 0; r < kItems; ++r) key[r] = i0 + r < n ? kin[i0 + r] : 0u;
    }
    uint32_t cur = 0xFFFFFFFFu, cnt = 0;
#pragma unroll
    for (int r = 0; r < kItems; ++r) {
        if (i0 + r >= n) break;
        const uint32_t dig = (sort_key(key[r], sent, first) >> shift) & (radix - 1);
        if (dig != cur) {
            if (cnt) atomicAdd(&hist[cur], cnt);
            cur = dig;
            cnt = 0;
        }
        ++cnt;
    }
    if (cnt) atomicAdd(&hist[cur], cnt);
    __syncthreads();
    for (int d = threadIdx.x; d < radix; d += kHThreads) {
        const uint32_t c = hist[d];
        counts[(size_t)d * ntiles + blockIdx.x] = c;
        if (c) atomicAdd(dtot + d, c);
    }
}

// Output position of the first element of every (tile, digit): the elements
// of all lower digits, plus those of digit d in earlier tiles; written to
// offsets[tile][d].  Each block of OT
// threads first scans the pass's digit totals (all of them) for the elements
// of the lower digits; then a warp per digit scans the digit's counts over the
// tiles, 32 tiles a round, with the loads of 16 rounds issued together (every
// tile of a batch of up to 2M lookups in one round trip).
#ifndef MLKV_OFFSETS_THREADS
#define MLKV_OFFSETS_THREADS 256
#endif
constexpr int kOThreads = MLKV_OFFSETS_THREADS;
#ifndef MLKV_OFFSETS_PDL
#define MLKV_OFFSETS_PDL 0
#endif
__global__ void __launch_bounds__(kOThreads) k_sort_offsets(const uint32_t* __restrict__ counts,
                                                            const uint32_t* __restrict__ dtot,
                                                            uint32_t* __restrict__ offsets, uint32_t ntiles,
                                                            int radix) {
    pdl_enter();
    constexpr int kPer = kMaxRadix / kOThreads;  // digit totals per thread
    constexpr int kRounds = 16;
    __shared__ uint32_t lower[kMaxRadix];  // elements of the digits below each digit
    {
        const int i0 = kPer * threadIdx.x;
        uint32_t v[kPer], sum = 0;
#pragma unroll
        for (int k = 0; k < kPer; ++k) {
            v[k] = i0 + k < radix ? __ldg(dtot + i0 + k) : 0u;
            sum += v[k];
        }
        uint32_t total;
        uint32_t ex = block_exclusive_scan_n<kOThreads>(sum, total);
#pragma unroll
        for (int k = 0; k < kPer; ++k) {
            lower[i0 + k] = ex;
            ex += v[k];
        }
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int d = blockIdx.x * (kOThreads / 32) + (threadIdx.x >> 5);
    if (d >= radix) return;  // warp-uniform
    const uint32_t* row = counts + (size_t)d * ntiles;
    uint32_t run = lower[d];
    for (uint32_t t0 = 0; t0 < ntiles; t0 += 32 * kRounds) {
        uint32_t c[kRounds];
#pragma unroll
        for (int k = 0; k < kRounds; ++k) {
            const uint32_t t = t0 + 32 * k + lane;
            c[k] = t < ntiles ? __ldg(row + t) : 0u;
        }
#pragma unroll
        for (int k = 0; k < kRounds; ++k) {
            if (t0 + 32 * k >= ntiles) break;  // warp-uniform
            const uint32_t t = t0 + 32 * k + lane;
            uint32_t x = c[k];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            if (t < ntiles) offsets[(size_t)t * radix + d] = run + x - c[k];
            run += __shfl_sync(0xffffffffu, x, 31);
        }
    }
}

// Stable rank of each element of the tile among equal digits; the tile is
// then laid out in shared memory in sorted order and written out so that
// consecutive threads write consecutive addresses of a digit's run (a direct
// scatter from registers costs one L2 sector per element).  The block has
// THREADS threads; warp w owns elements w*kSItems*32 .. of the tile, in
// rounds of 32 consecutive elements (more warps a tile: fewer rounds each).
// An element of digit d goes to offsets[tile][d] plus its rank among the
// tile's elements of digit d.  With nshift >= 0 the element's digit of the
// next pass (bits nshift ..) is added to the count of the tile of the next
// pass that holds its output position, ncounts[digit][dst / TILE] (zero on
// entry), and to the next pass's digit totals ndtot.  The counts this pass's
// offsets came from (`counts`, read by the offsets kernel, which has
// finished) are zeroed, for the pass after next to count into.
// threads of the scatter's block for the small tiles (4 elements a thread)
#ifndef MLKV_SCATTER_SMALL_THREADS
#define MLKV_SCATTER_SMALL_THREADS (kSortTileSmall / 4)
#endif
#ifndef MLKV_SCATTER_MIN_BLOCKS
#define MLKV_SCATTER_MIN_BLOCKS 3
#endif
template <int TILE, int THREADS>
__global__ void __launch_bounds__(THREADS, THREADS == 512 ? MLKV_SCATTER_MIN_BLOCKS : 4) k_sort_scatter(
    const uint32_t* __restrict__ kin, const uint32_t* __restrict__ vin, uint32_t* __restrict__ kout,
    uint32_t* __restrict__ vout, uint32_t n, const uint32_t* __restrict__ offsets, uint32_t ntiles, int shift,
    int radix, uint32_t sent, int first, uint32_t* __restrict__ dtot, int nshift, uint32_t* __restrict__ ncounts,
    uint32_t* __restrict__ ndtot, uint32_t* __restrict__ counts) {
    constexpr int kSWarps = THREADS / 32;
    constexpr int kSItems = TILE / THREADS;
    constexpr int kTileShift = TILE == 4096 ? 12 : TILE == 2048 ? 11 : TILE == 1024 ? 10 : 9;
    static_assert(TILE == (1 << kTileShift), "tiles of 512 .. 4096");
    pdl_enter();
    // the pass's digit totals were read by the offsets kernel, which has
    // finished: zero them for the next sort (the totals are zero between sorts)
    if (blockIdx.x == 0)
        for (int d = threadIdx.x; d < radix; d += THREADS) dtot[d] = 0u;
    // ... and this tile's column of the counts (radix x ntiles, a column a block)
    for (int d = threadIdx.x; d < radix; d += THREADS) counts[(size_t)d * ntiles + blockIdx.x] = 0u;
    // the per-warp digit counts, then (once every position is known) the sorted tile
    __shared__ uint32_t pool[2 * TILE];
    constexpr bool kShare = kSWarps * kMaxRadix <= 2 * TILE;  // the counts fit the tile buffer
    __shared__ uint32_t wpool[kShare ? 1 : kSWarps * kMaxRadix];
    uint32_t (*wcnt)[kMaxRadix] = reinterpret_cast<uint32_t (*)[kMaxRadix]>(kShare ? pool : wpool);
    uint32_t* skey = pool;
    uint32_t* sval = pool + TILE;
    __shared__ uint32_t gbase[kMaxRadix];   // output position of the tile's first element of each digit
    __shared__ uint32_t lbase[kMaxRadix];   // position in the sorted tile of its first element of each digit
    __shared__ uint32_t ntot[kMaxRadix];    // the tile's elements of each digit of the next pass
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < kSWarps * kMaxRadix; i += THREADS) (&wcnt[0][0])[i] = 0;
    for (int d = threadIdx.x; d < radix; d += THREADS) {
        gbase[d] = offsets[(size_t)blockIdx.x * radix + d];
        ntot[d] = 0u;
    }
    __syncthreads();
    const uint32_t tile0 = blockIdx.x * TILE;
    const uint32_t base = tile0 + w * (kSItems * 32);
    const int digit_bits = __ffs(radix) - 1;
    const uint32_t lt = lanemask_lt();
    uint32_t key[kSItems], val[kSItems], rnk[kSItems];
    // all loads first, so they are in flight together
#pragma unroll
    for (int r = 0; r < kSItems; ++r) {
        const uint32_t i = base + r * 32 + lane;
        key[r] = i < n ? sort_key(kin[i], sent, first) : 0u;
        val[r] = i < n ? (first ? i : vin[i]) : 0u;
    }
#pragma unroll
    for (int r = 0; r < kSItems; ++r) {
        const bool valid = base + r * 32 + lane < n;
        const uint32_t dig = (key[r] >> shift) & (radix - 1);
        const uint32_t peers = digit_peers(dig, valid, digit_bits);
        uint32_t before = 0;
        if (valid) before = wcnt[w][dig];
        __syncwarp();
        if (valid && lane == __ffs(peers) - 1) wcnt[w][dig] = before + __popc(peers);
        __syncwarp();
        rnk[r] = valid ? before + __popc(peers & lt) : 0xFFFFFFFFu;
    }
    __syncthreads();
    // per digit: exclusive prefix over the warps; per tile: exclusive prefix
    // over the digits (thread t owns digits t*dpt .. t*dpt+dpt-1, in order)
    constexpr int kDpt = kMaxRadix > THREADS ? kMaxRadix / THREADS : 1;
    const int dpt = radix > THREADS ? radix / THREADS : 1;
    uint32_t tot[kDpt], mine = 0;
#pragma unroll
    for (int j = 0; j < kDpt; ++j) {
        const int d = threadIdx.x * dpt + j;
        tot[j] = 0;
        if (j >= dpt || d >= radix) continue;
#pragma unroll
        for (int ww = 0; ww < kSWarps; ++ww) {
            const uint32_t c = wcnt[ww][d];
            wcnt[ww][d] = tot[j];
            tot[j] += c;
        }
        mine += tot[j];
    }
    uint32_t all;
    uint32_t run = block_exclusive_scan_n<THREADS>(mine, all);
#pragma unroll
    for (int j = 0; j < kDpt; ++j) {
        const int d = threadIdx.x * dpt + j;
        if (j >= dpt || d >= radix) continue;
        lbase[d] = run;
        run += tot[j];
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kSItems; ++r) {
        if (rnk[r] == 0xFFFFFFFFu) continue;
        const uint32_t dig = (key[r] >> shift) & (radix - 1);
        rnk[r] += lbase[dig] + wcnt[w][dig];  // position in the sorted tile
    }
    __syncthreads();  // the counts are dead: the buffer takes the sorted tile
#pragma unroll
    for (int r = 0; r < kSItems; ++r) {
        if (rnk[r] == 0xFFFFFFFFu) continue;
        skey[rnk[r]] = key[r];
        sval[rnk[r]] = val[r];
    }
    __syncthreads();
    const uint32_t cnt = n - tile0 < (uint32_t)TILE ? n - tile0 : (uint32_t)TILE;
    if (nshift < 0) {
        for (uint32_t l = threadIdx.x; l < cnt; l += THREADS) {
            const uint32_t k = skey[l];
            const uint32_t dig = (k >> shift) & (radix - 1);
            const uint32_t dst = gbase[dig] + (l - lbase[dig]);
            kout[dst] = k;
            vout[dst] = sval[l];
        }
        return;
    }
    // every lane of the warp takes part in each round (the last may be partial)
    for (uint32_t l0 = threadIdx.x - lane; l0 < cnt; l0 += THREADS) {
        const uint32_t l = l0 + lane;
        const bool valid = l < cnt;
        uint32_t target = 0xFFFFFFFFu, e = 0;
        if (valid) {
            const uint32_t k = skey[l];
            const uint32_t dig = (k >> shift) & (radix - 1);
            const uint32_t dst = gbase[dig] + (l - lbase[dig]);
            kout[dst] = k;
            vout[dst] = sval[l];
            e = (k >> nshift) & (radix - 1);
            target = e * ntiles + (dst >> kTileShift);
        }
        // consecutive lanes with one target (a hot row's lookups, a digit's
        // run within one tile) add their count once, from the run's first lane
        const uint32_t prev = __shfl_up_sync(0xffffffffu, target, 1);
        const bool head = valid && (lane == 0 || prev != target);
        const uint32_t heads = __ballot_sync(0xffffffffu, head);
        const uint32_t nvalid = __popc(__ballot_sync(0xffffffffu, valid));
        if (head) {
            const uint32_t later = heads & ~((2u << lane) - 1u);
            const uint32_t len = (later ? (uint32_t)(__ffs(later) - 1) : nvalid) - (uint32_t)lane;
            atomicAdd(ncounts + target, len);
            atomicAdd(&ntot[e], len);
        }
    }
    __syncthreads();
    for (int d = threadIdx.x; d < radix; d += THREADS) {
        const uint32_t c = ntot[d];
        if (c) atomicAdd(ndtot + d, c);
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
    pdl_enter();
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
    pdl_enter();
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
                            const uint32_t* __restrict__ seg_start, CallCounters* cur,
                            int64_t* __restrict__ uniq, int32_t* __restrict__ counts, int64_t* num) {
    pdl_enter();
    const uint32_t U = cur->n_unique, nv = cur->n_valid;
    if (blockIdx.x == 0 && threadIdx.x == 0) *num = (int64_t)U;
    for (uint32_t u = blockIdx.x * blockDim.x + threadIdx.x; u < U; u += gridDim.x * blockDim.x) {
        const uint32_t s = seg_start[u];
        const uint32_t e = u + 1 < U ? seg_start[u + 1] : nv;
        uniq[u] = keys[spos[s]];
        counts[u] = (int32_t)(e - s);
    }
    release_counters(cur, gridDim.x);  // the dedup's last kernel
}

inline unsigned tiles(int64_t n) { return (unsigned)((n + kTile - 1) / kTile); }

}  // namespace

namespace {
// Passes and digit width for ids of `bits` bits: the fewest passes of at most
// kSortMaxDigitBits bits, the bits spread evenly over them.
void sort_geometry(int bits, int& passes, int& D) {
    passes = (bits + kSortMaxDigitBits - 1) / kSortMaxDigitBits;
    D = (bits + passes - 1) / passes;
}
}  // namespace

inline unsigned sort_tiles(int64_t n) {
    const int sh = sort_tile_shift(n);
    return (unsigned)((n + (1 << sh) - 1) >> sh);
}

FirstCounts first_counts(mlkv_table* t, int64_t n) {
    int passes, D;
    sort_geometry(t->sort_bits, passes, D);
    return FirstCounts{t->s.sort_counts, t->s.sort_dtot, sort_tiles(n), 1 << D,
                       (uint32_t)((1ull << t->sort_bits) - 1), sort_tile_shift(n)};
}

namespace {
template <int TILE, int THREADS>
void sort_passes(mlkv_table* t, int64_t n, cudaStream_t st, const uint32_t** srow, const uint32_t** spos,
                 bool first_counted, int passes, int D) {
    const int radix = 1 << D;
    const uint32_t sent = (uint32_t)((1ull << t->sort_bits) - 1);
    const unsigned nt = sort_tiles(n);
    // two count buffers in turn: pass p's counts are in counts[p & 1], and its
    // scatter counts pass p + 1 into counts[(p + 1) & 1]
    uint32_t* counts[2] = {t->s.sort_counts, t->s.sort_counts2};
    uint32_t* offsets = t->s.sort_offsets;
    // the digit totals of every pass, and the second count buffer, are zero
    // between sorts (the arena starts zeroed; each pass's scatter zeroes its
    // pass's totals and the counts its offsets came from; the first pass's
    // counts are written whole by the probe or the histogram kernel)
    const uint32_t* kin = t->s.row_of_pos;
    const uint32_t* vin = nullptr;
    int out = 0;
    for (int p = 0; p < passes; ++p) {
        const int first = p == 0;
        uint32_t* dtot = t->s.sort_dtot + p * kMaxRadix;
        if (first && !first_counted)
            MLKV_LAUNCH(t, 0, k_sort_hist<TILE>, nt, TILE >= 1024 ? kThreads : TILE / 4, 0, st, kin, (uint32_t)n,
                        counts[0], dtot, nt, 0,
                        radix, sent, first);
        // launched after the kernel before it has finished, not beside its
        // drain: placed early, its few blocks landed on the SMs the scatter
        // left room on (a tenth of them) and took twice as long
        MLKV_LAUNCH_PDL(MLKV_OFFSETS_PDL != 0, t, 0, k_sort_offsets,
                        (unsigned)((radix + kOThreads / 32 - 1) / (kOThreads / 32)), kOThreads, 0, st,
                        counts[p & 1], dtot, offsets, nt, radix);
        // every pass but the last counts the next one
        const int nshift = p + 1 < passes ? (p + 1) * D : -1;
        MLKV_LAUNCH(t, MLKV_K_SORT_SCATTER, (k_sort_scatter<TILE, THREADS>), nt, THREADS, 0, st, kin, vin,
                    t->s.sk[out], t->s.sv[out], (uint32_t)n, offsets, nt, p * D, radix, sent, first, dtot, nshift,
                    counts[(p + 1) & 1], nshift < 0 ? nullptr : t->s.sort_dtot + (p + 1) * kMaxRadix,
                    counts[p & 1]);
        kin = t->s.sk[out];
        vin = t->s.sv[out];
        out ^= 1;
    }
    *srow = kin;
    *spos = vin;
}
}  // namespace

cudaError_t launch_sort_rows(mlkv_table* t, int64_t n, cudaStream_t st, const uint32_t** srow,
                             const uint32_t** spos, bool first_counted) {
    int passes, D;
    sort_geometry(t->sort_bits, passes, D);
    if (sort_tile_shift(n) == 12)
        sort_passes<kSortTile, 512>(t, n, st, srow, spos, first_counted, passes, D);
    else
        sort_passes<kSortTileSmall, MLKV_SCATTER_SMALL_THREADS>(t, n, st, srow, spos, first_counted, passes, D);
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
