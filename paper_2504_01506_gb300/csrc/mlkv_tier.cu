// Tiered store: an HBM cache of rows over a host-memory tier.  MLKV keeps its
// store on disk behind an in-memory buffer and prefetches future keys into that
// buffer (Section 3.3.2, look-ahead prefetching); here the backing tier is
// pinned host memory reached over the host link, and the buffer is HBM.
//
// Every row (with its Adagrad state) lives in exactly one place: a cache line,
// or a host slot.  Metadata (device):
//   row_loc[row]     a cache line (< LOC_HOST), LOC_HOST | host slot, or
//                    LOC_CLAIMED while a fetch of the row is in progress
//   line_row[line]   row held by the line, or LINE_NONE
//   line_stamp[line] epoch of the last call that used the line (all ones
//                    until the line is first handed out)
// Row r starts in host slot r.  A call (epoch e) runs, after the probe:
//   resolve  per lookup: a hit pins its line (stamp = max(stamp, e)); the first
//            lookup of a row held in a host slot claims the row (CAS slot ->
//            CLAIMED) and lists (row, slot) for fetch;
//   fetch    per listed row: take a never-used line or the next line of a
//            clock sweep whose stamp is older than keep_from (so lines of the
//            current call, and of a look-ahead in flight, are never taken),
//            then swap: the row comes in from its host slot and the victim goes
//            out to that same slot;
//   remap    per lookup: row id -> line id; the Get / apply kernels then work
//            on the cache as their slot array.
// With the swap no row has a fixed home and no dirty flags are kept: every
// victim is written back, changed or not (under Adagrad every cached row has
// changed).  Writing it to the 1 KiB just read needs no second address
// translation, which halves the cost on host memory reached through the CPU's
// page tables; on the driver-allocated tier it costs the same as a write-back
// elsewhere.
// Host-tier rows are moved by the GPU itself (zero-copy loads and stores over
// the mapped host memory): the fetch list never leaves the device, so the
// copies overlap other work without a host round trip.
#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

constexpr uint32_t LINE_NONE = 0xFFFFFFFFu;

// Blocks of the fetch kernel (8 warps each; set at build time).  The host link
// needs a few hundred rows in flight, not the whole GPU: more warps only queue
// on it, and a small grid leaves the SMs to the apply that runs beside a
// look-ahead.
#ifndef MLKV_TIER_FETCH_BLOCKS
#define MLKV_TIER_FETCH_BLOCKS 38
#endif
constexpr int kSweepLimit = 1 << 16;  // bounded clock sweep per group of rows (32 lines a round)

__device__ __forceinline__ uint32_t ld_relaxed_u32(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__global__ void __launch_bounds__(256) k_tier_init(uint32_t* __restrict__ row_loc, uint32_t n) {
    for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < n; r += gridDim.x * blockDim.x)
        row_loc[r] = LOC_HOST | r;
}

__global__ void __launch_bounds__(256) k_tier_resolve(TierArgs ta, const uint32_t* __restrict__ row_of_pos,
                                                      uint32_t n, uint2* fetch, uint32_t* n_fetch) {
    pdl_enter();
    const uint32_t p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n) return;
    const uint32_t r = row_of_pos[p];
    if (r >= ROW_ABSENT) return;
    const uint32_t l = ld_relaxed_u32(ta.row_loc + r);
    if (l < LOC_HOST) {
        // hot rows are looked up 10^4-10^5 times a call: one atomic per line
        uint32_t old = ld_relaxed_u32(ta.line_stamp + l);
        if (old < ta.epoch) old = atomicMax(ta.line_stamp + l, ta.epoch);
        // a call overlapping a look-ahead may only use lines of the Get before it
        if (ta.strict && old < ta.keep_from) record_error(ta.err, MLKV_ERR_INVALID);
        return;
    }
    if (ta.strict) {
        record_error(ta.err, MLKV_ERR_INVALID);
        return;
    }
    if (l != LOC_CLAIMED && atomicCAS(ta.row_loc + r, l, LOC_CLAIMED) == l) {
        const unsigned m = __activemask();
        const int lane = threadIdx.x & 31, leader = __ffs(m) - 1;
        uint32_t base = 0;
        if (lane == leader) base = atomicAdd(n_fetch, (uint32_t)__popc(m));
        base = __shfl_sync(m, base, leader);
        fetch[base + __popc(m & lanemask_lt())] = make_uint2(r, l & ~LOC_HOST);
    }
}

// One warp per group of up to 32 fetched rows (rows warp, warp + nwarps, ...).
// The warp first takes a line for each row of the group: never-used lines
// first (one atomic for the group; an unused line's stamp is the maximum, so
// the sweep never sees it), then the clock sweep, 32 lines a round, where the
// lines whose stamp is older than keep_from are claimed by CAS in lane order.
// Then it swaps each row: the row comes in from its host slot, the line's
// victim goes out to that slot.  A slot (row + state) is `stride` floats,
// moved as float4, KV per lane.
template <int KV>
__global__ void __launch_bounds__(256) k_tier_fetch(TierArgs ta, const uint2* __restrict__ fetch,
                                                    const uint32_t* n_fetch) {
    pdl_enter();
    __shared__ uint32_t s_line[8][32];
    const uint32_t nf = *n_fetch;
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const uint32_t warp = blockIdx.x * (blockDim.x >> 5) + wib;
    const uint32_t nwarps = gridDim.x * (blockDim.x >> 5);
    const int nvec = ta.stride / 4;
    uint32_t* lines = s_line[wib];
    uint32_t fetched = 0, written = 0;
    for (uint32_t g0 = warp; g0 < nf; g0 += 32 * nwarps) {
        const uint32_t left = (nf - g0 + nwarps - 1) / nwarps;
        const uint32_t need = left < 32 ? left : 32;
        lines[lane] = LINE_NONE;
        uint32_t got = 0;
        unsigned long long f0 = 0;
        if (lane == 0 && ld_relaxed_u64(ta.free_next) < ta.C) f0 = atomicAdd(ta.free_next, (unsigned long long)need);
        else if (lane == 0) f0 = ta.C;
        f0 = __shfl_sync(0xffffffffu, f0, 0);
        if (f0 < ta.C) {
            const uint32_t room = (uint32_t)(ta.C - f0);
            got = need < room ? need : room;
            if ((uint32_t)lane < got) {
                lines[lane] = (uint32_t)f0 + lane;
                ta.line_stamp[f0 + lane] = ta.epoch;  // the line is this warp's alone
            }
        }
        for (int it = 0; got < need && it < kSweepLimit; ++it) {
            unsigned long long h0 = 0;
            if (lane == 0) h0 = atomicAdd(ta.clock, 32ull);
            h0 = __shfl_sync(0xffffffffu, h0, 0);
            const uint32_t h = (uint32_t)((h0 + lane) % ta.C);
            const uint32_t st = ld_relaxed_u32(ta.line_stamp + h);
            const unsigned elig = __ballot_sync(0xffffffffu, st < ta.keep_from);
            const uint32_t rank = __popc(elig & lanemask_lt());
            const bool won = ((elig >> lane) & 1u) && got + rank < need &&
                             atomicCAS(ta.line_stamp + h, st, ta.epoch) == st;
            const unsigned wins = __ballot_sync(0xffffffffu, won);
            __syncwarp();
            if (won) lines[got + __popc(wins & lanemask_lt())] = h;
            got += __popc(wins);
        }
        __syncwarp();
        for (uint32_t j = 0; j < need; ++j) {
            const uint2 fr = fetch[g0 + j * nwarps];  // (row, host slot)
            const uint32_t line = lines[j];
            if (line == LINE_NONE) {  // the sweep gave up: every line is held by the current call
                if (lane == 0) {
                    record_error(ta.err, MLKV_ERR_FULL);
                    ta.row_loc[fr.x] = LOC_HOST | fr.y;
                }
                continue;
            }
            const uint32_t victim = ta.line_row[line];
            float4* hs = reinterpret_cast<float4*>(ta.host + (size_t)fr.y * ta.stride);
            float4* cl = reinterpret_cast<float4*>(ta.cache + (size_t)line * ta.stride);
            float4 in[KV], out[KV];
#pragma unroll
            for (int k = 0; k < KV; ++k)
                if (lane + 32 * k < nvec) in[k] = hs[lane + 32 * k];
            if (victim != LINE_NONE) {
#pragma unroll
                for (int k = 0; k < KV; ++k)
                    if (lane + 32 * k < nvec) out[k] = cl[lane + 32 * k];
#pragma unroll
                for (int k = 0; k < KV; ++k)
                    if (lane + 32 * k < nvec) hs[lane + 32 * k] = out[k];
            }
#pragma unroll
            for (int k = 0; k < KV; ++k)
                if (lane + 32 * k < nvec) cl[lane + 32 * k] = in[k];
            if (lane == 0) {
                // the next kernel on the stream (remap) reads row_loc: no fence needed
                if (victim != LINE_NONE) ta.row_loc[victim] = LOC_HOST | fr.y;
                ta.line_row[line] = fr.x;
                ta.row_loc[fr.x] = line;
            }
            ++fetched;
            written += victim != LINE_NONE;
        }
        __syncwarp();
    }
    if (lane == 0 && fetched) {
        atomicAdd(ta.totals, (unsigned long long)fetched);
        if (written) atomicAdd(ta.totals + 1, (unsigned long long)written);
    }
}

__global__ void __launch_bounds__(256) k_tier_remap(TierArgs ta, uint32_t* __restrict__ row_of_pos, uint32_t n) {
    pdl_enter();
    const uint32_t p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n) return;
    const uint32_t r = row_of_pos[p];
    if (r >= ROW_ABSENT) return;
    const uint32_t l = ta.row_loc[r];
    row_of_pos[p] = l < LOC_HOST ? l : ROW_ABSENT;
}

// Get from the cache: the warp's lane groups copy the rows of 32 lookups.
template <int V, int KV>
__global__ void __launch_bounds__(256) k_gather_lines(const float* __restrict__ slots, int stride, int d, int NV,
                                                      int G, const uint32_t* __restrict__ row_of_pos, uint32_t n,
                                                      float* __restrict__ out) {
    pdl_enter();
    using VT = typename Vec<V>::T;
    const int lane = threadIdx.x & 31;
    const uint32_t base = (blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5)) * 32u;
    if (base >= n) return;
    const uint32_t row = base + lane < n ? row_of_pos[base + lane] : ROW_PENDING;
    const int R = 32 / G, glane = lane & (G - 1), gid = lane / G;
    for (int it = 0; it < G; ++it) {
        const int q = it * R + gid;
        const uint32_t r = __shfl_sync(0xffffffffu, row, q);
        if (r == ROW_PENDING) continue;
        const VT* src = reinterpret_cast<const VT*>(slots + (size_t)(r < ROW_ABSENT ? r : 0) * stride);
        VT* dst = reinterpret_cast<VT*>(out + (size_t)(base + q) * d);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < NV) __stcs(dst + j, r >= ROW_ABSENT ? Vec<V>::nan() : __ldg(src + j));
        }
    }
}

template <int V, int KV>
cudaError_t run_gather(mlkv_table* t, const uint32_t* rows, int64_t n, float* out, cudaStream_t st) {
    const RowGeom& g = t->geom;
    MLKV_LAUNCH(t, MLKV_K_GET_GATHER, (k_gather_lines<V, KV>), (unsigned)((n + 255) / 256), 256, 0, st, t->slots,
                g.stride, g.d, g.NV, g.G, rows, (uint32_t)n, out);
    return cudaGetLastError();
}

}  // namespace

TierArgs tier_args(mlkv_table* t, uint32_t epoch, uint32_t keep_from, int strict) {
    TierArgs ta;
    ta.row_loc = t->tier.row_loc;
    ta.line_row = t->tier.line_row;
    ta.line_stamp = t->tier.line_stamp;
    ta.cache = t->tier.cache;
    ta.host = t->tier.host_dev;
    ta.stride = t->geom.stride;
    ta.C = (uint32_t)t->cfg.hbm_cache_rows;
    ta.free_next = t->tier.ctr;
    ta.clock = t->tier.ctr + 1;
    ta.totals = t->tier.ctr + 2;
    ta.epoch = epoch;
    ta.keep_from = keep_from;
    ta.strict = (uint32_t)strict;
    ta.err = ErrSink{&t->dstate->status, t->status_dev_alias};
    return ta;
}

cudaError_t launch_tier_init(mlkv_table* t, cudaStream_t st) {
    const int64_t n = t->cfg.capacity;
    int64_t g = (n + 255) / 256;
    if (g > (int64_t)t->num_sms * 8) g = (int64_t)t->num_sms * 8;
    k_tier_init<<<(unsigned)g, 256, 0, st>>>(t->tier.row_loc, (uint32_t)n);
    return cudaGetLastError();
}

cudaError_t launch_tier_resolve(mlkv_table* t, const TierArgs& ta, uint32_t* row_of_pos, int64_t n, uint2* fetch,
                                uint32_t* n_fetch, bool remap, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(n_fetch, 0, sizeof(uint32_t), st);
    if (e != cudaSuccess) return e;
    const unsigned g = (unsigned)((n + 255) / 256);
    MLKV_LAUNCH(t, 0, k_tier_resolve, g, 256, 0, st, ta, row_of_pos, (uint32_t)n, fetch, n_fetch);
    if (!ta.strict) {
        // a warp per fetched row; at most one row per lookup
        int64_t fg = (n + 7) / 8;
        const int64_t cap = MLKV_TIER_FETCH_BLOCKS;
        if (fg > cap) fg = cap;
        if (fg < 1) fg = 1;
        const int kv = (t->geom.stride / 4 + 31) / 32;
        if (kv <= 2)
            MLKV_LAUNCH(t, MLKV_K_TIER_FETCH, k_tier_fetch<2>, (unsigned)fg, 256, 0, st, ta, fetch, n_fetch);
        else if (kv <= 4)
            MLKV_LAUNCH(t, MLKV_K_TIER_FETCH, k_tier_fetch<4>, (unsigned)fg, 256, 0, st, ta, fetch, n_fetch);
        else if (kv <= 8)
            MLKV_LAUNCH(t, MLKV_K_TIER_FETCH, k_tier_fetch<8>, (unsigned)fg, 256, 0, st, ta, fetch, n_fetch);
        else
            MLKV_LAUNCH(t, MLKV_K_TIER_FETCH, k_tier_fetch<16>, (unsigned)fg, 256, 0, st, ta, fetch, n_fetch);
    }
    if (remap) MLKV_LAUNCH(t, 0, k_tier_remap, g, 256, 0, st, ta, row_of_pos, (uint32_t)n);
    return cudaGetLastError();
}

cudaError_t launch_gather_lines(mlkv_table* t, const uint32_t* rows, int64_t n, float* out, cudaStream_t st) {
    const RowGeom& g = t->geom;
    if (g.V == 4) {
        switch (g.KV) {
            case 1: return run_gather<4, 1>(t, rows, n, out, st);
            case 2: return run_gather<4, 2>(t, rows, n, out, st);
            case 4: return run_gather<4, 4>(t, rows, n, out, st);
            default: return run_gather<4, 8>(t, rows, n, out, st);
        }
    }
    switch (g.KV) {
        case 1: return run_gather<1, 1>(t, rows, n, out, st);
        case 2: return run_gather<1, 2>(t, rows, n, out, st);
        case 4: return run_gather<1, 4>(t, rows, n, out, st);
        default: return run_gather<1, 8>(t, rows, n, out, st);
    }
}

}  // namespace mlkv
