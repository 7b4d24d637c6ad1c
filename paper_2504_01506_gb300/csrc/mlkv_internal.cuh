// Internal declarations of the GB300 embedding key-value store: the table
// object, its HBM layout, device helpers and the launchers each .cu exports.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "../../include/mlkv_gpu.h"

namespace mlkv {

// ---------------------------------------------------------------------------
// Index slot: 16 bytes, two per 32-byte sector.  An empty slot holds the
// reserved key ~0 with row = ROW_PENDING and aux = AUX_IDLE, so a key made
// visible by a compare-and-swap is always paired with a pending row.
struct __align__(16) Slot {
    unsigned long long key;
    uint32_t row;  // dense row id, or ROW_PENDING while the key is being inserted
    uint32_t aux;  // insertion: first position of the key in the batch; Put: last position
};

constexpr unsigned long long EMPTY_KEY = ~0ull;
constexpr uint32_t ROW_PENDING = 0xFFFFFFFFu;   // key present, row not handed out yet
constexpr uint32_t ROW_ABSENT = 0xFFFFFFFEu;    // key absent (or rejected)
constexpr uint32_t AUX_IDLE = 0xFFFFFFFFu;
constexpr int PROBE_LIMIT = MLKV_PROBE_LIMIT;
constexpr int kSortMaxPasses = 4;      // row ids have at most 31 bits
constexpr int kSortMaxDigitBits = 9;   // radix <= 512
constexpr int kSortMaxRadix = 1 << kSortMaxDigitBits;
constexpr int kSortTile = 4096;        // lookups per tile of a sort pass ...
#ifndef MLKV_SORT_SMALL_TILE_SHIFT
#define MLKV_SORT_SMALL_TILE_SHIFT 10
#endif
constexpr int kSortTileSmallShift = MLKV_SORT_SMALL_TILE_SHIFT;
constexpr int kSortTileSmall = 1 << kSortTileSmallShift;  // ... and in batches of fewer than kSortSmallBatch lookups
static_assert(kSortTileSmallShift >= 9 && kSortTileSmallShift <= 11, "small tiles of 512 .. 2048 lookups");
#ifndef MLKV_SORT_SMALL_BATCH
#define MLKV_SORT_SMALL_BATCH (1u << 19)
#endif
constexpr uint32_t kSortSmallBatch = MLKV_SORT_SMALL_BATCH;
// log2 of the sort's tile for a batch of n lookups: small batches take small
// tiles, so that a pass still spreads over the SMs (200k lookups are 49 tiles
// of 4096 but 196 of 1024)
inline int sort_tile_shift(int64_t n) { return n < (int64_t)kSortSmallBatch ? kSortTileSmallShift : 12; }
constexpr int kSmallRun = 4;           // runs of 2 .. kSmallRun lookups carry their positions in their record
constexpr int64_t kMaxStaleness = MLKV_MAX_STALENESS;  // largest bound kept below no bound

// Per-call counters.  Two copies: a call uses cc[p] and its first kernel
// zeroes cc[p ^ 1] for the next call, so no memset is enqueued.
struct CallCounters {
    uint32_t n_miss;     // lookups whose key had no row yet
    uint32_t n_new;      // distinct new keys (first occurrences)
    uint32_t n_unique;   // distinct rows after the sort
    uint32_t n_valid;    // lookups with a row
    uint32_t n_long;     // runs longer than MLKV_SEQ_SEGMENT_MAX
    uint32_t n_items;    // chunks of the long runs
    uint32_t n_short;    // runs of at most MLKV_SEQ_SEGMENT_MAX lookups
    uint32_t n_big;      // long runs whose chunk sums are combined by the wide blocks
    uint32_t n_single;   // runs of one lookup
    uint32_t short_next; // next chunk of short runs to claim (k_short's dynamic hand-out)
    uint32_t n_small;    // runs of 2 .. kSmallRun lookups (their positions in the record)
    uint32_t bar[4];     // arrivals at the miss kernel's grid barriers
    uint32_t done;       // blocks of the call's last kernel that have finished (release_counters)
};

struct DevState {
    unsigned long long next_row;  // rows handed out so far
    uint32_t status;              // first device-detected error (MLKV_ERR_*), sticky
    uint32_t last_unique;         // distinct rows of the last gradient apply
    CallCounters cc[2];           // the counters of every call but the gradient apply, in turn
    CallCounters cca[2];          // the gradient apply's, in turn
    uint32_t chk[3];              // bounds-checked build: first failed check (site, index, bound)
};

// Row-kernel geometry: a row of d floats is NV vectors of V floats; a group of
// G lanes (a power of two <= 32) owns one row, each lane KV vectors of it.
struct RowGeom {
    int d;        // dim
    int V;        // 4 (float4) or 1
    int NV;       // vectors per row
    int G;        // lanes per row
    int KV;       // vectors per lane, 1/2/4/8
    int dpad;     // row and state stride inside a slot (floats, multiple of 8)
    int stride;   // floats per slot (row + state) = 2 * dpad
};

// The table.  Device memory layout in HBM:
//   slots   [capacity][2 * dpad] fp32: w[0..d) | pad | G[0..d) | pad  (32-byte aligned)
//   index   [nslots] Slot, nslots = 2^k >= 2 * capacity
//   scratch arena sized for max_batch (see Scratch)
struct Scratch {
    uint32_t* row_of_pos;   // [max_batch]
    uint32_t* slot_of_pos;  // [max_batch] (Put)
    int64_t* memo_key;      // [max_batch] key of each position of the last Get (see Memo)
    uint32_t* memo_row;     // [max_batch] its row, ROW_PENDING at open
    uint32_t* miss_pos;     // [max_batch]
    uint32_t* miss_slot;    // [max_batch]
    uint32_t* first_flag;   // [max_batch], zero at rest
    uint32_t* rank;         // [max_batch]
    uint32_t* sk[2];        // sort keys (row ids), ping-pong [max_batch]
    uint32_t* sv[2];        // sort values (positions), ping-pong [max_batch]
    uint32_t* sort_counts;  // [512][tiles] digit counts of the sort's even passes ...
    uint32_t* sort_counts2; // ... and of its odd passes (zero between sorts)
    uint32_t* sort_offsets; // [tiles][512] output position of each tile's first element of each digit
    uint32_t* sort_dtot;    // [kSortMaxPasses][512] digit totals of each pass, zero between sorts
    uint32_t* tile_sums;    // [max(scan tiles, SMs)]: per-tile sums of the dedup's scan, per-block of the miss kernel
    uint32_t* seg_start;    // [max_batch + 1] run starts in sorted order (dedup)
    uint32_t* run_row;      // [max_batch] row of each run (dedup)
    uint32_t* run_p0;       // [max_batch] first lookup position of each run (dedup)
    uint4* short_runs;      // [max_batch] the apply's runs of 2 .. MLKV_SEQ_SEGMENT_MAX lookups
    uint2* single_runs;     // [max_batch] its runs of one lookup: (row, lookup position)
    uint4* small_runs;      // [max_batch] runs of 2 .. kSmallRun lookups: (row, p0, p1, p2)
    uint32_t* small_p3;     // [max_batch] their fourth position (or none)
    uint32_t* long_s;       // [max_long] long runs: first sorted position
    uint32_t* long_e;       // [max_long] one past the last
    uint32_t* long_row;     // [max_long]
    uint32_t* long_base;    // [max_long] first chunk item
    uint32_t* item_s;       // [max_items] first sorted position of each chunk
    uint32_t* item_e;       // [max_items] one past its last
    uint32_t* big_runs;     // [max_long] long runs with many chunks (combined by wide blocks)
    float* partial;         // [max_items][2][dpad] chunk sums: compensated (sum, compensation) pairs
    int64_t max_long;
    int64_t max_items;
    int64_t tile_sums_len;
    int64_t sort_counts_bytes;
};

// Tiered store (hbm_cache_rows > 0): see mlkv_tier.cu.
struct Tier {
    float* host_dev;        // host tier [capacity][stride]: pinned host memory mapped for the device
    size_t host_bytes;      // mapped bytes (whole chunks)
    size_t host_chunk;      // bytes per allocation handle
    unsigned long long* host_handles;  // one per chunk (CUmemGenericAllocationHandle)
    int64_t host_mapped;    // chunks mapped so far
    float* cache;           // HBM cache [C][stride]
    uint32_t* row_loc;      // [capacity] cache line, LOC_HOST | host slot, or LOC_CLAIMED
    uint32_t* line_row;     // [C]
    uint32_t* line_stamp;   // [C]
    unsigned long long* ctr;  // free_next, clock, rows fetched, rows written back
    uint2* fetch;           // [max_batch] (row, host slot) to fetch, main calls
    uint32_t* n_fetch;
    uint32_t* la_rows;      // [max_batch] row of each look-ahead key
    uint2* la_fetch;        // [max_batch]
    uint32_t* la_n_fetch;
    cudaStream_t la_stream;
    cudaEvent_t ev_main, ev_la;
    uint32_t epoch;         // epoch of the latest call (host side)
    int la_pending;         // a look-ahead was issued and not yet waited for
};

struct KernelTimer {
    int kernel_id = 0;
    int n_events = 0;
    static constexpr int kMax = 8192;
    cudaEvent_t* ev = nullptr;  // 2 * kMax events, created on first use
};

}  // namespace mlkv

struct mlkv_table {
    mlkv_config cfg;
    int device;
    int num_sms;
    mlkv::RowGeom geom;
    float* slots;                // slot array the row kernels use: the table, or the HBM cache
    mlkv::Slot* index;
    unsigned long long index_mask;
    int sort_bits;               // bits of the ids being sorted incl. the absent sentinel
    int bits_rows;               // ... for row ids
    int bits_lines;              // ... for cache line ids (tiered)
    int tiered;
    mlkv::Tier tier;
    mlkv::DevState* dstate;      // device
    uint32_t* status_host;       // mapped pinned word the kernels also write errors to
    uint32_t* status_dev_alias;  // its device alias
    mlkv::Scratch s;
    void* arena;                 // one allocation holding Scratch
    int64_t arena_bytes;
    // *_host staging, lazily allocated: [0] for every call of a bulk-synchronous
    // table; on a stale-synchronous one [1] for the applies, which run beside Gets
    int64_t* stage_keys[2];
    float* stage_vals[2];
    cudaStream_t last_stream;
    int parity;
    cudaStream_t last_apply_stream;
    int parity_apply;
    // Stale-synchronous mode (staleness_bound s >= 1): events order the Get's
    // stream and the apply's (see mlkv_get).
    int64_t stale;               // the bound kept: 0, 1..kMaxStaleness, or INT64_MAX (no bound)
    int64_t ring;                // events in ev_apply
    cudaEvent_t* ev_apply;       // [ring]: apply number j records ev_apply[j % ring]
    cudaEvent_t ev_other;        // after the last call other than an apply
    int other_recorded;
    // The apply's independent reduce kernels run on the call's stream and
    // these, forked after the run lists are made and joined before the long
    // runs' combine.
    cudaStream_t branch[2];
    cudaEvent_t ev_fork;
    cudaEvent_t ev_join[2];
    int64_t n_applies;
    int64_t launches;
    mlkv::KernelTimer timer;
    double timed_ms;
    int64_t timed_launches;
    char last_error[512];
};

namespace mlkv {

// Everything a kernel needs to record an error.
struct ErrSink {
    uint32_t* dev;             // DevState::status
    volatile uint32_t* host;   // mapped pinned mirror
    uint32_t* chk;             // DevState::chk (bounds-checked build), or null
};

__device__ __forceinline__ void record_error(const ErrSink& e, uint32_t code) {
    if (atomicCAS(e.dev, 0u, code) == 0u && e.host) *e.host = code;
}

// Called by every block of a call's last kernels (`total` blocks in all: one
// kernel, or the last kernel of each of the apply's streams) once it has read
// the call's counters for the last time: the last block to get here zeroes
// them, so the counters are zero when their next call starts, however that
// call was launched (a replayed graph passes through no host code).
__device__ __forceinline__ void release_counters(CallCounters* c, uint32_t total) {
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(&c->done, 1u) == total - 1) {
            uint32_t* w = reinterpret_cast<uint32_t*>(c);
            for (unsigned i = 0; i < sizeof(CallCounters) / 4; ++i) w[i] = 0u;
        }
    }
}

// Bounds-checked build (-DMLKV_CHECK=1): the reduce kernels test the indices
// they are about to use (rows, lookup positions, list entries); a failed test
// records the first failing site with its index and bound and
// MLKV_ERR_INVALID, and the access is skipped.  mlkv_sync reports the site.
// In the normal build every test is compiled out.
#ifndef MLKV_CHECK
#define MLKV_CHECK 0
#endif
__device__ __forceinline__ bool in_bounds(const ErrSink& e, uint32_t site, unsigned long long idx,
                                          unsigned long long bound) {
    if (!MLKV_CHECK || idx < bound) return true;
    if (e.chk && atomicCAS(e.chk, 0u, site) == 0u) {
        e.chk[1] = (uint32_t)idx;
        e.chk[2] = (uint32_t)bound;
    }
    record_error(e, MLKV_ERR_INVALID);
    return false;
}

// row_loc encoding of the tiered store
constexpr uint32_t LOC_HOST = 0x80000000u;     // | host slot: the row is in the host tier
constexpr uint32_t LOC_CLAIMED = 0xFFFFFFFFu;  // a fetch of the row is in progress

struct TierArgs {
    uint32_t* row_loc;
    uint32_t* line_row;
    uint32_t* line_stamp;
    float* cache;
    float* host;
    int stride;
    uint32_t C;
    unsigned long long* free_next;
    unsigned long long* clock;
    unsigned long long* totals;
    uint32_t epoch;
    uint32_t keep_from;   // lines stamped >= keep_from are not taken
    uint32_t strict;      // 1: no fetch; hits must be stamped >= keep_from
    ErrSink err;
};

// MurmurHash3 fmix64 finaliser (Appleby): spreads structured keys such as
// table_id * 2^32 + row over the index.
__device__ __forceinline__ unsigned long long hash_key(unsigned long long k) {
    k ^= k >> 33;
    k *= 0xff51afd7ed558ccdull;
    k ^= k >> 33;
    k *= 0xc4ceb9fe1a85ec53ull;
    k ^= k >> 33;
    return k;
}

// SplitMix64 output function (Steele, Lea & Flood 2014) and the counter-based
// row initialisation stated in mlkv_gpu.h.
__device__ __forceinline__ unsigned long long splitmix64(unsigned long long z) {
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ float init_element(unsigned long long seed, unsigned long long key,
                                              uint32_t j, float lo, float span) {
    unsigned long long x = splitmix64(seed ^ splitmix64(key ^ ((unsigned long long)j * 0x9E3779B97F4A7C15ull)));
    float u = __fmul_rn((float)(uint32_t)(x >> 40), 5.9604644775390625e-8f);  // exact: 24-bit int * 2^-24
    return __fadd_rn(lo, __fmul_rn(u, span));
}

// One Adagrad element, each operation rounded on its own (no contraction):
//   G' = G + g*g ; w' = w - (lr*g) / (sqrt(G') + eps)
__device__ __forceinline__ void adagrad_element(float& w, float& G, float g, float lr, float eps) {
    float Gn = __fadd_rn(G, __fmul_rn(g, g));
    float den = __fadd_rn(__fsqrt_rn(Gn), eps);
    float u = __fdiv_rn(__fmul_rn(lr, g), den);
    G = Gn;
    w = __fsub_rn(w, u);
}

// Compensated addition (TwoSum of Knuth and Moller): s <- fl(s + x) and the
// rounding error of that sum, which is exact, added to the running
// compensation c.  s + c then carries the sum to about twice fp32's precision.
// Each operation is rounded on its own (the kernels are built without fused
// multiply-adds or any other contraction).
__device__ __forceinline__ void comp_add(float& s, float& c, float x) {
    const float t = __fadd_rn(s, x);
    const float bp = __fsub_rn(t, s);
    const float e = __fadd_rn(__fsub_rn(s, __fsub_rn(t, bp)), __fsub_rn(x, bp));
    s = t;
    c = __fadd_rn(c, e);
}

// Packed fp32 pairs (sm_100 and later: add/sub .f32x2).  Each half is an
// IEEE round-to-nearest operation, so a packed add gives the same bits as two
// scalar __fadd_rn, with half the instructions.
__device__ __forceinline__ float2 add_x2(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 pa, pb, pr;\n\t"
        "mov.b64 pa, {%2, %3};\n\t"
        "mov.b64 pb, {%4, %5};\n\t"
        "add.rn.f32x2 pr, pa, pb;\n\t"
        "mov.b64 {%0, %1}, pr;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 sub_x2(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 pa, pb, pr;\n\t"
        "mov.b64 pa, {%2, %3};\n\t"
        "mov.b64 pb, {%4, %5};\n\t"
        "sub.rn.f32x2 pr, pa, pb;\n\t"
        "mov.b64 {%0, %1}, pr;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

// comp_add on a pair, with packed operations.
__device__ __forceinline__ void comp_add_x2(float2& s, float2& c, float2 x) {
    const float2 t = add_x2(s, x);
    const float2 bp = sub_x2(t, s);
    const float2 e = add_x2(sub_x2(s, sub_x2(t, bp)), sub_x2(x, bp));
    s = t;
    c = add_x2(c, e);
}

template <int V> struct Vec;
template <> struct Vec<4> {
    using T = float4;
    static __device__ __forceinline__ T zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }
    static __device__ __forceinline__ T nan() {
        float q = __int_as_float(0x7fc00000);
        return make_float4(q, q, q, q);
    }
    static __device__ __forceinline__ void add(T& a, const T& b) {
        const float2 lo = add_x2(make_float2(a.x, a.y), make_float2(b.x, b.y));
        const float2 hi = add_x2(make_float2(a.z, a.w), make_float2(b.z, b.w));
        a = make_float4(lo.x, lo.y, hi.x, hi.y);
    }
    static __device__ __forceinline__ void cadd(T& s, T& c, const T& x) {
        float2 s0 = make_float2(s.x, s.y), s1 = make_float2(s.z, s.w);
        float2 c0 = make_float2(c.x, c.y), c1 = make_float2(c.z, c.w);
        comp_add_x2(s0, c0, make_float2(x.x, x.y));
        comp_add_x2(s1, c1, make_float2(x.z, x.w));
        s = make_float4(s0.x, s0.y, s1.x, s1.y);
        c = make_float4(c0.x, c0.y, c1.x, c1.y);
    }
    static __device__ __forceinline__ void adagrad(T& w, T& G, const T& g, float lr, float eps) {
        adagrad_element(w.x, G.x, g.x, lr, eps); adagrad_element(w.y, G.y, g.y, lr, eps);
        adagrad_element(w.z, G.z, g.z, lr, eps); adagrad_element(w.w, G.w, g.w, lr, eps);
    }
    static __device__ __forceinline__ T splat(float v) { return make_float4(v, v, v, v); }
    static __device__ __forceinline__ T from(const float* e) { return make_float4(e[0], e[1], e[2], e[3]); }
    static __device__ __forceinline__ T shfl_down(const T& v, int delta) {
        return make_float4(__shfl_down_sync(0xffffffffu, v.x, delta), __shfl_down_sync(0xffffffffu, v.y, delta),
                           __shfl_down_sync(0xffffffffu, v.z, delta), __shfl_down_sync(0xffffffffu, v.w, delta));
    }
};
template <> struct Vec<1> {
    using T = float;
    static __device__ __forceinline__ T zero() { return 0.f; }
    static __device__ __forceinline__ T nan() { return __int_as_float(0x7fc00000); }
    static __device__ __forceinline__ void add(T& a, const T& b) { a = __fadd_rn(a, b); }
    static __device__ __forceinline__ void cadd(T& s, T& c, const T& x) { comp_add(s, c, x); }
    static __device__ __forceinline__ void adagrad(T& w, T& G, const T& g, float lr, float eps) {
        adagrad_element(w, G, g, lr, eps);
    }
    static __device__ __forceinline__ T splat(float v) { return v; }
    static __device__ __forceinline__ T from(const float* e) { return e[0]; }
    static __device__ __forceinline__ T shfl_down(const T& v, int delta) {
        return __shfl_down_sync(0xffffffffu, v, delta);
    }
};

// Programmatic dependent launch.  MLKV_LAUNCH lets a kernel start while the
// kernel before it on the stream drains, which hides the launch and ramp-up
// of the ~25 kernels of a step.  Every kernel begins with pdl_enter():
//   - griddepcontrol.wait returns once the grid this launch depends on has
//     completed and its writes are visible (at once when the launch has no
//     such dependency).  Every kernel waits, on every path, before touching
//     memory, so the completion of a kernel implies the completion of all the
//     kernels before it;
//   - griddepcontrol.launch_dependents lets the next kernel's blocks be
//     scheduled (once every block of this grid has issued it or exited);
//     they in turn wait for this grid.  Issued after the wait, it keeps at
//     most one grid waiting ahead of the running one.
#ifndef MLKV_PDL_TRIGGER_FIRST
#define MLKV_PDL_TRIGGER_FIRST 0
#endif
__device__ __forceinline__ void pdl_enter() {
    if (MLKV_PDL_TRIGGER_FIRST) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (!MLKV_PDL_TRIGGER_FIRST) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ uint32_t lanemask_lt() {
    uint32_t m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// Parameters shared by the index kernels.
struct IndexArgs {
    Slot* index;
    unsigned long long mask;
    uint32_t identity_hash;
    ErrSink err;
};

// The (key, row) of every lookup position of the last Get.  A key's row never
// changes once handed out, so a later probe whose key at position p equals
// memo key[p] may take memo row[p] (when it is a row: pending and absent
// lookups are probed again) instead of walking the index; the gradient apply
// that follows a Get on the same keys then costs no index accesses.
struct Memo {
    int64_t* key;
    uint32_t* row;
};
enum class MemoUse { None, Read, Save };

// The first sort pass's digit counts, made by the gradient apply: its probe
// writes every tile's column of counts[digit][tile] for the lookups whose row
// it found (and adds them to the pass's totals dtot); the miss kernel adds the
// lookups it gave rows.  The sort's first pass then needs no histogram kernel.
struct FirstCounts {
    uint32_t* counts;
    uint32_t* dtot;
    uint32_t ntiles;
    int radix;       // digits of the first pass
    uint32_t sent;   // sort key of a lookup without a row
    int tile_shift;  // log2 of the sort's tile (sort_tile_shift)
};

// ---------------------------------------------------------------------------
// Host-side launchers (each returns cudaGetLastError() of its launches).
enum class MissMode : int { Init = 0, Put = 1, Get = 2 };

// mlkv_index.cu
cudaError_t launch_probe(mlkv_table* t, const int64_t* keys, int64_t n, bool insert, MemoUse memo,
                         bool want_slot, bool report_absent, cudaStream_t st, CallCounters* cur,
                         CallCounters* nxt, uint32_t* rows_out = nullptr, const FirstCounts* fc = nullptr);
cudaError_t launch_get(mlkv_table* t, const int64_t* keys, int64_t n, float* out, cudaStream_t st,
                       CallCounters* cur, CallCounters* nxt);
// release: the miss kernel is the last of the call to read its counters, and
// zeroes them when done (release_counters).  fc: the first sort pass's counts
// the apply's probe made, to which the lookups given rows here are added.
cudaError_t launch_resolve_misses(mlkv_table* t, const int64_t* keys, int64_t n, MissMode mode,
                                  float* out, cudaStream_t st, CallCounters* cur, bool release,
                                  const FirstCounts* fc = nullptr);
cudaError_t launch_put_scatter(mlkv_table* t, const float* vals, const float* state, int64_t n, cudaStream_t st);
cudaError_t launch_dump_keys(mlkv_table* t, int64_t* out, int64_t n_rows, cudaStream_t st);
// Every index slot of a key without a row goes back to idle (aux) after a call cut short.
cudaError_t launch_reset_pending(mlkv_table* t, cudaStream_t st);
cudaError_t launch_find(mlkv_table* t, const int64_t* keys, int64_t n, int64_t* rows,
                        cudaStream_t st, CallCounters* nxt);
cudaError_t launch_export(mlkv_table* t, const int64_t* keys, int64_t n, float* rows,
                          float* state, cudaStream_t st, CallCounters* nxt);

// mlkv_sort.cu
// The first pass's counts for the probe to make (t->sort_bits rows, n lookups).
FirstCounts first_counts(mlkv_table* t, int64_t n);
// first_counted: the first pass's counts were made by the apply's probe and
// miss kernel (FirstCounts).
cudaError_t launch_sort_rows(mlkv_table* t, int64_t n, cudaStream_t st, const uint32_t** srow,
                             const uint32_t** spos, bool first_counted = false);
cudaError_t launch_segments(mlkv_table* t, const uint32_t* srow, const uint32_t* spos, int64_t n,
                            cudaStream_t st, CallCounters* cur);
cudaError_t launch_dedup_out(mlkv_table* t, const int64_t* keys, const uint32_t* spos, int64_t n,
                             int64_t* uniq, int32_t* counts, int64_t* num, cudaStream_t st,
                             CallCounters* cur);

// mlkv_tier.cu
TierArgs tier_args(mlkv_table* t, uint32_t epoch, uint32_t keep_from, int strict);
cudaError_t launch_tier_resolve(mlkv_table* t, const TierArgs& ta, uint32_t* row_of_pos, int64_t n,
                                uint2* fetch, uint32_t* n_fetch, bool remap, cudaStream_t st);
cudaError_t launch_tier_init(mlkv_table* t, cudaStream_t st);
cudaError_t launch_gather_lines(mlkv_table* t, const uint32_t* rows, int64_t n, float* out, cudaStream_t st);

// mlkv_apply.cu
int64_t long_runs_bound(int64_t max_batch);   // runs longer than MLKV_SEQ_SEGMENT_MAX, worst case
int64_t long_items_bound(int64_t max_batch);  // chunks of those runs, worst case
cudaError_t launch_reduce_apply(mlkv_table* t, const float* grads, const uint32_t* srow,
                                const uint32_t* spos, int64_t n, uint32_t sent, cudaStream_t st,
                                CallCounters* cur);

// mlkv_table.cu: launch bookkeeping and optional per-kernel timing; the host
// side of mlkv_debug_fail's wait injection (true once, for the armed launch).
bool take_injected_wait();
void timer_before(mlkv_table* t, int kernel_id, cudaStream_t st);
void timer_after(mlkv_table* t, int kernel_id, cudaStream_t st);
int persistent_blocks(mlkv_table* t, const void* kernel, int threads);

}  // namespace mlkv

// Programmatic dependent launch of every kernel (off with -DMLKV_PDL=0: plain
// stream order; the kernels' pdl_wait() then returns at once).
#ifndef MLKV_PDL
#define MLKV_PDL 1
#endif

namespace mlkv {
template <typename... Params, typename... Args>
inline void launch_kernel(bool pdl, void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t st, Args&&... args) {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = MLKV_PDL && pdl ? 1 : 0;
    cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);  // an error stays in cudaGetLastError()
}
}  // namespace mlkv

// Launch helper: counts the launch and records timing events when asked.
#define MLKV_LAUNCH_PDL(pdl, t, kid, kernel, grid, block, smem, stream, ...)                      \
    do {                                                                                          \
        mlkv::timer_before((t), (kid), (stream));                                                 \
        mlkv::launch_kernel((pdl), kernel, dim3(grid), dim3(block), (smem), (stream), __VA_ARGS__); \
        mlkv::timer_after((t), (kid), (stream));                                                  \
        (t)->launches++;                                                                          \
    } while (0)
#define MLKV_LAUNCH(...) MLKV_LAUNCH_PDL(true, __VA_ARGS__)
// The persistent grids (one wave, each block a fixed share of the work) may
// start as the kernel before them drains too; -DMLKV_PDL_PERSISTENT=0 makes
// them wait for it in full (every SM free when their blocks are placed).
#ifndef MLKV_PDL_PERSISTENT
#define MLKV_PDL_PERSISTENT 1
#endif
#define MLKV_LAUNCH_PERSISTENT(...) MLKV_LAUNCH_PDL(MLKV_PDL_PERSISTENT != 0, __VA_ARGS__)
