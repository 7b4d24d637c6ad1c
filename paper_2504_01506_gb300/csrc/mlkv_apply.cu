// Segmented gradient reduction fused with the sparse Adagrad read-modify-write.
//
// After the sort, the lookups of one row form a run (segment) of consecutive
// sorted positions, in occurrence order (the sort is stable); the segment
// kernels list the run starts.  For every run the sum g of its gradient rows
// is formed and one Adagrad step is applied to the row and its state, each
// read once and written once:
//     G += g*g ;  w -= lr * g / (sqrt(G) + eps)          (element-wise)
// This is the per-key Rmw of MLKV Section 3.2 step 8, with the gradient of the
// embedding map E (Section 2.1) summed over the key's lookups.
//
//  k_short        one lane group per run; a run of <= MLKV_SEQ_SEGMENT_MAX
//                 lookups is summed in occurrence order and its row updated.
//                 Its positions are loaded lane-parallel and the row and state
//                 loads are issued next to the gradient loads, so a run costs
//                 about three dependent memory round trips.  Longer runs are
//                 listed for the next two kernels.
//  k_long_sum     one lane group per chunk of kChunk lookups of a long run
//                 (Zipf-hot keys reach 10^4-10^5 lookups): chunk sum to scratch.
//  k_long_combine one block per long run: the chunk sums are split over the
//                 block's lane groups in a fixed way, added in that order, and
//                 the row updated.
// All three keep registers low so that many warps are resident: the access
// pattern is random 512-byte rows, which HBM serves near its copy bandwidth
// only with many requests in flight.  Results do not depend on scheduling.
#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

constexpr int kChunk = 64;

// Tuning (set at build time): gradient rows in flight per lane group, and the
// minimum resident blocks per SM the register allocation must allow.
#ifndef MLKV_REDUCE_ROWS_IN_FLIGHT
#define MLKV_REDUCE_ROWS_IN_FLIGHT 4
#endif
#ifndef MLKV_REDUCE_MIN_BLOCKS
#define MLKV_REDUCE_MIN_BLOCKS 5
#endif
#ifndef MLKV_SHORT_MIN_BLOCKS
#define MLKV_SHORT_MIN_BLOCKS 5
#endif
#ifndef MLKV_LONG_ROWS_IN_FLIGHT
#define MLKV_LONG_ROWS_IN_FLIGHT 4
#endif
#ifndef MLKV_LONG_MIN_BLOCKS
#define MLKV_LONG_MIN_BLOCKS 5
#endif

struct RowArgs {
    float* slots;
    int stride;
    int dpad;
    int NV;
    int G;
    int d;
};

struct RunArgs {
    const float* grads;
    const uint32_t* srow;
    const uint32_t* spos;
    const uint32_t* seg_start;
    const uint32_t* run_row;   // row of each run
    const uint32_t* run_p0;    // first lookup position of each run
    CallCounters* cur;
    uint32_t* long_s;      // [max_long] first sorted position
    uint32_t* long_e;      // [max_long] one past the last
    uint32_t* long_row;    // [max_long]
    uint32_t* long_base;   // [max_long] first chunk item
    uint32_t* item_s;      // [max_items] first sorted position of each chunk
    uint32_t* item_e;      // [max_items] one past its last
    float* partial;        // [max_items][dpad]
    uint32_t max_long;
    uint32_t max_items;
    ErrSink err;
    float lr, eps;
};

__device__ __forceinline__ unsigned group_mask(int G, int gid) {
    return G == 32 ? 0xffffffffu : (((1u << G) - 1u) << (gid * G));
}

// acc += the gradient rows of sorted positions s .. s+len-1, in that order.
// The group loads up to G positions at a time (one per lane) and hands them
// round with group shuffles.
template <int V, int KV, int ROWS = MLKV_REDUCE_ROWS_IN_FLIGHT>
__device__ __forceinline__ void sum_rows(typename Vec<V>::T (&acc)[KV], const float* __restrict__ grads,
                                         const uint32_t* __restrict__ spos, uint32_t s, uint32_t len, int d,
                                         int NV, int G, int glane, unsigned gmask) {
    using VT = typename Vec<V>::T;
    constexpr int UNR = KV >= ROWS ? 1 : ROWS / KV;
    for (uint32_t base = 0; base < len; base += G) {
        const uint32_t cnt = min((uint32_t)G, len - base);
        const uint32_t pl = (uint32_t)glane < cnt ? __ldg(spos + s + base + glane) : 0u;
        for (uint32_t x = 0; x < cnt; x += UNR) {
            VT g[UNR][KV];
#pragma unroll
            for (int u = 0; u < UNR; ++u) {
                const uint32_t p = __shfl_sync(gmask, pl, (int)(x + u) & (G - 1), G);
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
                    if (x + u < cnt && glane + G * k < NV) Vec<V>::add(acc[k], g[u][k]);
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

// One lane group per run.  Its start, end, row and first lookup position are
// independent loads (the segment kernel wrote them side by side); then the
// row, the state and the first gradient row are loaded together, so a run
// of one lookup (most of them) costs two dependent round trips.
template <int V, int KV>
__global__ void __launch_bounds__(256, MLKV_SHORT_MIN_BLOCKS) k_short(RowArgs ra, RunArgs a) {
    using VT = typename Vec<V>::T;
    const uint32_t U = a.cur->n_unique, nv = a.cur->n_valid;
    const int lane = threadIdx.x & 31, G = ra.G, glane = lane & (G - 1), gid = lane / G;
    const unsigned gmask = group_mask(G, gid);
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) / G;
    const uint32_t ngroups = (gridDim.x * blockDim.x) / G;
    for (uint32_t u = group; u < U; u += ngroups) {  // uniform within the group
        const uint32_t s = __ldg(a.seg_start + u);
        const uint32_t e = u + 1 < U ? __ldg(a.seg_start + u + 1) : nv;
        const uint32_t row = __ldg(a.run_row + u);
        const uint32_t p0 = __ldg(a.run_p0 + u);
        const uint32_t len = e - s;
        if (len > MLKV_SEQ_SEGMENT_MAX) {
            if (glane == 0) {
                const uint32_t nit = (len + kChunk - 1) / kChunk;
                const uint32_t h = atomicAdd(&a.cur->n_long, 1u);
                const uint32_t ib = atomicAdd(&a.cur->n_items, nit);
                if (h < a.max_long && ib + nit <= a.max_items) {
                    a.long_s[h] = s;
                    a.long_e[h] = e;
                    a.long_row[h] = row;
                    a.long_base[h] = ib;
                    for (uint32_t k = 0; k < nit; ++k) {
                        a.item_s[ib + k] = s + k * kChunk;
                        a.item_e[ib + k] = min(s + (k + 1) * kChunk, e);
                    }
                } else {
                    record_error(a.err, MLKV_ERR_FULL);
                }
            }
            continue;
        }
        VT w[KV], Gs[KV], acc[KV];
        load_row_state<V, KV>(ra, row, w, Gs, glane);
        const VT* g0 = reinterpret_cast<const VT*>(a.grads + (size_t)p0 * ra.d);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            acc[k] = Vec<V>::zero();
            const int j = glane + G * k;
            if (j < ra.NV) Vec<V>::add(acc[k], __ldcs(g0 + j));  // 0 + g: first term, in order
        }
        if (len > 1) sum_rows<V, KV>(acc, a.grads, a.spos, s + 1, len - 1, ra.d, ra.NV, G, glane, gmask);
        adagrad_store<V, KV>(ra, row, w, Gs, acc, glane, a.lr, a.eps);
    }
}

template <int V, int KV>
__global__ void __launch_bounds__(256, MLKV_LONG_MIN_BLOCKS) k_long_sum(RowArgs ra, RunArgs a) {
    using VT = typename Vec<V>::T;
    const uint32_t NI = min(a.cur->n_items, a.max_items);
    const int lane = threadIdx.x & 31, G = ra.G, glane = lane & (G - 1), gid = lane / G;
    const unsigned gmask = group_mask(G, gid);
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) / G;
    const uint32_t ngroups = (gridDim.x * blockDim.x) / G;
    for (uint32_t it = group; it < NI; it += ngroups) {
        const uint32_t s = __ldg(a.item_s + it), e = __ldg(a.item_e + it);
        VT acc[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) acc[k] = Vec<V>::zero();
        sum_rows<V, KV, MLKV_LONG_ROWS_IN_FLIGHT>(acc, a.grads, a.spos, s, e > s ? e - s : 0u, ra.d, ra.NV, G,
                                                  glane, gmask);
        VT* part = reinterpret_cast<VT*>(a.partial + (size_t)it * ra.dpad);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < ra.NV) __stcg(part + j, acc[k]);
        }
    }
}

template <int V, int KV>
__global__ void __launch_bounds__(256) k_long_combine(RowArgs ra, RunArgs a, DevState* ds) {
    using VT = typename Vec<V>::T;
    extern __shared__ float sh[];  // [groups][dpad]
    const uint32_t nl = min(a.cur->n_long, a.max_long);
    if (blockIdx.x == 0 && threadIdx.x == 0) ds->last_unique = a.cur->n_unique;
    const int G = ra.G, glane = threadIdx.x & (G - 1);
    const int group = threadIdx.x / G;
    const int ngroups = blockDim.x / G;
    for (uint32_t h = blockIdx.x; h < nl; h += gridDim.x) {  // block-uniform
        const uint32_t base = a.long_base[h];
        const uint32_t m = (a.long_e[h] - a.long_s[h] + kChunk - 1) / kChunk;
        const uint32_t per = (m + ngroups - 1) / ngroups;
        const uint32_t k0 = min(m, group * per), k1 = min(m, k0 + per);
        VT acc[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) acc[k] = Vec<V>::zero();
        constexpr int UNR = KV >= 8 ? 1 : 8 / KV;
        for (uint32_t x = k0; x < k1; x += UNR) {
            VT g[UNR][KV];
#pragma unroll
            for (int u = 0; u < UNR; ++u) {
                const VT* src = reinterpret_cast<const VT*>(a.partial + (size_t)(base + x + u) * ra.dpad);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (x + u < k1 && j < ra.NV) g[u][k] = __ldcg(src + j);
                }
            }
#pragma unroll
            for (int u = 0; u < UNR; ++u)
#pragma unroll
                for (int k = 0; k < KV; ++k)
                    if (x + u < k1 && glane + G * k < ra.NV) Vec<V>::add(acc[k], g[u][k]);
        }
        VT* mine = reinterpret_cast<VT*>(sh + (size_t)group * ra.dpad);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < ra.NV) mine[j] = acc[k];
        }
        __syncthreads();
        if (group == 0) {
#pragma unroll
            for (int k = 0; k < KV; ++k) acc[k] = Vec<V>::zero();
            for (int gi = 0; gi < ngroups; ++gi) {
                const VT* src = reinterpret_cast<const VT*>(sh + (size_t)gi * ra.dpad);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (j < ra.NV) Vec<V>::add(acc[k], src[j]);
                }
            }
            VT w[KV], Gs[KV];
            const uint32_t row = a.long_row[h];
            load_row_state<V, KV>(ra, row, w, Gs, glane);
            adagrad_store<V, KV>(ra, row, w, Gs, acc, glane, a.lr, a.eps);
        }
        __syncthreads();
    }
}

template <int V, int KV>
cudaError_t run_reduce(mlkv_table* t, const float* grads, const uint32_t* srow, const uint32_t* spos,
                       int64_t n, cudaStream_t st, CallCounters* cur) {
    (void)n;
    RowArgs ra{t->slots, t->geom.stride, t->geom.dpad, t->geom.NV, t->geom.G, t->geom.d};
    RunArgs a{grads, srow, spos, t->s.seg_start, t->s.run_row, t->s.run_p0, cur, t->s.long_s, t->s.long_e,
              t->s.long_row, t->s.long_base, t->s.item_s, t->s.item_e, t->s.partial, (uint32_t)t->s.max_long,
              (uint32_t)t->s.max_items, ErrSink{&t->dstate->status, t->status_dev_alias}, t->cfg.lr, t->cfg.eps};
    const int gs = persistent_blocks(t, (const void*)k_short<V, KV>, 256);
    MLKV_LAUNCH(t, MLKV_K_REDUCE_SHORT, (k_short<V, KV>), gs, 256, 0, st, ra, a);
    const int gl = persistent_blocks(t, (const void*)k_long_sum<V, KV>, 256);
    MLKV_LAUNCH(t, MLKV_K_REDUCE_LONG, (k_long_sum<V, KV>), gl, 256, 0, st, ra, a);
    // small blocks, many of them: every long run can be combined at once
    const int cthreads = 64;
    const size_t smem = (size_t)(cthreads / t->geom.G) * t->geom.dpad * sizeof(float);
    MLKV_LAUNCH(t, MLKV_K_LONG_COMBINE, (k_long_combine<V, KV>), t->num_sms * 16, cthreads, smem, st, ra, a,
                t->dstate);
    return cudaGetLastError();
}

}  // namespace

int64_t long_runs_bound(int64_t max_batch) { return max_batch / (MLKV_SEQ_SEGMENT_MAX + 1) + 1; }

int64_t long_items_bound(int64_t max_batch) { return max_batch / kChunk + long_runs_bound(max_batch) + 1; }

cudaError_t launch_reduce_apply(mlkv_table* t, const float* grads, const uint32_t* srow,
                                const uint32_t* spos, int64_t n, cudaStream_t st, CallCounters* cur) {
    const RowGeom& g = t->geom;
    if (g.V == 4) {
        switch (g.KV) {
            case 1: return run_reduce<4, 1>(t, grads, srow, spos, n, st, cur);
            case 2: return run_reduce<4, 2>(t, grads, srow, spos, n, st, cur);
            case 4: return run_reduce<4, 4>(t, grads, srow, spos, n, st, cur);
            default: return run_reduce<4, 8>(t, grads, srow, spos, n, st, cur);
        }
    }
    switch (g.KV) {
        case 1: return run_reduce<1, 1>(t, grads, srow, spos, n, st, cur);
        case 2: return run_reduce<1, 2>(t, grads, srow, spos, n, st, cur);
        case 4: return run_reduce<1, 4>(t, grads, srow, spos, n, st, cur);
        default: return run_reduce<1, 8>(t, grads, srow, spos, n, st, cur);
    }
}

}  // namespace mlkv
