// Segmented gradient reduction fused with the sparse Adagrad read-modify-write.
//
// After the sort, the lookups of one row form a segment of consecutive sorted
// positions, in occurrence order (the sort is stable).  For every segment the
// sum g of its gradient rows is formed and one Adagrad step is applied to the
// row and its state, each read once and written once:
//     G += g*g ;  w -= lr * g / (sqrt(G) + eps)          (element-wise)
// This is the per-key Rmw of MLKV Section 3.2 step 8, with the gradient of the
// embedding map E (Section 2.1) summed over the key's lookups.
//
// Short segments (<= MLKV_SEQ_SEGMENT_MAX lookups, nearly all of them): one
// lane group sums the segment in occurrence order and applies the step.
// Long segments (Zipf-hot keys, up to ~10^5 lookups): split into chunks of
// kChunk lookups; each chunk's sum goes to scratch and the last chunk to
// finish adds the chunk sums in chunk order and applies the step.  The result
// does not depend on scheduling, so runs are bit-reproducible.
#include "mlkv_internal.cuh"

namespace mlkv {

namespace {

constexpr int kChunk = 64;

struct RowArgs {
    float* slots;
    int stride;
    int dpad;
    int NV;
    int G;
    int d;
};

// acc += sum of grads[spos[p]] for p in [s, e), in order.
template <int V, int KV>
__device__ __forceinline__ void sum_segment(typename Vec<V>::T (&acc)[KV], const float* __restrict__ grads,
                                            const uint32_t* __restrict__ spos, uint32_t s, uint32_t e,
                                            int d, int NV, int G, int glane) {
    using VT = typename Vec<V>::T;
    constexpr int UNR = KV >= 8 ? 1 : 8 / KV;
    uint32_t p = s;
    for (; p + UNR <= e; p += UNR) {
        VT g[UNR][KV];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            const VT* src = reinterpret_cast<const VT*>(grads + (size_t)__ldg(spos + p + u) * d);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int j = glane + G * k;
                if (j < NV) g[u][k] = __ldcs(src + j);
            }
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u)
#pragma unroll
            for (int k = 0; k < KV; ++k)
                if (glane + G * k < NV) Vec<V>::add(acc[k], g[u][k]);
    }
    for (; p < e; ++p) {
        const VT* src = reinterpret_cast<const VT*>(grads + (size_t)__ldg(spos + p) * d);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < NV) Vec<V>::add(acc[k], __ldcs(src + j));
        }
    }
}

template <int V, int KV>
__device__ __forceinline__ void adagrad_row(const RowArgs& ra, uint32_t row, const typename Vec<V>::T (&g)[KV],
                                            int glane, float lr, float eps) {
    using VT = typename Vec<V>::T;
    float* slot = ra.slots + (size_t)row * ra.stride;
    VT* wv = reinterpret_cast<VT*>(slot);
    VT* gv = reinterpret_cast<VT*>(slot + ra.dpad);
#pragma unroll
    for (int k = 0; k < KV; ++k) {
        const int j = glane + ra.G * k;
        if (j < ra.NV) {
            VT w = wv[j], G = gv[j];
            Vec<V>::adagrad(w, G, g[k], lr, eps);
            wv[j] = w;
            gv[j] = G;
        }
    }
}

__device__ __forceinline__ unsigned group_mask(int G, int gid) {
    return G == 32 ? 0xffffffffu : (((1u << G) - 1u) << (gid * G));
}

template <int V, int KV>
__global__ void __launch_bounds__(256) k_reduce_short(RowArgs ra, const float* __restrict__ grads,
                                                      const uint32_t* __restrict__ srow,
                                                      const uint32_t* __restrict__ spos,
                                                      const uint32_t* __restrict__ seg_start,
                                                      CallCounters* cur, uint32_t* __restrict__ long_seg,
                                                      uint32_t* __restrict__ long_base,
                                                      uint32_t* __restrict__ long_cnt,
                                                      uint32_t* __restrict__ item_seg, uint32_t max_long,
                                                      uint32_t max_items, float lr, float eps, ErrSink err) {
    using VT = typename Vec<V>::T;
    const uint32_t U = cur->n_unique, nv = cur->n_valid;
    const int lane = threadIdx.x & 31, G = ra.G, R = 32 / G, glane = lane & (G - 1), gid = lane / G;
    const unsigned gmask = group_mask(G, gid);
    const uint32_t warp = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const uint32_t nwarps = gridDim.x * (blockDim.x >> 5);
    for (uint32_t b = warp * R; b < U; b += nwarps * R) {
        const uint32_t u = b + gid;
        if (u >= U) continue;
        const uint32_t s = __ldg(seg_start + u);
        const uint32_t e = u + 1 < U ? __ldg(seg_start + u + 1) : nv;
        const uint32_t len = e - s;
        if (len > MLKV_SEQ_SEGMENT_MAX) {
            const uint32_t nit = (len + kChunk - 1) / kChunk;
            uint32_t h = 0, ib = 0;
            if (glane == 0) {
                h = atomicAdd(&cur->n_long, 1u);
                ib = atomicAdd(&cur->n_items, nit);
            }
            h = __shfl_sync(gmask, h, 0, G);
            ib = __shfl_sync(gmask, ib, 0, G);
            if (h >= max_long || ib + nit > max_items) {
                if (glane == 0) record_error(err, MLKV_ERR_FULL);
                continue;
            }
            if (glane == 0) {
                long_seg[h] = u;
                long_base[h] = ib;
                long_cnt[h] = 0u;
            }
            for (uint32_t k = glane; k < nit; k += G) item_seg[ib + k] = h;
            continue;
        }
        VT acc[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) acc[k] = Vec<V>::zero();
        sum_segment<V, KV>(acc, grads, spos, s, e, ra.d, ra.NV, G, glane);
        adagrad_row<V, KV>(ra, __ldg(srow + s), acc, glane, lr, eps);
    }
}

template <int V, int KV>
__global__ void __launch_bounds__(256) k_reduce_long(RowArgs ra, const float* __restrict__ grads,
                                                     const uint32_t* __restrict__ srow,
                                                     const uint32_t* __restrict__ spos,
                                                     const uint32_t* __restrict__ seg_start,
                                                     const CallCounters* cur, const uint32_t* __restrict__ long_seg,
                                                     const uint32_t* __restrict__ long_base,
                                                     uint32_t* __restrict__ long_cnt,
                                                     const uint32_t* __restrict__ item_seg,
                                                     float* __restrict__ partial, float lr, float eps) {
    using VT = typename Vec<V>::T;
    const uint32_t NI = cur->n_items, U = cur->n_unique, nv = cur->n_valid;
    const int lane = threadIdx.x & 31, G = ra.G, R = 32 / G, glane = lane & (G - 1), gid = lane / G;
    const unsigned gmask = group_mask(G, gid);
    const uint32_t warp = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const uint32_t nwarps = gridDim.x * (blockDim.x >> 5);
    for (uint32_t b = warp * R; b < NI; b += nwarps * R) {
        const uint32_t it = b + gid;
        if (it >= NI) continue;
        const uint32_t h = item_seg[it];
        const uint32_t u = long_seg[h], ib = long_base[h];
        const uint32_t s0 = __ldg(seg_start + u);
        const uint32_t e0 = u + 1 < U ? __ldg(seg_start + u + 1) : nv;
        const uint32_t nit = (e0 - s0 + kChunk - 1) / kChunk;
        const uint32_t s = s0 + (it - ib) * kChunk;
        const uint32_t e = min(s + kChunk, e0);
        VT acc[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) acc[k] = Vec<V>::zero();
        sum_segment<V, KV>(acc, grads, spos, s, e, ra.d, ra.NV, G, glane);
        VT* part = reinterpret_cast<VT*>(partial + (size_t)it * ra.dpad);
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int j = glane + G * k;
            if (j < ra.NV) __stcg(part + j, acc[k]);
        }
        __threadfence();
        __syncwarp(gmask);
        uint32_t done = 0;
        if (glane == 0) done = atomicAdd(&long_cnt[h], 1u);
        done = __shfl_sync(gmask, done, 0, G);
        if (done != nit - 1) continue;
        // last chunk of this segment: add the chunk sums in chunk order
        __threadfence();
#pragma unroll
        for (int k = 0; k < KV; ++k) acc[k] = Vec<V>::zero();
        constexpr int UNR = KV >= 8 ? 1 : 8 / KV;
        uint32_t m = 0;
        for (; m + UNR <= nit; m += UNR) {
            VT g[UNR][KV];
#pragma unroll
            for (int q = 0; q < UNR; ++q) {
                const VT* src = reinterpret_cast<const VT*>(partial + (size_t)(ib + m + q) * ra.dpad);
#pragma unroll
                for (int k = 0; k < KV; ++k) {
                    const int j = glane + G * k;
                    if (j < ra.NV) g[q][k] = __ldcg(src + j);
                }
            }
#pragma unroll
            for (int q = 0; q < UNR; ++q)
#pragma unroll
                for (int k = 0; k < KV; ++k)
                    if (glane + G * k < ra.NV) Vec<V>::add(acc[k], g[q][k]);
        }
        for (; m < nit; ++m) {
            const VT* src = reinterpret_cast<const VT*>(partial + (size_t)(ib + m) * ra.dpad);
#pragma unroll
            for (int k = 0; k < KV; ++k) {
                const int j = glane + G * k;
                if (j < ra.NV) Vec<V>::add(acc[k], __ldcg(src + j));
            }
        }
        adagrad_row<V, KV>(ra, __ldg(srow + s0), acc, glane, lr, eps);
    }
}

template <int V, int KV>
cudaError_t run_reduce(mlkv_table* t, const float* grads, const uint32_t* srow, const uint32_t* spos,
                       int64_t n, cudaStream_t st, CallCounters* cur) {
    RowArgs ra{t->slots, t->geom.stride, t->geom.dpad, t->geom.NV, t->geom.G, t->geom.d};
    ErrSink err{&t->dstate->status, t->status_dev_alias};
    const int gs = persistent_blocks(t, (const void*)k_reduce_short<V, KV>, 256);
    MLKV_LAUNCH(t, MLKV_K_REDUCE_SHORT, (k_reduce_short<V, KV>), gs, 256, 0, st, ra, grads, srow, spos,
                t->s.seg_start, cur, t->s.long_seg, t->s.long_base, t->s.long_cnt, t->s.item_seg,
                (uint32_t)t->s.max_long, (uint32_t)t->s.max_items, t->cfg.lr, t->cfg.eps, err);
    const int gl = persistent_blocks(t, (const void*)k_reduce_long<V, KV>, 256);
    MLKV_LAUNCH(t, MLKV_K_REDUCE_LONG, (k_reduce_long<V, KV>), gl, 256, 0, st, ra, grads, srow, spos,
                t->s.seg_start, cur, t->s.long_seg, t->s.long_base, t->s.long_cnt, t->s.item_seg,
                t->s.partial, t->cfg.lr, t->cfg.eps);
    return cudaGetLastError();
}

}  // namespace

int64_t long_items_bound(int64_t max_batch) {
    return max_batch / kChunk + max_batch / (MLKV_SEQ_SEGMENT_MAX + 1) + 1;
}

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
