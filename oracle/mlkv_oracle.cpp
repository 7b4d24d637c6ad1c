// MLKV embedding-store oracle -- TEST INFRASTRUCTURE ONLY.
//
// A plain, sequential CPU statement of what the batched embedding key-value
// path computes.  Only the tests, the smoke check and the CPU-baseline leg of
// the benchmark may load this library; the product path never does, and the
// two share no code, header, constant table or helper.
//
// What it follows (MLKV, arXiv 2504.01506):
//   * Section 3.1 (interfaces): Open(model_id, dim, staleness_bound),
//     Get(keys) -> values, Put(keys, values) is an upsert, Lookahead(keys).
//   * Section 3.2 (workflow, step 8) and Figure 2 (the Put of
//     values + emb_optimizer(gradients)): the gradient update is a per-key
//     read-modify-write of the stored embedding.
//   * Section 2.1 (the embedding map E): a lookup returns the d-dim row of a
//     sparse feature id; the gradient of E with respect to a row is the sum of
//     the gradients of all lookups of that id in the batch.
// The optimizer is element-wise Adagrad (Duchi, Hazan & Singer, 2011):
//     G <- G + g*g ;  w <- w - lr * g / (sqrt(G) + eps)
// applied once per distinct key on the summed gradient g of that key.
//
// Readings where the paper is silent (each is listed in the design notes):
//   * rows of new keys are initialised by a counter-based uniform draw,
//     init(seed,key,j) below, so any implementation can reproduce them;
//   * row ids are dense and handed out in first-occurrence order, call by call;
//   * duplicate keys inside one Put: the last occurrence wins;
//   * a Get (or gradient apply) of an absent key inserts it when
//     insert_on_miss is set, otherwise the Get writes NaN and reports
//     ORACLE_NOT_FOUND and the apply skips the key.
//   * checkpoints (Section 2.2 keeps a store's data by periodic checkpoints):
//     a checkpoint is every key in row order with its row and state; a
//     restore upserts them in that order (oracle_keys, oracle_export,
//     oracle_import), so the restored table has the same row ids.
//
// Arithmetic modes.  Rows and state are stored in fp32 (the table's storage
// type).  precision == 32 evaluates every operation as its own correctly
// rounded fp32 operation, in the order written above, gradient sums taken in
// occurrence order.  precision == 64 accumulates the gradient sums and
// evaluates the Adagrad step in fp64 and rounds to fp32 only when storing.
// Build with -ffp-contract=off so that no multiply-add is fused.
//
// ORACLE_MUTANT (compile-time, default 0) plants one deliberate mistake; it is
// used only by the test that shows the pins catch plausible errors.

#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <unordered_map>
#include <vector>

#ifndef ORACLE_MUTANT
#define ORACLE_MUTANT 0
#endif

namespace {

// SplitMix64 output function (Steele, Lea & Flood, "Fast splittable
// pseudorandom number generators", OOPSLA 2014): the value produced by a
// SplitMix64 generator whose state is z, i.e. mix(z + golden gamma).
uint64_t splitmix64(uint64_t z) {
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// Counter-based row initialisation U[lo, hi): element j of the row of `key`.
//   x = splitmix64(seed ^ splitmix64(key ^ (j * gamma)))
//   u = (x >> 40) * 2^-24          (exact: a 24-bit integer in fp32)
//   v = lo + u * (hi - lo)         (three separately rounded fp32 ops)
float init_value(uint64_t seed, uint64_t key, int64_t j, float lo, float hi) {
    const uint64_t gamma = 0x9E3779B97F4A7C15ull;
    uint64_t x = splitmix64(seed ^ splitmix64(key ^ ((uint64_t)j * gamma)));
    float u = (float)(x >> 40) * (1.0f / 16777216.0f);
    float span = hi - lo;
#if ORACLE_MUTANT == 7
    return u * span;  // planted: drops the offset lo
#else
    return lo + u * span;
#endif
}

struct Table {
    int32_t dim;
    float lr, eps, state_init, init_lo, init_hi;
    uint64_t seed;
    int32_t insert_on_miss;
    int32_t precision;
    std::unordered_map<uint64_t, int64_t> index;  // key -> dense row id
    std::vector<uint64_t> key_of_row;
    std::vector<float> w;  // [rows][dim]
    std::vector<float> G;  // [rows][dim]

    int64_t find(uint64_t k) const {
        auto it = index.find(k);
        return it == index.end() ? -1 : it->second;
    }
    // Inserts k with the counter-based init row and state_init; returns its row.
    int64_t insert_init(uint64_t k) {
        int64_t r = (int64_t)key_of_row.size();
        index.emplace(k, r);
        key_of_row.push_back(k);
        for (int32_t j = 0; j < dim; ++j) {
            w.push_back(init_value(seed, k, j, init_lo, init_hi));
#if ORACLE_MUTANT == 9
            G.push_back(0.0f);  // planted: ignores state_init
#else
            G.push_back(state_init);
#endif
        }
        return r;
    }
};

}  // namespace

extern "C" {

enum { ORACLE_OK = 0, ORACLE_ERR_INVALID = 1, ORACLE_NOT_FOUND = 7 };

uint64_t oracle_splitmix64(uint64_t z) { return splitmix64(z); }

float oracle_init_value(uint64_t seed, uint64_t key, int64_t j, float lo, float hi) {
    return init_value(seed, key, j, lo, hi);
}

int32_t oracle_mutant(void) { return ORACLE_MUTANT; }

void* oracle_open(int32_t dim, float lr, float eps, float state_init, float init_lo,
                  float init_hi, uint64_t seed, int32_t insert_on_miss, int32_t precision) {
    if (dim <= 0 || (precision != 32 && precision != 64)) return nullptr;
    Table* t = new Table();
    t->dim = dim;
    t->lr = lr;
    t->eps = eps;
    t->state_init = state_init;
    t->init_lo = init_lo;
    t->init_hi = init_hi;
    t->seed = seed;
    t->insert_on_miss = insert_on_miss;
    t->precision = precision;
    return t;
}

void oracle_close(void* h) { delete static_cast<Table*>(h); }

int64_t oracle_size(const void* h) {
    return (int64_t) static_cast<const Table*>(h)->key_of_row.size();
}

// Get(keys): sequential; out[i*dim..] = row of keys[i]; rows[i] = its row id
// (rows may be null).  Absent keys are inserted when insert_on_miss is set.
int32_t oracle_get(void* h, const int64_t* keys, int64_t n, float* out, int64_t* rows) {
    Table* t = static_cast<Table*>(h);
    if (n < 0) return ORACLE_ERR_INVALID;
    int32_t rc = ORACLE_OK;
    const int32_t d = t->dim;
#if ORACLE_MUTANT == 10
    // planted: presence decided for the whole batch up front, so every
    // occurrence of a new key inserts another row
    std::vector<char> absent(n);
    for (int64_t i = 0; i < n; ++i) absent[i] = t->find((uint64_t)keys[i]) < 0;
#endif
    for (int64_t i = 0; i < n; ++i) {
        uint64_t k = (uint64_t)keys[i];
        int64_t r = t->find(k);
#if ORACLE_MUTANT == 10
        if (absent[i] && t->insert_on_miss) r = t->insert_init(k);
#else
        if (r < 0 && t->insert_on_miss) r = t->insert_init(k);
#endif
        if (rows) rows[i] = r;
        if (r < 0) {
            rc = ORACLE_NOT_FOUND;
            for (int32_t j = 0; j < d; ++j) out[i * d + j] = std::numeric_limits<float>::quiet_NaN();
            continue;
        }
        std::memcpy(out + i * d, t->w.data() + r * d, sizeof(float) * d);
    }
    return rc;
}

// Put(keys, values): sequential upsert.  Present keys keep their state; new
// keys get state_init.  Duplicates: the later occurrence overwrites.
int32_t oracle_put(void* h, const int64_t* keys, int64_t n, const float* vals) {
    Table* t = static_cast<Table*>(h);
    if (n < 0) return ORACLE_ERR_INVALID;
    const int32_t d = t->dim;
#if ORACLE_MUTANT == 6
    for (int64_t i = n - 1; i >= 0; --i) {  // planted: first occurrence wins
#else
    for (int64_t i = 0; i < n; ++i) {
#endif
        uint64_t k = (uint64_t)keys[i];
        int64_t r = t->find(k);
        if (r < 0) r = t->insert_init(k);
        std::memcpy(t->w.data() + r * d, vals + i * d, sizeof(float) * d);
    }
    return ORACLE_OK;
}

// Import(keys, rows, state): sequential upsert of the row and, when state is
// not null, the state of each key (a new key without state gets state_init,
// a present one keeps its state).  Duplicates: the later occurrence
// overwrites.  With the keys of a checkpoint in row order, a fresh table gets
// the checkpoint's row ids.
int32_t oracle_import(void* h, const int64_t* keys, int64_t n, const float* rows, const float* state) {
    Table* t = static_cast<Table*>(h);
    if (n < 0) return ORACLE_ERR_INVALID;
    const int32_t d = t->dim;
    for (int64_t i = 0; i < n; ++i) {
        uint64_t k = (uint64_t)keys[i];
        int64_t r = t->find(k);
        if (r < 0) r = t->insert_init(k);
        std::memcpy(t->w.data() + r * d, rows + i * d, sizeof(float) * d);
#if ORACLE_MUTANT == 11
        (void)state;  // planted: the state is not restored
#else
        if (state) std::memcpy(t->G.data() + r * d, state + i * d, sizeof(float) * d);
#endif
    }
    return ORACLE_OK;
}

// Every key in row order (out has oracle_size entries).
int64_t oracle_keys(const void* h, int64_t* out) {
    const Table* t = static_cast<const Table*>(h);
    for (size_t r = 0; r < t->key_of_row.size(); ++r) out[r] = (int64_t)t->key_of_row[r];
    return (int64_t)t->key_of_row.size();
}

// Insert-if-absent with the init row (preloading a key set).
int32_t oracle_insert(void* h, const int64_t* keys, int64_t n) {
    Table* t = static_cast<Table*>(h);
    if (n < 0) return ORACLE_ERR_INVALID;
    for (int64_t i = 0; i < n; ++i) {
        uint64_t k = (uint64_t)keys[i];
        if (t->find(k) < 0) t->insert_init(k);
    }
    return ORACLE_OK;
}

// Gradient apply (the Rmw of Section 3.2 with Adagrad as emb_optimizer):
//  1. in occurrence order, acc[key] += grads[i]  (the sparse gradient of E);
//  2. for each distinct key, in first-occurrence order, one Adagrad step on
//     its summed gradient.
int32_t oracle_apply_grad(void* h, const int64_t* keys, int64_t n, const float* grads) {
    Table* t = static_cast<Table*>(h);
    if (n < 0) return ORACLE_ERR_INVALID;
    const int32_t d = t->dim;
    int32_t rc = ORACLE_OK;
    std::unordered_map<uint64_t, int64_t> slot;  // key -> index into order
    std::vector<int64_t> row_of;                 // per distinct key
    std::vector<float> acc32;
    std::vector<double> acc64;
    for (int64_t i = 0; i < n; ++i) {
        uint64_t k = (uint64_t)keys[i];
        auto ins = slot.emplace(k, (int64_t)row_of.size());
        int64_t s = ins.first->second;
        if (ins.second) {
            int64_t r = t->find(k);
            if (r < 0 && t->insert_on_miss) r = t->insert_init(k);
            if (r < 0) rc = ORACLE_NOT_FOUND;
            row_of.push_back(r);
            acc32.resize(acc32.size() + d, 0.0f);
            acc64.resize(acc64.size() + d, 0.0);
        }
        const float* g = grads + i * d;
        for (int32_t j = 0; j < d; ++j) {
#if ORACLE_MUTANT == 5
            acc32[s * d + j] = g[j];  // planted: drops the earlier occurrences
            acc64[s * d + j] = (double)g[j];
#else
            acc32[s * d + j] = acc32[s * d + j] + g[j];
            acc64[s * d + j] = acc64[s * d + j] + (double)g[j];
#endif
        }
#if ORACLE_MUTANT == 4
        // planted: one step per occurrence instead of one per distinct key
        if (row_of[s] >= 0) {
            for (int32_t j = 0; j < d; ++j) {
                float a = g[j];
                float* wp = &t->w[row_of[s] * d + j];
                float* Gp = &t->G[row_of[s] * d + j];
                *Gp = *Gp + a * a;
                *wp = *wp - t->lr * a / (std::sqrt(*Gp) + t->eps);
            }
        }
#endif
    }
#if ORACLE_MUTANT == 4
    return rc;
#endif
    for (size_t s = 0; s < row_of.size(); ++s) {
        int64_t r = row_of[s];
        if (r < 0) continue;
        for (int32_t j = 0; j < d; ++j) {
            float& wr = t->w[r * d + j];
            float& Gr = t->G[r * d + j];
            if (t->precision == 32) {
                const float a = acc32[s * d + j];
                const float t1 = a * a;
#if ORACLE_MUTANT == 2
                const float q0 = std::sqrt(Gr);  // planted: uses the old state
                const float Gn = Gr + t1;
                const float q = q0;
#else
                const float Gn = Gr + t1;
#if ORACLE_MUTANT == 1
                const float q = std::sqrt(Gn + t->eps) - t->eps;  // planted: sqrt(G + eps)
#else
                const float q = std::sqrt(Gn);
#endif
#endif
                const float den = q + t->eps;
                const float num = t->lr * a;
                const float u = num / den;
                Gr = Gn;
#if ORACLE_MUTANT == 3
                wr = wr + u;  // planted: wrong sign
#else
                wr = wr - u;
#endif
            } else {
                const double a = acc64[s * d + j];
                const double Gn = (double)Gr + a * a;
                const double wn = (double)wr - (double)t->lr * a / (std::sqrt(Gn) + (double)t->eps);
                Gr = (float)Gn;
                wr = (float)wn;
            }
        }
    }
    return rc;
}

// key -> row id, -1 when absent.
int32_t oracle_find(const void* h, const int64_t* keys, int64_t n, int64_t* rows) {
    const Table* t = static_cast<const Table*>(h);
    if (n < 0) return ORACLE_ERR_INVALID;
    for (int64_t i = 0; i < n; ++i) rows[i] = t->find((uint64_t)keys[i]);
    return ORACLE_OK;
}

// Row and state of each key (NaN when absent).  Returns the number found.
int64_t oracle_export(const void* h, const int64_t* keys, int64_t n, float* w, float* G) {
    const Table* t = static_cast<const Table*>(h);
    const int32_t d = t->dim;
    int64_t found = 0;
    for (int64_t i = 0; i < n; ++i) {
        int64_t r = t->find((uint64_t)keys[i]);
        for (int32_t j = 0; j < d; ++j) {
            float nan = std::numeric_limits<float>::quiet_NaN();
            if (w) w[i * d + j] = r < 0 ? nan : t->w[r * d + j];
            if (G) G[i * d + j] = r < 0 ? nan : t->G[r * d + j];
        }
        found += r >= 0;
    }
    return found;
}

// Distinct keys of a batch in first-occurrence order with their occurrence
// counts and first positions.  Returns the number of distinct keys.
int64_t oracle_dedup(const int64_t* keys, int64_t n, int64_t* uniq, int64_t* counts,
                     int64_t* first_pos) {
    std::unordered_map<uint64_t, int64_t> slot;
    int64_t u = 0;
    for (int64_t i = 0; i < n; ++i) {
        auto ins = slot.emplace((uint64_t)keys[i], u);
        int64_t s = ins.first->second;
        if (ins.second) {
            uniq[u] = keys[i];
            counts[u] = 0;
#if ORACLE_MUTANT == 8
            first_pos[u] = -1;  // planted: filled with the last position below
#else
            first_pos[u] = i;
#endif
            ++u;
        }
        counts[s] += 1;
#if ORACLE_MUTANT == 8
        first_pos[s] = i;
#endif
    }
    return u;
}

// Per distinct key (first-occurrence order) the sum of its gradient rows,
// taken in occurrence order, in fp32 (precision 32) or fp64 rounded to fp32
// (precision 64).  Returns the number of distinct keys.
int64_t oracle_segment_sums(const int64_t* keys, int64_t n, const float* grads, int32_t dim,
                            int32_t precision, int64_t* uniq, float* sums) {
    std::unordered_map<uint64_t, int64_t> slot;
    std::vector<double> acc64;
    std::vector<float> acc32;
    int64_t u = 0;
    for (int64_t i = 0; i < n; ++i) {
        auto ins = slot.emplace((uint64_t)keys[i], u);
        int64_t s = ins.first->second;
        if (ins.second) {
            uniq[u++] = keys[i];
            acc64.resize(acc64.size() + dim, 0.0);
            acc32.resize(acc32.size() + dim, 0.0f);
        }
        for (int32_t j = 0; j < dim; ++j) {
            acc32[s * dim + j] = acc32[s * dim + j] + grads[i * dim + j];
            acc64[s * dim + j] = acc64[s * dim + j] + (double)grads[i * dim + j];
        }
    }
    for (int64_t k = 0; k < u * dim; ++k) sums[k] = precision == 64 ? (float)acc64[k] : acc32[k];
    return u;
}

}  // extern "C"
