// Coded shuffling (Sec. IV): the master's planner, host only.
//
// Before every iteration the q data rows are partitioned into n sets S_i of
// q/n rows (Sec. IV-A).  Cache i holds s rows: S_i plus s - q/n rows that the
// cache update rule keeps, drawn without replacement from the old cache
// outside the new set (Sec. IV-B).  For the transition t -> t+1 the master
// sends, for every worker set I with |I| >= 2, the zero-padded sum over i in I
// of the rows of S_i^{t+1} that are cached exactly by I \ {i} (Alg. 1).  A
// row r of S_i^{t+1} missing from cache i is cached by some set H of workers
// (at least its previous owner), so it belongs to exactly one message, the
// one of I = H + {i}; worker i recovers it by subtracting the other rows of
// its message row, all of which it caches (decoding by subtraction).
//
// The planner turns one transition into row programs for the device:
//   encode  message row m = sum of data rows enc_src[enc_ptr[m] .. enc_ptr[m+1])
//   decode  for every entry x of a message row (one received row): received
//           row dec_dst[x] = message row dec_msg[x] minus the cache slots
//           dec_slot[dec_ptr[x] .. dec_ptr[x+1]) of the receiving worker;
//           entries run in message order, so the readers of one message
//           row are adjacent (one HBM read of it, the rest from L2, as one
//           multicast reaching every worker of I)
//   commit  received row t goes to cache slot com_dst[t] (a slot freed by a
//           row the cache update rule dropped)
// Message rows are ordered by the bit mask of I, then by position in the
// zero-padded blocks; within a block the rows of S_i ascend, and the entries
// of a message row ascend by worker.  Received rows are ordered by worker,
// then by data row.
//
// Random draws (SplitMix64, Steele, Lea and Flood 2014: state = seed + index
// * 0x9E3779B97F4A7C15, then the finaliser): the partition of iteration t
// orders the rows by (key of index t q + r under partition_seed, r) and gives
// positions [i q/n, (i+1) q/n) to worker i; a cache refill of worker i at
// iteration t keeps the s - q/n candidates with the smallest (key of index
// (t n + i) q + r under cache_seed, r).  At t = 0 the candidates are all rows
// outside S_i^0, so C_i^0 \ S_i^0 is uniform without replacement (the
// marginal law the rule maintains).
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <thread>
#include <unordered_map>
#include <vector>

#include "shuffle_internal.h"

namespace {

inline uint64_t mix64(uint64_t seed, uint64_t index)
{
    uint64_t z = seed + index * 0x9E3779B97F4A7C15ull;
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

// Runs body(j) for j = 0 .. count-1 on up to hardware_concurrency threads.
// Returns false if a body ran out of memory.
template <class Body>
bool parallel_for(int count, Body body)
{
    const int hw = std::max(1u, std::thread::hardware_concurrency());
    const int T = std::min(count, hw);
    std::atomic<bool> ok{true};
    auto run = [&](int tid) {
        try {
            for (int j = tid; j < count; j += T) body(j);
        } catch (const std::bad_alloc &) {
            ok = false;
        }
    };
    if (T <= 1) {
        run(0);
        return ok;
    }
    std::vector<std::thread> th;
    th.reserve(T - 1);
    for (int tid = 1; tid < T; ++tid) th.emplace_back(run, tid);
    run(0);
    for (auto &x : th) x.join();
    return ok;
}

struct Keyed {
    uint64_t key;
    int32_t row;
};

// Sorts by (key, row): one counting pass on the top 11 bits of the key, then
// every bucket (about 2^-11 of the rows, cache resident) sorted on its own,
// the buckets spread over threads.
void sort_keyed(std::vector<Keyed> &a)
{
    constexpr int kBits = 11;
    const size_t B = (size_t)1 << kBits;
    std::vector<int64_t> start(B + 1, 0);
    for (const Keyed &k : a) ++start[(k.key >> (64 - kBits)) + 1];
    for (size_t b = 0; b < B; ++b) start[b + 1] += start[b];
    std::vector<Keyed> out(a.size());
    {
        std::vector<int64_t> at(start.begin(), start.end() - 1);
        for (const Keyed &k : a) out[at[k.key >> (64 - kBits)]++] = k;
    }
    auto less = [](const Keyed &x, const Keyed &y) {
        return x.key != y.key ? x.key < y.key : x.row < y.row;
    };
    const int T = (int)std::max(1u, std::thread::hardware_concurrency());
    if (!parallel_for(T, [&](int tid) {
            for (size_t b = (size_t)tid; b < B; b += (size_t)T)
                std::sort(out.begin() + start[b], out.begin() + start[b + 1], less);
        }))
        throw std::bad_alloc();
    a.swap(out);
}

void draw_partition(const cm_shuffle &S, int64_t t, std::vector<int32_t> &owner)
{
    std::vector<Keyed> keys(S.q);
    for (int64_t r = 0; r < S.q; ++r)
        keys[r] = {mix64(S.partition_seed, (uint64_t)t * (uint64_t)S.q + (uint64_t)r),
                   (int32_t)r};
    sort_keyed(keys);
    owner.assign(S.q, 0);
    for (int64_t pos = 0; pos < S.q; ++pos) owner[keys[pos].row] = (int32_t)(pos / S.per);
}

// The s - q/n rows kept by cache i at iteration t: among the rows r with
// is_candidate(r), those with the smallest (key, r).
template <class Pred>
std::vector<int32_t> draw_kept(const cm_shuffle &S, int64_t t, int32_t i, Pred is_candidate)
{
    std::vector<Keyed> cand;
    cand.reserve((size_t)S.s);
    const uint64_t base = ((uint64_t)t * (uint64_t)S.n + (uint64_t)i) * (uint64_t)S.q;
    for (int64_t r = 0; r < S.q; ++r)
        if (is_candidate(r)) cand.push_back({mix64(S.cache_seed, base + (uint64_t)r), (int32_t)r});
    const size_t keep = std::min((size_t)(S.s - S.per), cand.size());
    auto less = [](const Keyed &a, const Keyed &b) {
        return a.key != b.key ? a.key < b.key : a.row < b.row;
    };
    if (cand.size() > keep) std::nth_element(cand.begin(), cand.begin() + keep, cand.end(), less);
    std::vector<int32_t> rows(keep);
    for (size_t c = 0; c < keep; ++c) rows[c] = cand[c].row;
    return rows;
}

// Cache masks of iteration t: S_i plus the kept rows of every worker.
std::vector<uint64_t> cache_masks(const cm_shuffle &S, const std::vector<int32_t> &owner,
                                  const std::vector<std::vector<int32_t>> &kept)
{
    std::vector<uint64_t> mask(S.q, 0);
    for (int64_t r = 0; r < S.q; ++r) mask[r] = 1ull << owner[r];
    for (int32_t i = 0; i < S.n; ++i)
        for (int32_t r : kept[i]) mask[r] |= 1ull << i;
    return mask;
}

// Stable counting sort of `idx` by key(idx[u]) in [0, buckets).
template <class Key>
void counting_sort(std::vector<int32_t> &idx, size_t buckets, Key key)
{
    std::vector<int64_t> start(buckets + 1, 0);
    for (int32_t u : idx) ++start[key(u) + 1];
    for (size_t b = 0; b < buckets; ++b) start[b + 1] += start[b];
    std::vector<int32_t> out(idx.size());
    for (int32_t u : idx) out[start[key(u)]++] = u;
    idx.swap(out);
}

cm_status plan_transition(cm_shuffle &S)
{
    const int32_t n = S.n;
    const int64_t q = S.q, s = S.s;
    const int64_t t1 = S.t + 1;
    S.planned = false;   // no program of this transition is usable until it is complete
    std::vector<int32_t> owner1;
    draw_partition(S, t1, owner1);

    // rows of S_i^{t+1} missing from cache i, scanned in ascending row order
    std::vector<int32_t> row, worker;
    std::vector<uint64_t> set;
    for (int64_t r = 0; r < q; ++r) {
        const int32_t i = owner1[r];
        const uint64_t have = S.cached[r];
        if (have & (1ull << i)) continue;
        row.push_back((int32_t)r);
        worker.push_back(i);
        set.push_back(have | (1ull << i));   // I = workers caching r, plus i
    }
    const int64_t R = (int64_t)row.size();

    // received-row order: (worker, row), a stable sort by worker
    std::vector<int32_t> byw(R);
    for (int64_t u = 0; u < R; ++u) byw[u] = (int32_t)u;
    counting_sort(byw, (size_t)n, [&](int32_t u) { return (size_t)worker[u]; });
    // message order: (I, worker, row), a stable sort of that by the rank of I
    // among the distinct sets (ids by first appearance, then ranked)
    std::vector<int32_t> rank(R);
    std::vector<uint64_t> masks;
    if (n <= 20) {
        std::vector<int32_t> id((size_t)1 << n, -1);
        for (int64_t u = 0; u < R; ++u) {
            int32_t &v = id[set[u]];
            if (v < 0) {
                v = (int32_t)masks.size();
                masks.push_back(set[u]);
            }
            rank[u] = v;
        }
    } else {
        std::unordered_map<uint64_t, int32_t> id;
        for (int64_t u = 0; u < R; ++u) {
            auto it = id.emplace(set[u], (int32_t)masks.size());
            if (it.second) masks.push_back(set[u]);
            rank[u] = it.first->second;
        }
    }
    {
        std::vector<int32_t> order(masks.size());
        for (size_t d = 0; d < masks.size(); ++d) order[d] = (int32_t)d;
        std::sort(order.begin(), order.end(),
                  [&](int32_t x, int32_t y) { return masks[x] < masks[y]; });
        std::vector<int32_t> to_rank(masks.size());
        for (size_t d = 0; d < order.size(); ++d) to_rank[order[d]] = (int32_t)d;
        for (int64_t u = 0; u < R; ++u) rank[u] = to_rank[rank[u]];
    }
    std::vector<int32_t> byset(byw);
    counting_sort(byset, masks.size(), [&](int32_t u) { return (size_t)rank[u]; });
    // the needed rows in message order, as contiguous arrays
    std::vector<int32_t> krow(R), kworker(R), krank(R);
    for (int64_t k = 0; k < R; ++k) {
        const int32_t u = byset[k];
        krow[k] = row[u];
        kworker[k] = worker[u];
        krank[k] = rank[u];
    }

    // Alg. 1: one zero-padded block sum per I, as rows of a CSR program
    std::vector<int32_t> msg_of(R), entry_of(R);    // indexed by position k
    S.enc_ptr.assign(1, 0);
    S.enc_src.resize(R);
    S.msg_worker.resize(R);
    S.msg_set.clear();
    S.message_sets = (int64_t)masks.size();
    std::vector<int64_t> run_begin, run_len;
    int32_t x = 0;
    for (int64_t g = 0; g < R;) {
        int64_t h = g;
        while (h < R && krank[h] == krank[g]) ++h;
        run_begin.clear();
        run_len.clear();
        int64_t ell = 0;
        for (int64_t a = g; a < h;) {          // one run per worker of I
            int64_t b = a;
            while (b < h && kworker[b] == kworker[a]) ++b;
            run_begin.push_back(a);
            run_len.push_back(b - a);
            ell = std::max(ell, b - a);
            a = b;
        }
        const uint64_t I = set[byset[g]];
        for (int64_t j = 0; j < ell; ++j) {
            const int32_t m = (int32_t)S.msg_set.size();
            for (size_t w = 0; w < run_begin.size(); ++w) {
                if (j >= run_len[w]) continue;          // shorter block: zero row
                const int64_t k = run_begin[w] + j;
                msg_of[k] = m;
                entry_of[k] = x;
                S.enc_src[x] = krow[k];
                S.msg_worker[x] = kworker[k];
                ++x;
            }
            S.enc_ptr.push_back(x);
            S.msg_set.push_back(I);
        }
        g = h;
    }
    // position k of every needed row u
    std::vector<int32_t> pos(R);
    for (int64_t k = 0; k < R; ++k) pos[byset[k]] = (int32_t)k;

    // received rows, and the decode program in entry order
    S.recv_row.resize(R);
    S.recv_ptr.assign(n + 1, 0);
    S.dec_msg.resize(R);
    S.dec_dst.resize(R);
    S.dec_ptr.resize(R + 1);
    std::vector<int32_t> entry_w(R);     // entry of the v-th received row
    for (int64_t v = 0; v < R; ++v) {
        const int32_t u = byw[v], k = pos[u];
        S.recv_row[v] = row[u];
        ++S.recv_ptr[worker[u] + 1];
        entry_w[v] = entry_of[k];
        S.dec_msg[entry_of[k]] = msg_of[k];
        S.dec_dst[entry_of[k]] = (int32_t)v;
    }
    for (int32_t i = 0; i < n; ++i) S.recv_ptr[i + 1] += S.recv_ptr[i];
    S.dec_ptr[0] = 0;
    for (int64_t x = 0; x < R; ++x) {
        const int32_t m = S.dec_msg[x];
        S.dec_ptr[x + 1] = S.dec_ptr[x] + (S.enc_ptr[m + 1] - S.enc_ptr[m] - 1);
    }
    S.dec_slot.resize(S.dec_ptr[R]);
    // slots of the subtracted rows, one worker per thread (its slot table only)
    std::atomic<bool> consistent{true};
    bool ok = parallel_for(n, [&](int32_t i) {
        const int32_t *slot_of = S.slot_of.data() + (int64_t)i * q;
        for (int64_t v = S.recv_ptr[i]; v < S.recv_ptr[i + 1]; ++v) {
            const int32_t x = entry_w[v], m = S.dec_msg[x];
            int32_t at = S.dec_ptr[x];
            for (int32_t y = S.enc_ptr[m]; y < S.enc_ptr[m + 1]; ++y) {
                if (y == x) continue;
                const int32_t slot = slot_of[S.enc_src[y]];
                if (slot < 0) consistent = false;   // unreachable: the rows of I \ {i} are cached at i
                S.dec_slot[at++] = (int32_t)(i * s + slot);
            }
        }
    });
    if (!ok) return CM_ENOMEM;
    if (!consistent) return CM_EINVAL;

    // cache update rule: S_i^{t+1} plus s - q/n rows of C_i^t \ S_i^{t+1}
    std::vector<std::vector<int32_t>> kept(n);
    ok = parallel_for(n, [&](int32_t i) {
        const uint64_t bit = 1ull << i;
        kept[i] = draw_kept(S, t1, i, [&](int64_t r) {
            return (S.cached[r] & bit) && owner1[r] != i;
        });
    });
    if (!ok) return CM_ENOMEM;
    std::vector<uint64_t> next = cache_masks(S, owner1, kept);

    // commit: received rows of worker i fill, in order, the slots of cache i
    // whose rows were dropped (as many as rows received: both caches hold s)
    S.com_dst.resize(R);
    ok = parallel_for(n, [&](int32_t i) {
        const uint64_t bit = 1ull << i;
        int32_t *slot_of = S.slot_of.data() + (int64_t)i * q;
        int64_t v = S.recv_ptr[i];
        for (int64_t c = 0; c < s; ++c) {
            const int64_t g = (int64_t)i * s + c;
            const int32_t old = S.slot_row[g];
            if (next[old] & bit) continue;
            if (v >= S.recv_ptr[i + 1]) {      // unreachable
                consistent = false;
                return;
            }
            slot_of[old] = -1;
            S.com_dst[v++] = (int32_t)g;
        }
        if (v != S.recv_ptr[i + 1]) consistent = false;   // unreachable
        for (v = S.recv_ptr[i]; v < S.recv_ptr[i + 1]; ++v) {
            const int32_t g = S.com_dst[v];
            S.slot_row[g] = S.recv_row[v];
            slot_of[S.recv_row[v]] = (int32_t)(g - i * s);
        }
    });
    if (!ok) return CM_ENOMEM;
    if (!consistent) return CM_EINVAL;
    S.cached.swap(next);
    S.owner.swap(owner1);
    S.t = t1;
    S.n_coded = (int64_t)S.msg_set.size();
    S.n_recv = R;
    S.n_sub = (int64_t)S.dec_slot.size();
    S.planned = true;
    return CM_OK;
}

void fill_stats(const cm_shuffle &S, cm_shuffle_stats *st)
{
    st->iteration = S.t;
    st->message_sets = S.planned ? S.message_sets : 0;
    st->coded_rows = S.planned ? S.n_coded : 0;
    st->uncoded_rows = S.planned ? S.n_recv : 0;
    st->subtractions = S.planned ? S.n_sub : 0;
}

int64_t up64(int64_t x) { return (x + 63) & ~(int64_t)63; }

}  // namespace

ShuffleLayout shuffle_layout(int32_t n, int64_t q, int64_t s)
{
    ShuffleLayout L;
    int64_t at = 0;
    L.enc_ptr = at;  at += up64(q + 1);
    L.enc_src = at;  at += up64(q);
    L.dec_msg = at;  at += up64(q);
    L.dec_ptr = at;  at += up64(q + 1);
    L.dec_slot = at; at += up64(q * (int64_t)(n - 1));
    L.dec_dst = at;  at += up64(q);
    L.com_dst = at;  at += up64(q);
    L.fill_row = at; at += up64((int64_t)n * s);
    L.total = at;
    return L;
}

extern "C" {

cm_status cm_shuffle_create(int32_t n, int64_t q, int64_t s, uint64_t partition_seed,
                            uint64_t cache_seed, cm_shuffle **out)
{
    if (!out) return CM_EINVAL;
    *out = nullptr;
    if (n < 2 || n > 64 || q < n || q % n != 0 || s < q / n || s > q) return CM_EINVAL;
    if (q * (int64_t)n >= ((int64_t)1 << 31)) return CM_EINVAL;
    cm_shuffle *S = new (std::nothrow) cm_shuffle();
    if (!S) return CM_ENOMEM;
    try {
        S->n = n;
        S->q = q;
        S->s = s;
        S->per = q / n;
        S->partition_seed = partition_seed;
        S->cache_seed = cache_seed;
        S->t = 0;
        draw_partition(*S, 0, S->owner);
        std::vector<std::vector<int32_t>> kept(n);
        const cm_shuffle &C = *S;
        if (!parallel_for(n, [&](int32_t i) {
                kept[i] = draw_kept(C, 0, i, [&](int64_t r) { return C.owner[r] != i; });
            }))
            throw std::bad_alloc();
        S->cached = cache_masks(*S, S->owner, kept);
        // slots of cache i hold its rows in ascending order
        S->slot_row.resize((size_t)n * s);
        S->slot_of.assign((size_t)n * q, -1);
        for (int32_t i = 0; i < n; ++i) {
            int64_t c = 0;
            for (int64_t r = 0; r < q; ++r) {
                if (!(S->cached[r] & (1ull << i))) continue;
                S->slot_row[(size_t)i * s + c] = (int32_t)r;
                S->slot_of[(size_t)i * q + r] = (int32_t)c;
                ++c;
            }
        }
    } catch (const std::bad_alloc &) {
        delete S;
        return CM_ENOMEM;
    }
    *out = S;
    return CM_OK;
}

void cm_shuffle_destroy(cm_shuffle *S) { delete S; }

cm_status cm_shuffle_next(cm_shuffle *S, cm_shuffle_stats *stats)
{
    if (!S || S->device_ws) return CM_EINVAL;   // device-planned instances plan on the device
    cm_status st;
    try {
        st = plan_transition(*S);
    } catch (const std::bad_alloc &) {
        return CM_ENOMEM;
    }
    if (st == CM_OK && stats) fill_stats(*S, stats);
    return st;
}

cm_status cm_shuffle_query(const cm_shuffle *S, cm_shuffle_stats *stats)
{
    if (!S || !stats) return CM_EINVAL;
    fill_stats(*S, stats);
    return CM_OK;
}

cm_status cm_shuffle_plan(const cm_shuffle *S, int32_t *msg_ptr, int32_t *msg_src,
                          int32_t *msg_worker, uint64_t *msg_set)
{
    if (!S) return CM_EINVAL;
    if (!S->planned) return CM_EINVAL;
    if (S->device_ws) return shuffle_device_plan(S, msg_ptr, msg_src, msg_worker, msg_set);
    auto put = [](void *dst, const void *src, size_t bytes) {
        if (dst && bytes) std::memcpy(dst, src, bytes);
    };
    put(msg_ptr, S->enc_ptr.data(), sizeof(int32_t) * S->enc_ptr.size());
    put(msg_src, S->enc_src.data(), sizeof(int32_t) * S->enc_src.size());
    put(msg_worker, S->msg_worker.data(), sizeof(int32_t) * S->msg_worker.size());
    put(msg_set, S->msg_set.data(), sizeof(uint64_t) * S->msg_set.size());
    return CM_OK;
}

cm_status cm_shuffle_received(const cm_shuffle *S, int32_t *recv_ptr, int32_t *recv_row)
{
    if (!S || !S->planned) return CM_EINVAL;
    if (S->device_ws) return shuffle_device_received(S, recv_ptr, recv_row);
    if (recv_ptr) std::memcpy(recv_ptr, S->recv_ptr.data(), sizeof(int32_t) * (S->n + 1));
    if (recv_row && !S->recv_row.empty())
        std::memcpy(recv_row, S->recv_row.data(), sizeof(int32_t) * S->recv_row.size());
    return CM_OK;
}

cm_status cm_shuffle_caches(const cm_shuffle *S, int32_t *owner, int32_t *slot_row)
{
    if (!S) return CM_EINVAL;
    if (S->device_ws) return shuffle_device_caches(S, owner, slot_row);
    if (owner) std::memcpy(owner, S->owner.data(), sizeof(int32_t) * S->q);
    if (slot_row) std::memcpy(slot_row, S->slot_row.data(), sizeof(int32_t) * S->slot_row.size());
    return CM_OK;
}

// Rate of the coded scheme as the series the proof of the coded shuffling
// rate theorem sums before its closed form: R_c = sum_{i=2}^n C(n,i) (q/n)
// ((i-1)/n) p^{i-2} (1-p)^{n-i+1}, p = (s - q/n)/(q - q/n).  Every term is
// non-negative, so the sum stays accurate as p -> 0, where the closed form
// cancels (its limit there is R_u / 2).  R_u = q (1 - s/q).
cm_status cm_shuffle_rates(int32_t n, double q, double s, double *coded, double *uncoded)
{
    if (n < 2 || n > 1024 || !(q > 0.0) || !coded || !uncoded) return CM_EINVAL;
    if (!(s >= q / n) || !(s <= q)) return CM_EINVAL;
    const double p = (s - q / n) / (q - q / n);
    double sum = 0.0;
    for (int i = 2; i <= n; ++i) {
        const double lc = std::lgamma(n + 1.0) - std::lgamma(i + 1.0) - std::lgamma(n - i + 1.0);
        const double pw = (i == 2 ? 1.0 : std::pow(p, i - 2)) * std::pow(1.0 - p, n - i + 1);
        sum += std::exp(lc) * (i - 1) / n * pw;
    }
    *coded = q / n * sum;
    *uncoded = q * (1.0 - s / q);
    return CM_OK;
}

}  // extern "C"
