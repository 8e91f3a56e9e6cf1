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
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
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

using Keyed = std::pair<uint64_t, int32_t>;   // (key, row): ties broken by row

void draw_partition(const cm_shuffle &S, int64_t t, std::vector<int32_t> &owner)
{
    std::vector<Keyed> keys(S.q);
    for (int64_t r = 0; r < S.q; ++r)
        keys[r] = {mix64(S.partition_seed, (uint64_t)t * (uint64_t)S.q + (uint64_t)r),
                   (int32_t)r};
    std::sort(keys.begin(), keys.end());
    owner.assign(S.q, 0);
    for (int64_t pos = 0; pos < S.q; ++pos) owner[keys[pos].second] = (int32_t)(pos / S.per);
}

// Sets bit i of next[r] for every r in S_i (owner[r] == i) and for the
// s - q/n rows with candidate[r] != 0 whose keys are smallest.
void refill(const cm_shuffle &S, int64_t t, int32_t i, const std::vector<int32_t> &owner,
            const std::vector<char> &candidate, std::vector<uint64_t> &next)
{
    const uint64_t bit = 1ull << i;
    std::vector<Keyed> cand;
    for (int64_t r = 0; r < S.q; ++r) {
        if (owner[r] == i) {
            next[r] |= bit;
        } else if (candidate[r]) {
            const uint64_t idx = ((uint64_t)t * (uint64_t)S.n + (uint64_t)i) * (uint64_t)S.q + (uint64_t)r;
            cand.push_back({mix64(S.cache_seed, idx), (int32_t)r});
        }
    }
    const size_t keep = (size_t)(S.s - S.per);
    if (cand.size() > keep) std::nth_element(cand.begin(), cand.begin() + keep, cand.end());
    for (size_t c = 0; c < std::min(keep, cand.size()); ++c) next[cand[c].second] |= bit;
}

struct Needed {
    uint64_t set;     // I = workers caching r, plus i
    int32_t worker;   // i: new owner of r
    int32_t row;      // r
    int32_t msg;      // message row carrying r
    int32_t entry;    // index of r among the summed rows (message order)
};

cm_status plan_transition(cm_shuffle &S)
{
    const int32_t n = S.n;
    const int64_t q = S.q, s = S.s;
    const int64_t t1 = S.t + 1;
    std::vector<int32_t> owner1;
    draw_partition(S, t1, owner1);

    // rows of S_i^{t+1} missing from cache i, grouped by (I, i, r)
    std::vector<Needed> need;
    for (int64_t r = 0; r < q; ++r) {
        const int32_t i = owner1[r];
        const uint64_t have = S.cached[r];
        if (have & (1ull << i)) continue;
        need.push_back({have | (1ull << i), i, (int32_t)r, -1, -1});
    }
    std::sort(need.begin(), need.end(), [](const Needed &a, const Needed &b) {
        if (a.set != b.set) return a.set < b.set;
        if (a.worker != b.worker) return a.worker < b.worker;
        return a.row < b.row;
    });

    // Alg. 1: one zero-padded block sum per I, as rows of a CSR program
    S.enc_ptr.assign(1, 0);
    S.enc_src.clear();
    S.msg_worker.clear();
    S.msg_set.clear();
    S.message_sets = 0;
    std::vector<size_t> run_begin, run_len;
    for (size_t g = 0; g < need.size();) {
        size_t h = g;
        while (h < need.size() && need[h].set == need[g].set) ++h;
        run_begin.clear();
        run_len.clear();
        size_t ell = 0;
        for (size_t a = g; a < h;) {           // one run per worker of I
            size_t b = a;
            while (b < h && need[b].worker == need[a].worker) ++b;
            run_begin.push_back(a);
            run_len.push_back(b - a);
            ell = std::max(ell, b - a);
            a = b;
        }
        for (size_t j = 0; j < ell; ++j) {
            const int32_t m = (int32_t)S.msg_set.size();
            for (size_t w = 0; w < run_begin.size(); ++w) {
                if (j >= run_len[w]) continue;          // shorter block: zero row
                Needed &e = need[run_begin[w] + j];
                e.msg = m;
                e.entry = (int32_t)S.enc_src.size();
                S.enc_src.push_back(e.row);
                S.msg_worker.push_back(e.worker);
            }
            S.enc_ptr.push_back((int32_t)S.enc_src.size());
            S.msg_set.push_back(need[g].set);
        }
        ++S.message_sets;
        g = h;
    }

    // received rows in (worker, row) order; decode program in entry order
    std::sort(need.begin(), need.end(), [](const Needed &a, const Needed &b) {
        if (a.worker != b.worker) return a.worker < b.worker;
        return a.row < b.row;
    });
    const int64_t R = (int64_t)need.size();
    S.recv_row.resize(R);
    S.recv_ptr.assign(n + 1, 0);
    S.dec_msg.resize(R);
    S.dec_dst.resize(R);
    for (int64_t u = 0; u < R; ++u) {
        const Needed &e = need[u];
        S.recv_row[u] = e.row;
        ++S.recv_ptr[e.worker + 1];
        S.dec_msg[e.entry] = e.msg;
        S.dec_dst[e.entry] = (int32_t)u;
    }
    for (int32_t i = 0; i < n; ++i) S.recv_ptr[i + 1] += S.recv_ptr[i];
    S.dec_ptr.assign(1, 0);
    S.dec_slot.clear();
    for (int64_t x = 0; x < R; ++x) {
        const int32_t i = S.msg_worker[x], m = S.dec_msg[x];
        for (int32_t y = S.enc_ptr[m]; y < S.enc_ptr[m + 1]; ++y) {
            if (y == x) continue;
            const int32_t slot = S.slot_of[(int64_t)i * q + S.enc_src[y]];
            if (slot < 0) return CM_EINVAL;   // unreachable: every other row of I is cached at i
            S.dec_slot.push_back((int32_t)(i * s + slot));
        }
        S.dec_ptr.push_back((int32_t)S.dec_slot.size());
    }

    // cache update rule: S_i^{t+1} plus s - q/n rows of C_i^t \ S_i^{t+1}
    std::vector<uint64_t> next(q, 0);
    std::vector<char> keepable(q);
    for (int32_t i = 0; i < n; ++i) {
        const uint64_t bit = 1ull << i;
        for (int64_t r = 0; r < q; ++r) keepable[r] = (S.cached[r] & bit) && owner1[r] != i;
        refill(S, t1, i, owner1, keepable, next);
    }

    // commit: received rows of worker i fill, in order, the slots of cache i
    // whose rows were dropped (as many as rows received: both caches hold s)
    S.com_dst.resize(R);
    for (int32_t i = 0; i < n; ++i) {
        const uint64_t bit = 1ull << i;
        int64_t u = S.recv_ptr[i];
        for (int64_t c = 0; c < s; ++c) {
            const int64_t g = (int64_t)i * s + c;
            const int32_t old = S.slot_row[g];
            if (next[old] & bit) continue;
            if (u >= S.recv_ptr[i + 1]) return CM_EINVAL;   // unreachable
            S.slot_of[(int64_t)i * q + old] = -1;
            S.com_dst[u] = (int32_t)g;
            ++u;
        }
        if (u != S.recv_ptr[i + 1]) return CM_EINVAL;       // unreachable
        for (u = S.recv_ptr[i]; u < S.recv_ptr[i + 1]; ++u) {
            const int32_t g = S.com_dst[u];
            S.slot_row[g] = S.recv_row[u];
            S.slot_of[(int64_t)i * q + S.recv_row[u]] = (int32_t)(g - i * s);
        }
    }
    S.cached.swap(next);
    S.owner.swap(owner1);
    S.t = t1;
    S.planned = true;
    return CM_OK;
}

void fill_stats(const cm_shuffle &S, cm_shuffle_stats *st)
{
    st->iteration = S.t;
    st->message_sets = S.planned ? S.message_sets : 0;
    st->coded_rows = S.planned ? (int64_t)S.msg_set.size() : 0;
    st->uncoded_rows = S.planned ? (int64_t)S.recv_row.size() : 0;
    st->subtractions = S.planned ? (int64_t)S.dec_slot.size() : 0;
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
        S->cached.assign(q, 0);
        std::vector<char> outside(q);
        for (int32_t i = 0; i < n; ++i) {
            for (int64_t r = 0; r < q; ++r) outside[r] = S->owner[r] != i;
            refill(*S, 0, i, S->owner, outside, S->cached);
        }
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
    if (!S) return CM_EINVAL;
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
    if (recv_ptr) std::memcpy(recv_ptr, S->recv_ptr.data(), sizeof(int32_t) * (S->n + 1));
    if (recv_row && !S->recv_row.empty())
        std::memcpy(recv_row, S->recv_row.data(), sizeof(int32_t) * S->recv_row.size());
    return CM_OK;
}

cm_status cm_shuffle_caches(const cm_shuffle *S, int32_t *owner, int32_t *slot_row)
{
    if (!S) return CM_EINVAL;
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
