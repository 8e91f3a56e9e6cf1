// Internal state of a coded-shuffling instance (Sec. IV), shared by the host
// planner (shuffle.cpp) and the device side (k_shuffle.cu).
#pragma once

#include <stdint.h>

#include <vector>

#include "../../include/cm.h"

// Element offsets (int32 words) of the row programs inside a caller-provided
// device workspace; each offset is a multiple of 64 words (256 bytes).  The
// sizes are the worst case over every transition of the instance.
struct ShuffleLayout {
    int64_t enc_ptr, enc_src;            // encode: CSR over message rows
    int64_t dec_msg, dec_ptr, dec_slot;  // decode: message row + CSR of subtracted slots
    int64_t dec_dst;                     // decode: received row of each entry
    int64_t com_dst;                     // commit: destination slot of each decoded row
    int64_t fill_row;                    // fill: data row of every cache slot
    int64_t total;                       // words
};

struct cm_shuffle {
    int32_t n;
    int64_t q, s, per;                 // per = q / n rows of every S_i
    uint64_t partition_seed, cache_seed;
    int64_t t;                         // iteration of the current partition and caches
    std::vector<int32_t> owner;        // owner[r] = i with r in S_i^t
    std::vector<uint64_t> cached;      // bit i of cached[r]: r in C_i^t
    std::vector<int32_t> slot_row;     // slot_row[i s + c]: row in slot c of cache i
    std::vector<int32_t> slot_of;      // slot_of[i q + r]: slot of r in cache i, -1 if absent
    // Row programs of the transition t-1 -> t (empty before the first one).
    bool planned = false;
    std::vector<int32_t> enc_ptr, enc_src, msg_worker;
    std::vector<uint64_t> msg_set;
    std::vector<int32_t> dec_msg, dec_ptr, dec_slot, dec_dst, com_dst;
    std::vector<int32_t> recv_ptr, recv_row;
    int64_t message_sets = 0;
    // Sizes of the current programs: coded rows, received rows, subtracted rows
    int64_t n_coded = 0, n_recv = 0, n_sub = 0;
    // Workspace the current programs were last copied to, and for which t.
    const void *uploaded_ws = nullptr;
    int64_t uploaded_t = -1;
    // Device planning: once set, the partition, caches and programs live in
    // this workspace (the host tables above are stale), and dev_cur selects
    // the current copy of the double-buffered partition and cache masks.
    void *device_ws = nullptr;
    int dev_cur = 0;
    uint32_t sort_epoch = 0;           // tag of the device radix passes' tile flags
};

ShuffleLayout shuffle_layout(int32_t n, int64_t q, int64_t s);

// Device-mode queries (k_shuffle_plan.cu): copy the current tables out of
// the device workspace (synchronous).
cm_status shuffle_device_plan(const cm_shuffle *S, int32_t *msg_ptr, int32_t *msg_src,
                              int32_t *msg_worker, uint64_t *msg_set);
cm_status shuffle_device_received(const cm_shuffle *S, int32_t *recv_ptr, int32_t *recv_row);
cm_status shuffle_device_caches(const cm_shuffle *S, int32_t *owner, int32_t *slot_row);
