// seqtab_internal.h -- host state of a kv_seqtab (not part of the ABI).
#pragma once

#include <cstdint>
#include <vector>

#include "kvpool.h"

struct kv_seqtab {
    kv_pool *pool = nullptr;
    int layout = 0;
    int S = 0;           // slots
    int max_blocks = 0;  // table row length
    int bs = 0;
    std::vector<int32_t> table;    // [S][max_blocks], -1 = no block
    std::vector<int32_t> lens;     // [S]
    std::vector<int32_t> held;     // blocks held per slot (a prefix of the row)
    std::vector<uint8_t> pending;  // entry changed since the last sync
    std::vector<int32_t> changed;  // flat indices of pending entries
    bool full_dirty = true;        // the device copy has never been written
    kv_seqtab_counters counters;
};
