// lc_host.h -- host-side internals shared by the translation units of
// liblayercheck.so (not part of the public ABI).
#pragma once

#include <stdint.h>

#include "layercheck.h"

namespace lc {

// Layout of a context or a store: the number of layers and each layer's
// packed block size (§3.1 layout).
int32_t ctx_nlayers(const lc_ctx* ctx);
int32_t store_nlayers(const lc_store* st);
const uint64_t* store_layer_bytes(const lc_store* st);

// Appends a durable version of `layer` to a log store (versions_per_layer
// = 0) and returns the host address of its block (the layer's block size),
// or nullptr when the store is not a log or has no room.  The version's
// step is set later with store_set_step.
uint8_t* store_append(lc_store* st, int32_t layer, int64_t* index_out);
void store_set_step(lc_store* st, int64_t index, int64_t step);

// Sets the thread-local message of lc_last_error() (and returns `st`).
lc_status fail_status(lc_status st, const char* fmt, ...);
void set_last_error(const char* msg);

}  // namespace lc
