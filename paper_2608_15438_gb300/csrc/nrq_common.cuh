// Shared definitions of the per-query building blocks of the query path
// (nrq_route.cuh: route_warp, nrq_select.cuh: select_block,
// nrq_refine.cuh: refine_block).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"

namespace nrq {

constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kEmpty = ~0ull;

__device__ __forceinline__ void set_err(int *err, int code) { atomicCAS(err, 0, code); }

}  // namespace nrq
