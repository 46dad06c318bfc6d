// launch.h -- host-side launchers of the tile engines (one translation unit
// per engine) and access to each unit's device error word.
#pragma once

#include <cuda_runtime.h>

#include "engine_params.h"

namespace fbob {

// Dynamic shared memory a launch requests: at least the engine's plan and at
// least 120 KB, so that one CTA (holding all 512 TMEM columns) runs per SM.
inline int launch_smem(int plan_bytes) { return plan_bytes > 120 * 1024 ? plan_bytes : 120 * 1024; }

// drop: the instantiation with attention dropout (p.drop_* set)
cudaError_t launch_row(RowOp op, int d, bool drop, const EngineParams& p, int nblocks,
                       cudaStream_t s);
cudaError_t launch_col(ColOp op, int d, bool drop, const EngineParams& p, int nblocks,
                       cudaStream_t s);

// Read and clear the error word of the row / column engine unit (the
// head-dimension-256 unit: wide_launch.h).
cudaError_t take_row_error(uint32_t* word, cudaStream_t s);
cudaError_t take_col_error(uint32_t* word, cudaStream_t s);

}  // namespace fbob
