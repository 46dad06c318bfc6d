// wide_launch.h -- the head-dimension-256 kernels (wide_engine.cuh): their
// operations, launcher and device error word.
#pragma once

#include <cuda_runtime.h>

#include "engine_params.h"

namespace fbob {

// Fwd the forward (O and L, online softmax); Stats, DOut, DQ BoB Pass 1
// (alpha E D, dOtil, Qtil); StatsDO alpha E D and dOtil in one sweep; P2V,
// P2K BoB Pass 2 (Vtil, Ktil); BwdDQ, BwdDV, BwdDK the first backward.
enum class WOp { Fwd = 1, Stats, DOut, DQ, BwdDQ, P2V, P2K, BwdDV, BwdDK, StatsDO };

// drop: the instantiation with attention dropout (p.drop_* set)
cudaError_t launch_wide(WOp op, bool drop, const EngineParams& p, int nblocks, cudaStream_t s);

// Read and clear the error word of the head-dimension-256 unit.
cudaError_t take_wide_error(uint32_t* word, cudaStream_t s);

}  // namespace fbob
