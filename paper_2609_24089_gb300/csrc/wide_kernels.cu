// wide_kernels.cu -- instantiations and launcher of the head-dimension-256
// kernels (wide_engine.cuh): forward (eq. 1), first backward (eqs. 2-3) and
// both passes of BoB (Alg. 2), each with and without dropout.
#include "launch.h"
#include "wide_engine.cuh"
#include "wide_launch.h"

namespace fbob {

template <WOp OP, bool DROP>
static cudaError_t launch_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(WCfg<OP>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(wide_engine<OP, DROP>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  wide_engine<OP, DROP><<<nblocks, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <WOp OP>
static cudaError_t launch_op(bool drop, const EngineParams& p, int nblocks, cudaStream_t s) {
  return drop ? launch_one<OP, true>(p, nblocks, s) : launch_one<OP, false>(p, nblocks, s);
}

cudaError_t launch_wide(WOp op, bool drop, const EngineParams& p, int nblocks, cudaStream_t s) {
  switch (op) {
    case WOp::Fwd: return launch_op<WOp::Fwd>(drop, p, nblocks, s);
    case WOp::Stats: return launch_op<WOp::Stats>(drop, p, nblocks, s);
    case WOp::DOut: return launch_op<WOp::DOut>(drop, p, nblocks, s);
    case WOp::DQ: return launch_op<WOp::DQ>(drop, p, nblocks, s);
    case WOp::BwdDQ: return launch_op<WOp::BwdDQ>(drop, p, nblocks, s);
    case WOp::P2V: return launch_op<WOp::P2V>(drop, p, nblocks, s);
    case WOp::P2K: return launch_op<WOp::P2K>(drop, p, nblocks, s);
    case WOp::BwdDV: return launch_op<WOp::BwdDV>(drop, p, nblocks, s);
    case WOp::BwdDK: return launch_op<WOp::BwdDK>(drop, p, nblocks, s);
    case WOp::StatsDO: return launch_op<WOp::StatsDO>(drop, p, nblocks, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t take_wide_error(uint32_t* word, cudaStream_t s) {
  uint32_t zero = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(word, g_fbob_error_word, sizeof(uint32_t), 0,
                                            cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && *word)
    e = cudaMemcpyToSymbolAsync(g_fbob_error_word, &zero, sizeof(uint32_t), 0,
                                cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  return e;
}

}  // namespace fbob
