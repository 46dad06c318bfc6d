// row_kernels.cu -- instantiations and launcher of the row-block engine:
// forward (eq. 1), first-backward dQ (eqs. 2-3), BoB Pass 1 (Algorithm 2,
// first loop): one sweep at d = 64, row statistics + direct form at d = 128
// (and at d = 64 with dropout).  Each operation with and without dropout.
#include "attn_engine.cuh"
#include "launch.h"

namespace fbob {

template <RowOp OP, int D, bool DROP>
static cudaError_t launch_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(RowCfg<OP, D>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(row_engine<OP, D, DROP>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  row_engine<OP, D, DROP><<<nblocks, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <RowOp OP>
static cudaError_t launch_op(int d, bool drop, const EngineParams& p, int nblocks, cudaStream_t s) {
  if (d == 64)
    return drop ? launch_one<OP, 64, true>(p, nblocks, s) : launch_one<OP, 64, false>(p, nblocks, s);
  return drop ? launch_one<OP, 128, true>(p, nblocks, s) : launch_one<OP, 128, false>(p, nblocks, s);
}

cudaError_t launch_row(RowOp op, int d, bool drop, const EngineParams& p, int nblocks,
                       cudaStream_t s) {
  switch (op) {
    case RowOp::Fwd: return launch_op<RowOp::Fwd>(d, drop, p, nblocks, s);
    case RowOp::BwdDQ: return launch_op<RowOp::BwdDQ>(d, drop, p, nblocks, s);
    case RowOp::BobPass1:  // the one-sweep form serves d = 64 without dropout only
      return d == 64 && !drop ? launch_one<RowOp::BobPass1, 64, false>(p, nblocks, s)
                              : cudaErrorInvalidValue;
    case RowOp::BobStats: return launch_op<RowOp::BobStats>(d, drop, p, nblocks, s);
    case RowOp::BobPass1D: return launch_op<RowOp::BobPass1D>(d, drop, p, nblocks, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t take_row_error(uint32_t* word, cudaStream_t s) {
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
