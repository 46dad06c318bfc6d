// row_kernels.cu -- instantiations and launcher of the row-block engine:
// forward (eq. 1), first-backward dQ (eqs. 2-3), BoB Pass 1 (Algorithm 2,
// first loop): one sweep at d = 64, row statistics + direct form at d = 128.
#include "attn_engine.cuh"
#include "launch.h"

namespace fbob {

template <RowOp OP, int D>
static cudaError_t launch_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(RowCfg<OP, D>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(row_engine<OP, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  row_engine<OP, D><<<nblocks, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_row(RowOp op, int d, const EngineParams& p, int nblocks, cudaStream_t s) {
  switch (op) {
    case RowOp::Fwd:
      return d == 64 ? launch_one<RowOp::Fwd, 64>(p, nblocks, s)
                     : launch_one<RowOp::Fwd, 128>(p, nblocks, s);
    case RowOp::BwdDQ:
      return d == 64 ? launch_one<RowOp::BwdDQ, 64>(p, nblocks, s)
                     : launch_one<RowOp::BwdDQ, 128>(p, nblocks, s);
    case RowOp::BobPass1:  // the one-sweep form serves d = 64 only
      return d == 64 ? launch_one<RowOp::BobPass1, 64>(p, nblocks, s) : cudaErrorInvalidValue;
    case RowOp::BobStats:
      return d == 64 ? launch_one<RowOp::BobStats, 64>(p, nblocks, s)
                     : launch_one<RowOp::BobStats, 128>(p, nblocks, s);
    case RowOp::BobPass1D:
      return d == 64 ? launch_one<RowOp::BobPass1D, 64>(p, nblocks, s)
                     : launch_one<RowOp::BobPass1D, 128>(p, nblocks, s);
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
