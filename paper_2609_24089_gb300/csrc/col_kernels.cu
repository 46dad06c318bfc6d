// col_kernels.cu -- instantiations and launcher of the column-block engine:
// first-backward dK and dV (eqs. 2-3), BoB Pass 2 (Algorithm 2, second
// loop).
#include "attn_engine.cuh"
#include "launch.h"

namespace fbob {

template <ColOp OP, int D>
static cudaError_t launch_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(ColCfg<OP, D>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(col_engine<OP, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  col_engine<OP, D><<<nblocks, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_col(ColOp op, int d, const EngineParams& p, int nblocks, cudaStream_t s) {
  switch (op) {
    case ColOp::BwdDKDV:
      return d == 64 ? launch_one<ColOp::BwdDKDV, 64>(p, nblocks, s)
                     : launch_one<ColOp::BwdDKDV, 128>(p, nblocks, s);
    case ColOp::BobPass2:
      return d == 64 ? launch_one<ColOp::BobPass2, 64>(p, nblocks, s)
                     : launch_one<ColOp::BobPass2, 128>(p, nblocks, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t take_col_error(uint32_t* word, cudaStream_t s) {
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
