// col_kernels.cu -- instantiations and launcher of the column-block engine:
// first-backward dK and dV (eqs. 2-3), BoB Pass 2 (Algorithm 2, second
// loop).  Each operation with and without dropout, for head dims 32 (in
// 64-wide tiles), 64 and 128.
#include "attn_engine.cuh"
#include "launch.h"

namespace fbob {

// D: tile head dimension; DG: the tensors' head dimension (32 runs in 64-wide tiles)
template <ColOp OP, int D, bool DROP, int DG = D>
static cudaError_t launch_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(ColCfg<OP, D>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(col_engine<OP, D, DROP, DG>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  col_engine<OP, D, DROP, DG><<<nblocks, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <ColOp OP, bool DROP>
static cudaError_t launch_d(int d, const EngineParams& p, int nblocks, cudaStream_t s) {
  switch (d) {
    case 32: return launch_one<OP, 64, DROP, 32>(p, nblocks, s);
    case 64: return launch_one<OP, 64, DROP>(p, nblocks, s);
    case 128: return launch_one<OP, 128, DROP>(p, nblocks, s);
  }
  return cudaErrorInvalidValue;
}

template <ColOp OP>
static cudaError_t launch_op(int d, bool drop, const EngineParams& p, int nblocks, cudaStream_t s) {
  return drop ? launch_d<OP, true>(d, p, nblocks, s) : launch_d<OP, false>(d, p, nblocks, s);
}

cudaError_t launch_col(ColOp op, int d, bool drop, const EngineParams& p, int nblocks,
                       cudaStream_t s) {
  switch (op) {
    case ColOp::BwdDKDV: return launch_op<ColOp::BwdDKDV>(d, drop, p, nblocks, s);
    case ColOp::BobPass2: return launch_op<ColOp::BobPass2>(d, drop, p, nblocks, s);
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
