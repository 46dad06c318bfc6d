// row_kernels.cu -- instantiations and launcher of the row-block kernels:
// forward (eq. 1, fwd_engine.cuh), first-backward dQ (eqs. 2-3), BoB Pass 1 (Algorithm 2,
// first loop): one sweep with the affine fusion (at d = 128 over two CTAs per
// row block), or row statistics + direct form.  Each operation with and without dropout, for
// head dims 32 (in 64-wide tiles), 64 and 128.
#include "attn_engine.cuh"
#include "fwd_engine.cuh"
#include "launch.h"

namespace fbob {

// D: tile head dimension; DG: the tensors' head dimension (32 runs in 64-wide tiles)
template <RowOp OP, int D, bool DROP, int DG = D>
static cudaError_t launch_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(RowCfg<OP, D>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(row_engine<OP, D, DROP, DG>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  row_engine<OP, D, DROP, DG><<<nblocks, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <RowOp OP, bool DROP>
static cudaError_t launch_d(int d, const EngineParams& p, int nblocks, cudaStream_t s) {
  switch (d) {
    case 32: return launch_one<OP, 64, DROP, 32>(p, nblocks, s);
    case 64: return launch_one<OP, 64, DROP>(p, nblocks, s);
    case 128: return launch_one<OP, 128, DROP>(p, nblocks, s);
  }
  return cudaErrorInvalidValue;
}

template <RowOp OP>
static cudaError_t launch_op(int d, bool drop, const EngineParams& p, int nblocks, cudaStream_t s) {
  return drop ? launch_d<OP, true>(d, p, nblocks, s) : launch_d<OP, false>(d, p, nblocks, s);
}

// the forward: two query tiles per CTA (fwd_engine.cuh)
template <int D, bool DROP, int DG = D>
static cudaError_t launch_fwd_one(const EngineParams& p, int nblocks, cudaStream_t s) {
  const int smem = launch_smem(FwdCfg<D>::SMEM_BYTES);
  cudaError_t e = cudaFuncSetAttribute(fwd_engine<D, DROP, DG>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  fwd_engine<D, DROP, DG><<<nblocks, kFwdThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <bool DROP>
static cudaError_t launch_fwd(int d, const EngineParams& p, int nblocks, cudaStream_t s) {
  switch (d) {
    case 32: return launch_fwd_one<64, DROP, 32>(p, nblocks, s);
    case 64: return launch_fwd_one<64, DROP>(p, nblocks, s);
    case 128: return launch_fwd_one<128, DROP>(p, nblocks, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_row(RowOp op, int d, bool drop, const EngineParams& p, int nblocks,
                       cudaStream_t s) {
  switch (op) {
    case RowOp::Fwd:
      return drop ? launch_fwd<true>(d, p, nblocks, s) : launch_fwd<false>(d, p, nblocks, s);
    case RowOp::BwdDQ: return launch_op<RowOp::BwdDQ>(d, drop, p, nblocks, s);
    case RowOp::BobPass1:  // the one-sweep form (no dropout); at d = 128 nblocks
                           // counts both CTAs of each row block
      if (drop) return cudaErrorInvalidValue;
      return d == 64    ? launch_one<RowOp::BobPass1, 64, false>(p, nblocks, s)
             : d == 32  ? launch_one<RowOp::BobPass1, 64, false, 32>(p, nblocks, s)
             : d == 128 ? launch_one<RowOp::BobPass1, 128, false>(p, nblocks, s)
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
