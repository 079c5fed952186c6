// Decode attention kernels for binary16 metadata pairs (the 32-bit metadata
// storage model of Sec. 5.4), compiled apart from the fp32-pair set.
#include "hg_decode_kernel.cuh"

namespace hg {

cudaError_t launch_decode_m16(const DecodeParams& p, int grid_x, cudaStream_t s) {
  return launch_decode_mb<4>(p, grid_x, s);
}

}  // namespace hg
