// Host side of the decode attention kernel (templates in hg_decode_kernel.cuh):
// the merge's split limit, the check of the bounded tile wait, and the launch
// for fp32 metadata pairs (binary16 pairs: hg_decode_m16.cu).
#include "hg_decode_kernel.cuh"

namespace hg {

// The merging CTA stages every split's partial in its stage buffer and keeps
// one weight row per split.
int decode_max_splits(int G) {
  const int n = kBufBytes / (G * kPartialStride * 4);
  return n < kFwL ? n : kFwL;
}

// Check of the bounded wait that every decode tile wait uses: one mbarrier
// whose phase is completed (the wait must succeed: bit 1) and one that nothing
// ever arrives on (the wait must give up after `rounds` suspensions and flag
// kStatusWaitTimeout: bit 0).  Expected result 3.
__global__ void wait_probe_kernel(uint32_t* result, uint32_t rounds) {
  __shared__ __align__(8) uint64_t bars[2];
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  const uint32_t done = smem_u32(&bars[0]), never = smem_u32(&bars[1]);
  mbar_init(done, 1);
  mbar_init(never, 1);
  mbar_init_fence();
  abort_flag = 0;
  mbar_arrive_expect_tx(done, 0);  // completes phase 0 of `done`
  uint32_t r = 0;
  if (wait_tile(done, 0, &abort_flag, result, rounds)) r |= 2u;
  wait_tile(never, 0, &abort_flag, result, rounds);  // sets bit 0 of *result on timeout
  atomicOr(result, r);
}

cudaError_t launch_wait_probe(uint32_t* result, uint32_t rounds, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(result, rounds);
  return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeParams& p, int grid_x, cudaStream_t s) {
  return p.d.meta16 ? launch_decode_m16(p, grid_x, s) : launch_decode_mb<8>(p, grid_x, s);
}

}  // namespace hg
