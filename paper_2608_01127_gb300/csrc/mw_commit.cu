// Rolling KV cache commit (Sec. 3.5, structured rolling KV cache): a
// finished chunk's keys and values are written once into the FIFO ring at
// physical rows (slot + r) mod cap and never modified afterwards.
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {

int g_pdl_enabled = 1;

namespace {

// One thread per 16-byte piece of a row (d / 8 pieces, d a multiple of 8);
// both K and V.  grid: x covers rows * pieces of one head, y strides over
// the heads.
__global__ void __launch_bounds__(256) commit_kernel(const CommitJob j) {
  pdl_wait();  // the forward that read the ring has completed
  pdl_trigger();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= j.rows * (j.d / 8)) return;
  for (int bh = blockIdx.y; bh < j.BH; bh += gridDim.y) commit_piece(j, bh, idx);
}

}  // namespace

cudaError_t launch_commit(const CommitJob& j, cudaStream_t s) {
  const int per_head = j.rows * (j.d / 8);
  if (per_head == 0 || j.BH == 0) return cudaSuccess;
  const dim3 grid(static_cast<unsigned>((per_head + 255) / 256),
                  static_cast<unsigned>(j.BH < 65535 ? j.BH : 65535));
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr;
  pdl_config(cfg, attr, grid, dim3(256), 0, s);
  return cudaLaunchKernelEx(&cfg, commit_kernel, j);
}

}  // namespace mw
