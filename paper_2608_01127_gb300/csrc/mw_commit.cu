// Rolling KV cache commit (Sec. 3.5, structured rolling KV cache): a
// finished chunk's keys and values are written once into the FIFO ring at
// physical rows (slot + r) mod cap and never modified afterwards.
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {
namespace {

// One thread per 16-byte piece of a row (d / 8 pieces, d a multiple of 8);
// both K and V.
__global__ void __launch_bounds__(256) commit_kernel(__nv_bfloat16* __restrict__ kc,
                                                     __nv_bfloat16* __restrict__ vc,
                                                     const __nv_bfloat16* __restrict__ ks,
                                                     const __nv_bfloat16* __restrict__ vs, int cap,
                                                     int slot, int rows, int BH, int d) {
  const int pieces = d / 8;
  // grid: x covers rows * pieces of one head, y strides over the heads
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * pieces) return;
  const int piece = idx % pieces;
  const int r = idx / pieces;
  int dst = slot + r;
  if (dst >= cap) dst -= cap;  // slot < cap and rows <= cap
  for (int bh = blockIdx.y; bh < BH; bh += gridDim.y) {
    const size_t so = (static_cast<size_t>(bh) * rows + r) * d + piece * 8;
    const size_t dso = (static_cast<size_t>(bh) * cap + dst) * d + piece * 8;
    *reinterpret_cast<uint4*>(kc + dso) = *reinterpret_cast<const uint4*>(ks + so);
    *reinterpret_cast<uint4*>(vc + dso) = *reinterpret_cast<const uint4*>(vs + so);
  }
}

}  // namespace

cudaError_t launch_commit(int d, __nv_bfloat16* kc, __nv_bfloat16* vc, const __nv_bfloat16* ks,
                          const __nv_bfloat16* vs, int cap, int slot, int rows, int BH,
                          cudaStream_t s) {
  const int per_head = rows * (d / 8);
  if (per_head == 0 || BH == 0) return cudaSuccess;
  const dim3 grid(static_cast<unsigned>((per_head + 255) / 256),
                  static_cast<unsigned>(BH < 65535 ? BH : 65535));
  commit_kernel<<<grid, 256, 0, s>>>(kc, vc, ks, vs, cap, slot, rows, BH, d);
  return cudaGetLastError();
}

}  // namespace mw
