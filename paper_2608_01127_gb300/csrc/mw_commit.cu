// Rolling KV cache commit (Sec. 3.5, structured rolling KV cache): a
// finished chunk's keys and values are written once into the FIFO ring at
// physical rows (slot + r) mod cap and never modified afterwards.
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {
namespace {

// One thread per 16-byte piece of a row; both K and V.
template <int D>
__global__ void __launch_bounds__(256) commit_kernel(__nv_bfloat16* __restrict__ kc,
                                                     __nv_bfloat16* __restrict__ vc,
                                                     const __nv_bfloat16* __restrict__ ks,
                                                     const __nv_bfloat16* __restrict__ vs, int cap,
                                                     int slot, int rows, int BH) {
  constexpr int PIECES = D / 8;  // 16-byte pieces per row
  // grid: x covers rows * PIECES of one head, y strides over the heads
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * PIECES) return;
  const int piece = idx % PIECES;
  const int r = idx / PIECES;
  int dst = slot + r;
  if (dst >= cap) dst -= cap;  // slot < cap and rows <= cap
  for (int bh = blockIdx.y; bh < BH; bh += gridDim.y) {
    const size_t so = (static_cast<size_t>(bh) * rows + r) * D + piece * 8;
    const size_t dso = (static_cast<size_t>(bh) * cap + dst) * D + piece * 8;
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
  if (d == 64)
    commit_kernel<64><<<grid, 256, 0, s>>>(kc, vc, ks, vs, cap, slot, rows, BH);
  else
    commit_kernel<128><<<grid, 256, 0, s>>>(kc, vc, ks, vs, cap, slot, rows, BH);
  return cudaGetLastError();
}

}  // namespace mw
