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
  const size_t idx = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const size_t total = static_cast<size_t>(BH) * rows * PIECES;
  if (idx >= total) return;
  const int piece = static_cast<int>(idx % PIECES);
  const size_t src_row = idx / PIECES;  // over BH * rows
  const size_t bh = src_row / rows;
  const int r = static_cast<int>(src_row % rows);
  const int dst = (slot + r) % cap;
  const size_t so = src_row * D + piece * 8;
  const size_t dso = (bh * cap + dst) * D + piece * 8;
  *reinterpret_cast<uint4*>(kc + dso) = *reinterpret_cast<const uint4*>(ks + so);
  *reinterpret_cast<uint4*>(vc + dso) = *reinterpret_cast<const uint4*>(vs + so);
}

}  // namespace

cudaError_t launch_commit(int d, __nv_bfloat16* kc, __nv_bfloat16* vc, const __nv_bfloat16* ks,
                          const __nv_bfloat16* vs, int cap, int slot, int rows, int BH,
                          cudaStream_t s) {
  const size_t total = static_cast<size_t>(BH) * rows * (d / 8);
  if (total == 0) return cudaSuccess;
  const unsigned grid = static_cast<unsigned>((total + 255) / 256);
  if (d == 64)
    commit_kernel<64><<<grid, 256, 0, s>>>(kc, vc, ks, vs, cap, slot, rows, BH);
  else
    commit_kernel<128><<<grid, 256, 0, s>>>(kc, vc, ks, vs, cap, slot, rows, BH);
  return cudaGetLastError();
}

}  // namespace mw
