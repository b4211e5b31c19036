// QKV split with the temporal rotary embedding applied on the way (the input
// side of block-causal attention, Sec. 3.2; RoPE positions as in Sec. 3.5).
// The fused QKV projection leaves each token's heads interleaved as
// [B, N, 3, H, d]; the attention kernels read head-major [B, H, N, d] rows.
// One pass moves every element once and rotates the first rope_dims channels
// of Q and K: token t sits at frame first_frame + t / per_frame, and channel
// pair (2i, 2i+1) turns by frame * base^(-2i / rope_dims).  HBM-bound: each
// element is read and written once, 16 bytes per thread access.
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {
namespace {

constexpr int kQkvTokens = 32;  // tokens per CTA
constexpr int kMaxPairs = kMaxRopePairs;
constexpr int kUnroll = 4;      // heads whose 16-byte pieces are in flight at once

// grid.x: (b, block of kQkvTokens tokens); grid.y: groups of heads_per_block
// heads.  A thread owns one (token, 16-byte piece) of the block, fixed for
// the whole kernel, and walks Q, K, V and the group's heads with plain
// strides; each warp reads whole 128-byte row segments and writes 512
// contiguous bytes.
__global__ void __launch_bounds__(256) qkv_rope_kernel(const __nv_bfloat16* __restrict__ qkv,
                                                       __nv_bfloat16* __restrict__ q,
                                                       __nv_bfloat16* __restrict__ k,
                                                       __nv_bfloat16* __restrict__ v, int N, int H,
                                                       int d, int rope_dims, int heads_per_block,
                                                       const RopeFreq omega, int per_frame,
                                                       int first_frame) {
  __shared__ float2 table[kQkvTokens * kMaxPairs];  // (cos, sin) per (frame, pair)
  const int n_tb = (N + kQkvTokens - 1) / kQkvTokens;
  const int b = blockIdx.x / n_tb;
  const int t0 = (blockIdx.x % n_tb) * kQkvTokens;
  const int nt = min(kQkvTokens, N - t0);
  const int h0 = blockIdx.y * heads_per_block;
  const int h1 = min(H, h0 + heads_per_block);
  const int pairs = rope_dims / 2;
  const int f_lo = first_frame + t0 / per_frame;
  if (pairs > 0) {
    // frames of this token block: at most one per token
    const int nf = first_frame + (t0 + nt - 1) / per_frame - f_lo + 1;
    for (int e = threadIdx.x; e < nf * pairs; e += blockDim.x)
      table[e] = rope_cos_sin(f_lo + e / pairs, omega.hi[e % pairs], omega.lo[e % pairs]);
    __syncthreads();
  }
  const int pieces = d / 8;
  const int rot_pieces = (pairs + 3) / 4;  // pieces holding at least one rotated pair
  const size_t head_out = static_cast<size_t>(N) * d;  // output elements per head
  for (int r = threadIdx.x; r < nt * pieces; r += blockDim.x) {
    const int t = t0 + r / pieces;
    const int pc = r % pieces;
    // the piece's (cos, sin) pairs: index 4 pc + u < pairs turns
    const int np = pc < rot_pieces ? min(4, pairs - 4 * pc) : 0;
    float2 cs[4];
    if (np > 0) {
      const float2* row = table + (first_frame + t / per_frame - f_lo) * pairs + 4 * pc;
#pragma unroll
      for (int u = 0; u < 4; ++u) cs[u] = u < np ? row[u] : make_float2(1.f, 0.f);
    }
    const __nv_bfloat16* src = qkv + (static_cast<size_t>(b) * N + t) * 3 * H * d + pc * 8;
    const size_t dst0 = (static_cast<size_t>(b) * H * N + t) * d + pc * 8;
    for (int which = 0; which < 3; ++which) {
      __nv_bfloat16* out = which == 0 ? q : which == 1 ? k : v;
      const bool turn = which < 2 && np > 0;
      for (int h = h0; h < h1; h += kUnroll) {
        uint4 x[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
          if (h + u < h1)
            x[u] = *reinterpret_cast<const uint4*>(src + static_cast<size_t>(which * H + h + u) * d);
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          if (h + u >= h1) continue;
          if (turn) {
            x[u].x = rope_turn(x[u].x, cs[0]);
            if (np > 1) x[u].y = rope_turn(x[u].y, cs[1]);
            if (np > 2) x[u].z = rope_turn(x[u].z, cs[2]);
            if (np > 3) x[u].w = rope_turn(x[u].w, cs[3]);
          }
          *reinterpret_cast<uint4*>(out + dst0 + (h + u) * head_out) = x[u];
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_qkv_rope(const __nv_bfloat16* qkv, __nv_bfloat16* q, __nv_bfloat16* k,
                            __nv_bfloat16* v, int B, int N, int H, int d, int rope_dims,
                            const RopeFreq& omega, int per_frame, int first_frame,
                            cudaStream_t s) {
  if (B == 0 || N == 0 || H == 0) return cudaSuccess;
  const long long tb = static_cast<long long>(B) * ((N + kQkvTokens - 1) / kQkvTokens);
  // halve the heads per CTA until the grid holds enough CTAs to fill every SM
  // a few times over (the per-CTA (cos, sin) table is then amortised over as
  // many heads as the size allows)
  int hb = H;
  while (hb > 1 && tb * ((H + hb - 1) / hb) < 1216) hb = (hb + 1) / 2;
  const dim3 grid(static_cast<unsigned>(tb), static_cast<unsigned>((H + hb - 1) / hb));
  qkv_rope_kernel<<<grid, 256, 0, s>>>(qkv, q, k, v, N, H, d, rope_dims, hb, omega, per_frame,
                                       first_frame);
  return cudaGetLastError();
}

}  // namespace mw
