// Block-causal attention backward on sm_103a: the analytic gradient of
// softmax attention restricted to the chunk-causal mask of Sec. 3.2
// (training is bf16 mixed precision, Sec. 4.1).
//
//   pre : D_i = <dO_i, O_i>, LSE2_i = LSE_i * log2(e) (+inf on padding rows),
//         dQacc = 0
//   main: one CTA per 128-row key tile of one (b,h); it owns dK, dV in TMEM
//         and visits only the query tiles whose chunks can see it
//         (queries i >= chunk(k0) * T).  Per query tile:
//           S^T  = K Q^T              (tcgen05, TMEM)
//           dP^T = V dO^T             (tcgen05, TMEM)
//           P^T  = exp2(S^T scale log2e - LSE2)       -> TMEM (bf16)
//           dS^T = P^T (dP^T - D)                     -> shared memory (bf16)
//           dV  += P^T dO ;  dK += dS^T Q ;  dQ_tile = dS K  (tcgen05)
//           dQacc += dQ_tile (fp32 vector atomics)
//   post: dQ = scale * dQacc -> bf16
//
// Roles (320 threads): warps 0-3 P/dS (one thread per key row), warps 4-7
// dQ drain (one thread per query row), warp 8 TMA producer, warp 9 MMA.
// TMEM: dV [0, D), dK [D, 2D), S^T [2D, 2D+128), dP^T / dQ_tile [2D+128, 2D+256).
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {
namespace {

template <int D>
struct BwdLayout {
  static constexpr int REG = D / 64;
  static constexpr int REGION_BYTES = kTileRows * 128;
  static constexpr int TILE_BYTES = REG * REGION_BYTES;
  static constexpr int QSTAGES = 2;
  static constexpr int VEC_BYTES = kTileRows * 4;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + TILE_BYTES;
  static constexpr int OFF_Q = OFF_V + TILE_BYTES;                 // QSTAGES tiles
  static constexpr int OFF_DO = OFF_Q + QSTAGES * TILE_BYTES;      // QSTAGES tiles
  static constexpr int OFF_DS = OFF_DO + QSTAGES * TILE_BYTES;     // 128 x 128 bf16
  static constexpr int DS_BYTES = 2 * REGION_BYTES;
  static constexpr int OFF_LSE = OFF_DS + DS_BYTES;                // QSTAGES x 512 B
  static constexpr int OFF_DELTA = OFF_LSE + QSTAGES * VEC_BYTES;  // QSTAGES x 512 B
  static constexpr int OFF_BAR = OFF_DELTA + QSTAGES * VEC_BYTES;
  // kv_full, q_full[2], q_empty[2], st_full, dpt_full, p_ready, dq_full, dq_free, ds_free, dkv_full
  static constexpr int NBAR = 1 + 2 * QSTAGES + 7;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int BYTES = OFF_MISC + 16;
  static constexpr uint32_t DV_COL = 0;
  static constexpr uint32_t DK_COL = D;
  static constexpr uint32_t S_COL = 2 * D;
  static constexpr uint32_t DP_COL = 2 * D + 128;
  static constexpr int THREADS = 320;
};

__device__ __forceinline__ void red_add_v4(float* addr, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(addr), "f"(a), "f"(b),
               "f"(c), "f"(d)
               : "memory");
}

template <int D>
__global__ void __launch_bounds__(BwdLayout<D>::THREADS, 1)
    bca_bwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
                   const BwdParams p) {
  using L = BwdLayout<D>;
  constexpr int NS = L::QSTAGES;
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0u) {
    if (threadIdx.x == 0) atomicOr(p.status, kDevMisaligned);
    return;  // uniform across the CTA, before any barrier or TMEM use
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
  uint64_t* kv_full = bars;
  uint64_t* q_full = bars + 1;
  uint64_t* q_empty = q_full + NS;
  uint64_t* st_full = q_empty + NS;
  uint64_t* dpt_full = st_full + 1;
  uint64_t* p_ready = dpt_full + 1;
  uint64_t* dq_full = p_ready + 1;
  uint64_t* dq_free = dq_full + 1;
  uint64_t* ds_free = dq_free + 1;
  uint64_t* dkv_full = ds_free + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- work item: key tiles near the start see the most queries; go first
  const int bh = blockIdx.x % p.BH;
  const int kt = blockIdx.x / p.BH;
  const int k0 = kt * kTileRows;
  const int first_q = (k0 / p.T) * p.T;  // first query that sees key k0
  const int m_begin = first_q / kTileRows;
  const int m_end = p.N_pad / kTileRows;
  const int n_q = m_end - m_begin;

  if (threadIdx.x == 0) {
    mbar_init(kv_full, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&q_full[s], 1);
      mbar_init(&q_empty[s], 1);
    }
    mbar_init(st_full, 1);
    mbar_init(dpt_full, 1);
    mbar_init(p_ready, 4);
    mbar_init(dq_full, 1);
    mbar_init(dq_free, 4);
    mbar_init(ds_free, 1);
    mbar_init(dkv_full, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 9) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.status, p.budget_ns};

  uint8_t* sK = smem + L::OFF_K;
  uint8_t* sV = smem + L::OFF_V;
  uint8_t* sQ = smem + L::OFF_Q;
  uint8_t* sDO = smem + L::OFF_DO;
  uint8_t* sDS = smem + L::OFF_DS;
  float* sLSE = reinterpret_cast<float*>(smem + L::OFF_LSE);
  float* sDelta = reinterpret_cast<float*>(smem + L::OFF_DELTA);

  if (warp == 8) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_do);
      mbar_arrive_expect_tx(kv_full, 2 * L::TILE_BYTES);
      for (int r = 0; r < L::REG; ++r) {
        tma_load_3d(sK + r * L::REGION_BYTES, &tm_k, kv_full, 64 * r, k0, bh);
        tma_load_3d(sV + r * L::REGION_BYTES, &tm_v, kv_full, 64 * r, k0, bh);
      }
      int issued = 0;
      for (int i = 0; i < n_q; ++i) {
        const int st = i % NS;
        const uint32_t ph = (i / NS) & 1;
        const int q0 = (m_begin + i) * kTileRows;
        if (!mbar_wait(&q_empty[st], ph ^ 1, ctl)) break;
        mbar_arrive_expect_tx(&q_full[st], 2 * L::TILE_BYTES + 2 * L::VEC_BYTES);
        for (int r = 0; r < L::REG; ++r) {
          tma_load_3d(sQ + st * L::TILE_BYTES + r * L::REGION_BYTES, &tm_q, &q_full[st], 64 * r, q0, bh);
          tma_load_3d(sDO + st * L::TILE_BYTES + r * L::REGION_BYTES, &tm_do, &q_full[st], 64 * r, q0, bh);
        }
        const size_t voff = static_cast<size_t>(bh) * p.N_pad + q0;
        bulk_load(sLSE + st * kTileRows, p.lse2 + voff, L::VEC_BYTES, &q_full[st]);
        bulk_load(sDelta + st * kTileRows, p.delta + voff, L::VEC_BYTES, &q_full[st]);
        ++issued;
      }
      if (*abort_flag) {
        drain_wait(kv_full, 0, p.budget_ns);
        for (int i = max(0, issued - NS); i < issued; ++i)
          drain_wait(&q_full[i % NS], (i / NS) & 1, p.budget_ns);
      }
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_ss = idesc_bf16_f32(128, 128, false, false);   // S^T, dP^T
      constexpr uint32_t idesc_dv = idesc_bf16_f32(128, D, false, true);      // P^T dO
      constexpr uint32_t idesc_dk = idesc_bf16_f32(128, D, false, true);      // dS^T Q
      constexpr uint32_t idesc_dq = idesc_bf16_f32(128, D, true, true);       // dS K
      const uint32_t kb = smem_u32(sK), vb = smem_u32(sV), dsb = smem_u32(sDS);
      bool ok = mbar_wait(kv_full, 0, ctl);
      tc_fence_after();
      for (int i = 0; ok && i < n_q; ++i) {
        const int st = i % NS;
        const uint32_t ph = (i / NS) & 1;
        const uint32_t qb = smem_u32(sQ + st * L::TILE_BYTES);
        const uint32_t dob = smem_u32(sDO + st * L::TILE_BYTES);
        if (!(ok = mbar_wait(&q_full[st], ph, ctl))) break;
        tc_fence_after();
        // S^T = K Q^T
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::REGION_BYTES + (kk & 3) * 32;
          umma_ss(tmem + L::S_COL, sdesc_sw128(kb + off, 16, 1024), sdesc_sw128(qb + off, 16, 1024),
                  idesc_ss, kk > 0 ? 1u : 0u);
        }
        umma_commit(st_full);
        // dP^T = V dO^T (its TMEM columns held dQ of the previous tile)
        if (i > 0) {
          if (!(ok = mbar_wait(dq_free, (i - 1) & 1, ctl))) break;
          tc_fence_after();
        }
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::REGION_BYTES + (kk & 3) * 32;
          umma_ss(tmem + L::DP_COL, sdesc_sw128(vb + off, 16, 1024), sdesc_sw128(dob + off, 16, 1024),
                  idesc_ss, kk > 0 ? 1u : 0u);
        }
        umma_commit(dpt_full);
        if (!(ok = mbar_wait(p_ready, i & 1, ctl))) break;
        tc_fence_after();
        // dV += P^T dO   (P^T bf16 in TMEM over the S^T columns)
#pragma unroll
        for (int kk = 0; kk < kTileRows / 16; ++kk)
          umma_ts(tmem + L::DV_COL, tmem + L::S_COL + kk * 8,
                  sdesc_sw128(dob + kk * 2048, L::REGION_BYTES, 1024), idesc_dv,
                  (i > 0 || kk > 0) ? 1u : 0u);
        // dK += dS^T Q
#pragma unroll
        for (int kk = 0; kk < kTileRows / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::REGION_BYTES + (kk & 3) * 32;
          umma_ss(tmem + L::DK_COL, sdesc_sw128(dsb + off, 16, 1024),
                  sdesc_sw128(qb + kk * 2048, L::REGION_BYTES, 1024), idesc_dk,
                  (i > 0 || kk > 0) ? 1u : 0u);
        }
        // dQ_tile = dS K
#pragma unroll
        for (int kk = 0; kk < kTileRows / 16; ++kk)
          umma_ss(tmem + L::DP_COL, sdesc_sw128(dsb + kk * 2048, L::REGION_BYTES, 1024),
                  sdesc_sw128(kb + kk * 2048, L::REGION_BYTES, 1024), idesc_dq, kk > 0 ? 1u : 0u);
        umma_commit(dq_full);
        umma_commit(&q_empty[st]);
        umma_commit(ds_free);
      }
      if (ok) umma_commit(dkv_full);
    }
  } else if (warp < 4) {
    // ------------------------------------------------------------ P / dS (thread = key row)
    const int j_local = warp * 32 + lane;
    const int j = k0 + j_local;
    const bool j_valid = j < p.N;
    const int q_start = j_valid ? (j / p.T) * p.T : 0x7fffffff;  // first query seeing key j
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    const float sl2 = p.scale_log2;
    // dS^T row j_local, swizzled like a TMA 128-byte tile (two 64-column regions)
    uint8_t* ds_row = sDS + j_local * 128;
    const int sw = j_local & 7;
    bool ok = true;
    for (int i = 0; i < n_q; ++i) {
      const int st = i % NS;
      const int q0 = (m_begin + i) * kTileRows;
      const float* lse2 = sLSE + st * kTileRows;
      const float* delta = sDelta + st * kTileRows;
      if (!(ok = warp_wait(st_full, i & 1, ctl))) break;
      tc_fence_after();
      const int lim = q_start - q0;  // columns c < lim are masked
      float pr[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t r[32];
        tmem_ld32(lane_base + L::S_COL + 32 * c, r);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const int col = 32 * c + k;
          const float e = ex2_approx(fmaf(__uint_as_float(r[k]), sl2, -lse2[col]));
          pr[col] = (col < lim) ? 0.f : e;
        }
      }
      // P^T -> TMEM (bf16 pairs) for the dV MMA
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t packed[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) packed[k] = pack_bf16x2(pr[64 * h + 2 * k], pr[64 * h + 2 * k + 1]);
        tmem_st32(lane_base + L::S_COL + 32 * h, packed);
      }
      if (!(ok = warp_wait(dpt_full, i & 1, ctl))) break;
      tc_fence_after();
      if (i > 0 && !(ok = warp_wait(ds_free, (i - 1) & 1, ctl))) break;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t r[32];
        tmem_ld32(lane_base + L::DP_COL + 32 * c, r);
        tmem_wait_ld();
        uint32_t packed[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const int col = 32 * c + 2 * k;
          const float d0 = pr[col] * (__uint_as_float(r[2 * k]) - delta[col]);
          const float d1 = pr[col + 1] * (__uint_as_float(r[2 * k + 1]) - delta[col + 1]);
          packed[k] = pack_bf16x2(d0, d1);
        }
        // columns [32c, 32c+32) = region c/2, 16-byte chunks 4*(c&1) .. +3
        uint8_t* region = ds_row + (c >> 1) * L::REGION_BYTES;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int chunk = 4 * (c & 1) + q;
          *reinterpret_cast<uint4*>(region + ((chunk ^ sw) << 4)) =
              make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
        }
      }
      fence_proxy_async_smem();
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_ready);
    }
    // ---- epilogue: dK (x scale) and dV of this key tile
    const bool have = ok && warp_wait(dkv_full, 0, ctl);
    tc_fence_after();
    if (have) {
      const size_t row_off = (static_cast<size_t>(bh) * p.N + j) * D;
#pragma unroll
      for (int which = 0; which < 2; ++which) {
        const uint32_t col0 = which == 0 ? L::DK_COL : L::DV_COL;
        const float mul = which == 0 ? p.scale : 1.f;
        __nv_bfloat16* out = which == 0 ? p.dk : p.dv;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(lane_base + col0 + 32 * c, r);
          tmem_wait_ld();
          if (j_valid) {
            uint4* dst = reinterpret_cast<uint4*>(out + row_off + 32 * c);
#pragma unroll
            for (int k = 0; k < 4; ++k)
              dst[k] = make_uint4(pack_bf16x2(__uint_as_float(r[8 * k]) * mul, __uint_as_float(r[8 * k + 1]) * mul),
                                  pack_bf16x2(__uint_as_float(r[8 * k + 2]) * mul, __uint_as_float(r[8 * k + 3]) * mul),
                                  pack_bf16x2(__uint_as_float(r[8 * k + 4]) * mul, __uint_as_float(r[8 * k + 5]) * mul),
                                  pack_bf16x2(__uint_as_float(r[8 * k + 6]) * mul, __uint_as_float(r[8 * k + 7]) * mul));
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------ dQ drain (thread = query row)
    const int wq = warp & 3;
    const int row_local = wq * 32 + lane;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    for (int i = 0; i < n_q; ++i) {
      const int q0 = (m_begin + i) * kTileRows;
      if (!warp_wait(dq_full, i & 1, ctl)) break;
      tc_fence_after();
      float* dst = p.dq_acc + (static_cast<size_t>(bh) * p.N_pad + q0 + row_local) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(lane_base + L::DP_COL + 32 * c, r);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 8; ++k)
          red_add_v4(dst + 32 * c + 4 * k, __uint_as_float(r[4 * k]), __uint_as_float(r[4 * k + 1]),
                     __uint_as_float(r[4 * k + 2]), __uint_as_float(r[4 * k + 3]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(dq_free);
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// D_i = <dO_i, O_i>, LSE2_i = LSE_i log2(e) for i < N; padding rows get
// D = 0, LSE2 = +inf (so their P is exactly 0).  Also zeroes dQacc.
template <int D>
__global__ void __launch_bounds__(256) bwd_pre_kernel(const __nv_bfloat16* __restrict__ o,
                                                      const __nv_bfloat16* __restrict__ dout,
                                                      const float* __restrict__ lse,
                                                      float* __restrict__ lse2,
                                                      float* __restrict__ delta,
                                                      float* __restrict__ dq_acc, int BH, int N,
                                                      int N_pad) {
  const int gw = blockIdx.x * 8 + (threadIdx.x >> 5);  // one warp per padded row
  const int lane = threadIdx.x & 31;
  if (gw >= BH * N_pad) return;
  const int bh = gw / N_pad;
  const int i = gw % N_pad;
  constexpr int PER = D / 32;
  float4* acc = reinterpret_cast<float4*>(dq_acc + static_cast<size_t>(gw) * D);
  for (int k = lane; k < D / 4; k += 32) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
  float sum = 0.f;
  if (i < N) {
    const size_t off = (static_cast<size_t>(bh) * N + i) * D + lane * PER;
#pragma unroll
    for (int k = 0; k < PER; ++k) sum += __bfloat162float(o[off + k]) * __bfloat162float(dout[off + k]);
  }
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
  if (lane == 0) {
    delta[gw] = sum;
    lse2[gw] = (i < N) ? lse[static_cast<size_t>(bh) * N + i] * 1.4426950408889634f : INFINITY;
  }
}

template <int D>
__global__ void __launch_bounds__(256) bwd_post_kernel(const float* __restrict__ dq_acc,
                                                       __nv_bfloat16* __restrict__ dq, float scale,
                                                       int BH, int N, int N_pad) {
  const size_t idx = (static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x);  // 4 elements
  const size_t total = static_cast<size_t>(BH) * N * D / 4;
  if (idx >= total) return;
  const size_t e = idx * 4;
  const size_t row = e / D;  // over BH * N
  const int c = static_cast<int>(e % D);
  const size_t bh = row / N;
  const size_t i = row % N;
  const float4 v = *reinterpret_cast<const float4*>(dq_acc + (bh * N_pad + i) * D + c);
  uint2 out;
  out.x = pack_bf16x2(v.x * scale, v.y * scale);
  out.y = pack_bf16x2(v.z * scale, v.w * scale);
  *reinterpret_cast<uint2*>(dq + e) = out;
}

template <int D>
cudaError_t launch_bwd_main_t(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                              const CUtensorMap& tdo, const BwdParams& p, cudaStream_t s) {
  using L = BwdLayout<D>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(bca_bwd_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, L::BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const unsigned grid = static_cast<unsigned>(p.BH) * (p.N_pad / kTileRows);
  bca_bwd_kernel<D><<<grid, L::THREADS, L::BYTES, s>>>(tq, tk, tv, tdo, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_bwd_pre(int d, const __nv_bfloat16* o, const __nv_bfloat16* dout,
                           const float* lse, float* lse2, float* delta, float* dq_acc, int BH,
                           int N, int N_pad, cudaStream_t s) {
  const unsigned grid = static_cast<unsigned>((static_cast<size_t>(BH) * N_pad + 7) / 8);
  if (d == 64)
    bwd_pre_kernel<64><<<grid, 256, 0, s>>>(o, dout, lse, lse2, delta, dq_acc, BH, N, N_pad);
  else
    bwd_pre_kernel<128><<<grid, 256, 0, s>>>(o, dout, lse, lse2, delta, dq_acc, BH, N, N_pad);
  return cudaGetLastError();
}

cudaError_t launch_bwd_main(int d, const CUtensorMap& tq, const CUtensorMap& tk,
                            const CUtensorMap& tv, const CUtensorMap& tdo, const BwdParams& p,
                            cudaStream_t s) {
  if (d == 64) return launch_bwd_main_t<64>(tq, tk, tv, tdo, p, s);
  return launch_bwd_main_t<128>(tq, tk, tv, tdo, p, s);
}

cudaError_t launch_bwd_post(int d, const float* dq_acc, __nv_bfloat16* dq, float scale, int BH,
                            int N, int N_pad, cudaStream_t s) {
  const size_t total = static_cast<size_t>(BH) * N * d / 4;
  const unsigned grid = static_cast<unsigned>((total + 255) / 256);
  if (total == 0) return cudaSuccess;
  if (d == 64)
    bwd_post_kernel<64><<<grid, 256, 0, s>>>(dq_acc, dq, scale, BH, N, N_pad);
  else
    bwd_post_kernel<128><<<grid, 256, 0, s>>>(dq_acc, dq, scale, BH, N, N_pad);
  return cudaGetLastError();
}

}  // namespace mw
