// Block-causal attention backward on sm_103a: the analytic gradient of
// softmax attention restricted to the chunk-causal mask of Sec. 3.2
// (training is bf16 mixed precision, Sec. 4.1).
//
//   pre : D_i = <dO_i, O_i>, LSE2_i = LSE_i * log2(e) (+inf on padding rows),
//         dQacc = 0; at d = 64 also the bias rows (-LSE/scale and -D as tf32
//         high and low parts) that the main kernel's MMAs add
//   main: one CTA per 128-row key tile of one (b,h); it owns dK, dV in TMEM
//         and visits only the query rows whose chunks can see it
//         (queries i >= chunk(k0) * T), QN query rows per step j:
//           S^T  = K Q^T            (tcgen05 -> TMEM; d = 64: + the -LSE bias)
//           dP^T = V dO^T           (tcgen05 -> TMEM; d = 64: + the -D bias)
//           P^T  = exp2(scale log2e S^T - LSE2)     (registers)
//           dS^T = P^T (dP^T - D)                   (registers)
//           P^T (bf16) -> TMEM; dS^T (bf16) -> shared memory (d = 128: to
//                 TMEM as well, beside P^T)
//           dV += P^T dO            (tcgen05, A = P^T from TMEM)
//           dK += dS^T Q            (d = 64: A from shared memory; d = 128:
//                                    from TMEM)
//           d = 64 : dQ_j = dS K    (query rows in TMEM lanes)
//           d = 128: dQ_j^T = K^T dS^T (head-dim columns in TMEM lanes)
//           dQacc += dQ_j  (fp32: TMA reduce-add of swizzled shared-memory
//                           boxes at d = 64, red.global at d = 128)
//   post: dQ = scale * dQacc -> bf16
//
// Software pipeline: the P/dS warps copy S^T and dP^T into registers and
// release their TMEM columns at once, so S^T and dP^T of step j+1 are
// computed while they work on step j; P^T is handed over before dS is
// computed, so dV_j overlaps that math; dK, dQ of step j run while the P/dS
// warps start step j+1.  At d = 128 TMEM holds one block X for S^T, then
// dP^T, then P^T / dS^T in turn, so those steps follow one another.
//
// Roles (512 threads): warps 0-7 P/dS (two warpgroups, one half of the query
// columns each, one key row per thread), warps 8-11 dQ drain, warp 12 TMA
// producer, warp 13 MMA issuer (d = 64: warp 13 issues S^T, dV, dP^T and
// warp 14 dK, dQ).
// TMEM (512 columns): d = 64: dV [0,64), dK [64,128), S^T [128,256),
// dP^T [256,384), P^T [384,448), dQ [448,512); d = 128: dV [0,128),
// dK [128,256), X [256,384), dQ^T [384,512).
// CTA order: head by head, or (where the host's model of the launch says it
// ends sooner) in head groups whose key tiles run side by side, the first
// (longest) ones first.
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {
namespace {

// D: the head-dim width of the shared-memory tiles (64 or 128); DM <= D:
// the columns the MMAs cover (S^T and dP^T reduce over DM, dK and dV have DM
// columns), 80 for head dims up to 80 on the 128-wide tiles
template <int D, int DM = D>
struct BwdLayout {
  static_assert(DM % 16 == 0 && DM <= D, "MMA width");
  static constexpr int QN = bwd_q_rows(D);           // query rows per step
  static constexpr bool DQT = (D == 128);            // dQ produced transposed
  static constexpr int CW = QN / 2;                  // query columns per P/dS warpgroup
  static constexpr int REG = D / 64;                 // 64-column swizzle regions per row
  static constexpr int KREGION = kTileRows * 128;    // region of a 128-row tile
  static constexpr int QREGION = QN * 128;           // region of a QN-row tile
  static constexpr int KTILE = REG * KREGION;
  static constexpr int QTILE = REG * QREGION;
  static constexpr int STAGES = (D == 64) ? 3 : 2;   // Q and dO tiles in flight
  static constexpr int DS_BYTES = (QN / 64) * KREGION;  // dS^T: 128 key rows x QN columns
  // d = 64: two dS^T buffers, so dS^T_{j+1} is written while dK_j / dQ_j read dS^T_j
  static constexpr int DS_BUFS = (D == 64) ? 2 : 1;
  // d = 64: per drain warp, one 32 x 32 f32 box with the 128-byte swizzle (the
  // TMA reduce-add source); 1024-byte aligned
  static constexpr int STG_BYTES = DQT ? 0 : 4 * 32 * 32 * 4;
  // d = 64: the per-query LSE and D terms enter S^T and dP^T through one
  // tf32 MMA each (a QN x 32-byte bias tile in each Q stage, all-ones A
  // rows), so the P/dS warps read no LSE or D rows from shared memory
  static constexpr bool FOLD = (D == 64);
  static constexpr int BIAS_BYTES = FOLD ? QN * 32 : 0;
  static constexpr int QSTRIDE = QTILE + BIAS_BYTES;  // one Q stage
  static constexpr int VEC_BYTES = FOLD ? 0 : QN * 4;
  static constexpr int ONES_BYTES = FOLD ? 512 : 0;   // two 256-byte atoms of A rows
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + KTILE;
  static constexpr int OFF_Q = OFF_V + KTILE;
  static constexpr int OFF_DO = OFF_Q + STAGES * QSTRIDE;
  static constexpr int OFF_DS = OFF_DO + STAGES * QTILE;
  static constexpr int OFF_STG = OFF_DS + DS_BUFS * DS_BYTES;
  static constexpr int OFF_LSE = OFF_STG + STG_BYTES;
  static constexpr int OFF_DELTA = OFF_LSE + STAGES * VEC_BYTES;
  static constexpr int OFF_ONES = OFF_DELTA + STAGES * VEC_BYTES;
  static constexpr int OFF_BAR = OFF_ONES + ONES_BYTES;
  // kv_full, q_full[S], q_empty[S], do_full[S], do_empty[S], s_full, s_free,
  // dp_full, dp_free, pt_ready, pt_free, p_ready, dq_full, dq_free,
  // ds_free[DS_BUFS], dkv_full
  static constexpr int NBAR = 1 + 4 * STAGES + 10 + DS_BUFS;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int BYTES = OFF_MISC + 16;
  // d = 128 has no room for separate S^T / dP^T / P^T-dS^T columns: one
  // 128-column block X holds them in turn (each is copied to registers
  // before the next one lands there)
  static constexpr bool SHARED_X = (D == 128);
  static constexpr bool TWO_ISSUERS = !SHARED_X;  // MMA issue split over warps 13 and 14
  static constexpr uint32_t DV_COL = 0;
  static constexpr uint32_t DK_COL = D;
  static constexpr uint32_t S_COL = 2 * D;
  static constexpr uint32_t DP_COL = SHARED_X ? S_COL : 2 * D + QN;
  // P^T (bf16 pairs; at d = 128 followed by dS^T).  At d = 64 dK reads dS^T
  // from shared memory (the copy dQ reads too), so dQ has columns of its own.
  static constexpr uint32_t PDS_COL = SHARED_X ? S_COL : 384u;
  static constexpr uint32_t DQ_COL = SHARED_X ? 384u : 448u;
  static constexpr int THREADS = 512;
  // CTA order in head groups (BwdParams::head_groups).  The 128-wide MMA
  // variant runs head by head with the key tile taken straight from the CTA
  // index: with the group decode it measured 2-3% slower even in head-by-
  // head order, and its training shapes have no tail for groups to win back.
  static constexpr bool GROUPED = !(D == 128 && DM == 128);
  // registers per thread after the re-split: the P/dS warpgroups get more,
  // the drain warpgroup and the control warpgroup (TMA, MMA) less; the three
  // shares add up to exactly the launch's 512 threads x 128 registers (at
  // d = 64, 168 / 88 / 88 measured 1.4% faster than 176 / 80 / 80 and
  // compiles without spills)
  static constexpr int REGS_LAUNCH = 128;
  static constexpr int REGS_PDS = (D == 64) ? 168 : 152;
  static constexpr int REGS_DRAIN = (D == 64) ? 88 : 104;
  static constexpr int REGS_CONTROL = (D == 64) ? 88 : 104;
  static_assert(256 * REGS_PDS + 128 * REGS_DRAIN + 128 * REGS_CONTROL == THREADS * REGS_LAUNCH,
                "register re-split must hand out exactly the launch's registers");
  static_assert(SHARED_X ? (2 * D + QN <= 384) : (2 * D + 2 * QN <= 384), "TMEM columns");
  static_assert(BYTES <= 232448, "shared memory");
};

__device__ __forceinline__ void red_add(float* addr, float a) {
  asm volatile("red.global.add.f32 [%0], %1;" ::"l"(addr), "f"(a) : "memory");
}

template <int D, int DM>
__global__ void __launch_bounds__(BwdLayout<D, DM>::THREADS, 1)
    bca_bwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
                   const __grid_constant__ CUtensorMap tm_dq,
                   const __grid_constant__ CUtensorMap tm_bias, const BwdParams p) {
  using L = BwdLayout<D, DM>;
  constexpr int NS = L::STAGES;
  constexpr int QN = L::QN;
  constexpr int CW = L::CW;
  extern __shared__ __align__(1024) uint8_t smem[];
  // ---- work item: p.head_groups groups of heads one after another (sizes
  // differ by at most one, the larger first), so that the CTAs running
  // together share a few heads' Q, dO and dQ accumulator in L2; inside a
  // group the key tiles near the start (the most work) come first, those of
  // all the group's heads side by side, so that the longest CTAs of the last
  // group do not start near the end of the launch
  const int n_kt = p.N_pad / kTileRows;
  int bh_decoded, kt;
  if constexpr (!L::GROUPED) {
    bh_decoded = blockIdx.x / n_kt;
    kt = blockIdx.x % n_kt;
  } else {
    const int x = blockIdx.x;
    const int g_base = p.BH / p.head_groups, g_rem = p.BH % p.head_groups;
    const int big = (g_base + 1) * n_kt;  // CTAs of one larger group
    int gsize, h0, in_grp;
    if (x < g_rem * big) {
      gsize = g_base + 1;
      h0 = (x / big) * gsize;
      in_grp = x % big;
    } else {
      const int y = x - g_rem * big;
      gsize = g_base;
      h0 = g_rem * (g_base + 1) + (y / (g_base * n_kt)) * g_base;
      in_grp = y % (g_base * n_kt);
    }
    bh_decoded = h0 + in_grp % gsize;
    kt = in_grp / gsize;
  }
  if ((smem_u32(smem) & 1023u) != 0u) {
    // nothing runs without aligned shared memory: report it, and give this
    // key tile's dK and dV rows a defined value (zero) instead of leaving
    // stale ones behind
    if (threadIdx.x == 0) atomicOr(p.status, kDevMisaligned);
    const int krow = kt * kTileRows + static_cast<int>(threadIdx.x & 127);
    if (threadIdx.x < 256 && krow < p.N) {
      const int d_io = (D == 64) ? D : p.d_io;
      __nv_bfloat16* out = threadIdx.x < 128 ? p.dk : p.dv;
      uint4* dst = reinterpret_cast<uint4*>(out + (static_cast<size_t>(bh_decoded) * p.N + krow) * d_io);
      for (int c = 0; c < d_io / 8; ++c) dst[c] = make_uint4(0u, 0u, 0u, 0u);
    }
    return;  // uniform across the CTA, before any barrier or TMEM use
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
  uint64_t* kv_full = bars;
  uint64_t* q_full = bars + 1;
  uint64_t* q_empty = q_full + NS;
  uint64_t* do_full = q_empty + NS;
  uint64_t* do_empty = do_full + NS;
  uint64_t* s_full = do_empty + NS;
  uint64_t* s_free = s_full + 1;
  uint64_t* dp_full = s_free + 1;
  uint64_t* dp_free = dp_full + 1;
  uint64_t* pt_ready = dp_free + 1;
  uint64_t* pt_free = pt_ready + 1;
  uint64_t* p_ready = pt_free + 1;
  uint64_t* dq_full = p_ready + 1;
  uint64_t* dq_free = dq_full + 1;
  uint64_t* ds_free = dq_free + 1;
  uint64_t* dkv_full = ds_free + L::DS_BUFS;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);
  // In grouped order the head and key tile are read back from shared memory
  // by each role, so that nothing derived from the decode above is held in a
  // register from the kernel's start (the decode is too long for the
  // compiler to redo, and the P/dS warps of the 80-wide variant spilled for
  // it); head by head they come straight from the CTA index.
  volatile int* head_slot = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 8);
  volatile int* tile_slot = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 12);
  auto head = [&]() -> int { return L::GROUPED ? *head_slot : static_cast<int>(blockIdx.x) / n_kt; };
  struct Sweep {
    int k0;       // first key row of the tile
    int m_begin;  // first query tile that sees it
    int n_q;      // query tiles visited
    int q_rot;    // where the sweep starts: each key tile at its own offset,
                  // so that the key tiles of one head running side by side
                  // reduce into different dQ tiles instead of contending for
                  // the same L2 lines
  };
  auto sweep = [&]() {
    const int t = L::GROUPED ? *tile_slot : static_cast<int>(blockIdx.x) % n_kt;
    Sweep w;
    w.k0 = t * kTileRows;
    w.m_begin = (w.k0 / p.T) * p.T / QN;  // the first query that sees key k0, in tiles
    w.n_q = p.N_pad / QN - w.m_begin;
    w.q_rot = t % w.n_q;
    return w;
  };

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if constexpr (L::FOLD) {
    // A rows of the bias MMAs: [1 1 0 0 | 1 1 0 0] picks the LSE pair of a
    // bias row, [0 0 1 1 | 0 0 1 1] its D pair; both 16-byte halves alike, so
    // the 32-byte swizzle leaves them unchanged (8 rows of each)
    if (threadIdx.x < 128) {
      const int a = threadIdx.x >> 6, c = threadIdx.x & 7;
      reinterpret_cast<float*>(smem + L::OFF_ONES)[threadIdx.x] =
          (((c & 3) < 2) == (a == 0)) ? 1.f : 0.f;
      fence_proxy_async_smem();
    }
  }
  if (threadIdx.x == 0) {
    *head_slot = bh_decoded;
    *tile_slot = kt;
    mbar_init(kv_full, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&q_full[s], 1);
      mbar_init(&q_empty[s], 1);
      mbar_init(&do_full[s], 1);
      mbar_init(&do_empty[s], 1);
    }
    mbar_init(s_full, 1);
    mbar_init(s_free, 8);
    mbar_init(dp_full, 1);
    mbar_init(dp_free, 8);
    mbar_init(pt_ready, 8);
    mbar_init(pt_free, 1);
    mbar_init(p_ready, 8);
    mbar_init(dq_full, 1);
    mbar_init(dq_free, 4);
    for (int b = 0; b < L::DS_BUFS; ++b) mbar_init(&ds_free[b], 1);
    mbar_init(dkv_full, L::TWO_ISSUERS ? 2 : 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 13) {
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

  if (warp >= 12) {
  // warpgroup 3 (TMA, MMA issuers, one idle warp): one re-split for all four
  regs_dec<L::REGS_CONTROL>();
  if (warp == 12) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const int bh = head();
      const auto [k0, m_begin, n_q, q_rot] = sweep();
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_do);
      mbar_arrive_expect_tx(kv_full, 2 * L::KTILE);
      for (int r = 0; r < L::REG; ++r) {
        tma_load_3d(sK + r * L::KREGION, &tm_k, kv_full, 64 * r, k0, bh);
        tma_load_3d(sV + r * L::KREGION, &tm_v, kv_full, 64 * r, k0, bh);
      }
      int issued_q = 0, issued_do = 0;
      for (int j = 0; j < n_q; ++j) {
        const int st = j % NS;
        const uint32_t ph = (j / NS) & 1;
        const int q0 = (m_begin + (j + q_rot) % n_q) * QN;
        const size_t voff = static_cast<size_t>(bh) * p.N_pad + q0;
        if (!mbar_wait(&q_empty[st], ph ^ 1, ctl)) break;
        if (!p.debug_skip_q) {
          mbar_arrive_expect_tx(&q_full[st], L::QTILE + L::BIAS_BYTES + L::VEC_BYTES);
          for (int r = 0; r < L::REG; ++r)
            tma_load_3d(sQ + st * L::QSTRIDE + r * L::QREGION, &tm_q, &q_full[st], 64 * r, q0, bh);
          if constexpr (L::FOLD)
            tma_load_3d(sQ + st * L::QSTRIDE + L::QTILE, &tm_bias, &q_full[st], 0, q0, bh);
          else
            bulk_load(sLSE + st * QN, p.lse2 + voff, L::VEC_BYTES, &q_full[st]);
          ++issued_q;
        }
        if (!mbar_wait(&do_empty[st], ph ^ 1, ctl)) break;
        mbar_arrive_expect_tx(&do_full[st], L::QTILE + L::VEC_BYTES);
        for (int r = 0; r < L::REG; ++r)
          tma_load_3d(sDO + st * L::QTILE + r * L::QREGION, &tm_do, &do_full[st], 64 * r, q0, bh);
        if constexpr (!L::FOLD) bulk_load(sDelta + st * QN, p.delta + voff, L::VEC_BYTES, &do_full[st]);
        ++issued_do;
      }
      if (*abort_flag) {
        drain_wait(kv_full, 0, p.budget_ns);
        for (int j = max(0, issued_q - NS); j < issued_q; ++j)
          drain_wait(&q_full[j % NS], (j / NS) & 1, p.budget_ns);
        for (int j = max(0, issued_do - NS); j < issued_do; ++j)
          drain_wait(&do_full[j % NS], (j / NS) & 1, p.budget_ns);
      }
    }
  } else if (warp == 13 || (L::TWO_ISSUERS && warp == 14)) {
    // ------------------------------------------------------------ MMA issuers (whole warps)
    const int n_q = sweep().n_q;
    // d = 64: warp 13 issues S^T, dV and dP^T, warp 14 dK and dQ, so that one
    // warp's waits never leave the tensor core's short queue empty.  They
    // share no TMEM columns; the P/dS barriers order their operands.
    // d = 128 (S^T, dP^T, P^T and dS^T share columns): warp 13 issues all.
    {
      const bool role_a = !L::TWO_ISSUERS || warp == 13;  // S^T, dV, dP^T
      const bool role_b = !L::TWO_ISSUERS || warp == 14;  // dK, dQ
      constexpr uint32_t idesc_s = idesc_bf16_f32(128, QN, false, false);    // S^T, dP^T
      constexpr uint32_t idesc_tn = idesc_bf16_f32(128, DM, false, true);    // dV, dK
      // d = 64: dQ = dS K (M = query rows); d = 128: dQ^T = K^T dS^T (M = head dim)
      constexpr uint32_t idesc_dq = L::DQT ? idesc_bf16_f32(128, QN, true, true)
                                           : idesc_bf16_f32(128, D, true, true);
      // descriptors computed once; each MMA adds a compile-time offset
      const uint64_t k_kmaj = sdesc_sw128(smem_u32(sK), 16, 1024);
      const uint64_t v_kmaj = sdesc_sw128(smem_u32(sV), 16, 1024);
      const uint64_t k_mn = sdesc_sw128(smem_u32(sK), L::KREGION, 1024);
      const uint64_t q_kmaj0 = sdesc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t do_kmaj0 = sdesc_sw128(smem_u32(sDO), 16, 1024);
      const uint64_t q_mn0 = sdesc_sw128(smem_u32(sQ), L::QREGION, 1024);
      const uint64_t do_mn0 = sdesc_sw128(smem_u32(sDO), L::QREGION, 1024);
      const uint64_t ds_mn0 = sdesc_sw128(smem_u32(sDS), L::KREGION, 1024);
      const uint64_t ds_kmaj0 = sdesc_sw128(smem_u32(sDS), 16, 1024);
      // d = 64: S^T += ones x (-LSE/scale) and dP^T += ones x (-D), one tf32
      // MMA each (K = 8); the 256-byte A atoms serve every 8-row group (SBO 0)
      const uint64_t ones_l = sdesc_sw32(smem_u32(smem + L::OFF_ONES), 0);
      const uint64_t ones_d = sdesc_sw32(smem_u32(smem + L::OFF_ONES + 256), 0);
      const uint64_t bias0 = sdesc_sw32(smem_u32(sQ + L::QTILE), 256);
      auto add_bias = [&](uint32_t d_col, uint64_t ones, int stage) {
        if constexpr (L::FOLD)
          umma_ss_tf32(tmem + d_col, ones, sdesc_add(bias0, stage * L::QSTRIDE),
                       idesc_tf32_f32(128, QN), 1u);
      };
      // X = A B^T, both K-major over d (S^T = K Q^T, dP^T = V dO^T)
      auto issue_kmajor = [&](uint32_t d_col, uint64_t a, uint64_t b) {
#pragma unroll
        for (int kk = 0; kk < DM / 16; ++kk) {
          const uint32_t ka = (kk >> 2) * L::KREGION + (kk & 3) * 32;
          const uint32_t kq = (kk >> 2) * L::QREGION + (kk & 3) * 32;
          umma_ss(tmem + d_col, sdesc_add(a, ka), sdesc_add(b, kq), idesc_s, kk > 0 ? 1u : 0u);
        }
      };
      // TMEM columns of the k-th 16-query slice of P^T and of dS^T (bf16 pairs)
      auto pt_col = [](int kk) -> uint32_t {
        return L::SHARED_X ? L::PDS_COL + (kk >> 2) * 64 + (kk & 3) * 8 : L::PDS_COL + kk * 8;
      };
      auto dst_col = [](int kk) -> uint32_t {
        return L::SHARED_X ? L::PDS_COL + (kk >> 2) * 64 + 32 + (kk & 3) * 8
                           : L::PDS_COL + QN / 2 + kk * 8;
      };
      bool ok = warp_wait(kv_full, 0, ctl);
      if (ok && role_a) ok = warp_wait(&q_full[0], 0, ctl);
      tc_fence_after();
      if (ok && role_a) {
        issue_kmajor(L::S_COL, k_kmaj, q_kmaj0);
        add_bias(L::S_COL, ones_l, 0);
        umma_commit(s_full);
        if (L::SHARED_X) ok = warp_wait(s_free, 0, ctl);  // X holds S^T_0 until read
        if (ok) ok = warp_wait(&do_full[0], 0, ctl);
        tc_fence_after();
      }
      if (ok && role_a) {
        issue_kmajor(L::DP_COL, v_kmaj, do_kmaj0);
        add_bias(L::DP_COL, ones_d, 0);
        umma_commit(dp_full);
      }
      for (int j = 0; ok && j < n_q; ++j) {
        const int st = j % NS;
        const int st1 = (j + 1) % NS;
        const uint32_t ph1 = ((j + 1) / NS) & 1;
        const bool more = j + 1 < n_q;
        const uint64_t do_mn = sdesc_add(do_mn0, st * L::QTILE);
        const uint64_t q_mn = sdesc_add(q_mn0, st * L::QSTRIDE);
        if (role_a) {
          if (!L::SHARED_X && more) {
            // S^T of the next step as soon as the P/dS warps hold S^T_j
            if (!(ok = warp_wait(s_free, j & 1, ctl))) break;
            if (!(ok = warp_wait(&q_full[st1], ph1, ctl))) break;
            tc_fence_after();
            issue_kmajor(L::S_COL, k_kmaj, sdesc_add(q_kmaj0, st1 * L::QSTRIDE));
            add_bias(L::S_COL, ones_l, st1);
            umma_commit(s_full);
          }
          // dV += P^T dO_j as soon as P^T_j is in TMEM (while dS_j is computed)
          if (!(ok = warp_wait(pt_ready, j & 1, ctl))) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < QN / 16; ++kk)
            umma_ts(tmem + L::DV_COL, tmem + pt_col(kk), sdesc_add(do_mn, kk * 2048),
                    idesc_tn, (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(&do_empty[st]);
          if (!L::SHARED_X) umma_commit(pt_free);
          if (!L::SHARED_X && more) {
            // dP^T of the next step once the P/dS warps hold dP^T_j
            if (!(ok = warp_wait(dp_free, j & 1, ctl))) break;
            if (!(ok = warp_wait(&do_full[st1], ph1, ctl))) break;
            tc_fence_after();
            issue_kmajor(L::DP_COL, v_kmaj, sdesc_add(do_kmaj0, st1 * L::QTILE));
            add_bias(L::DP_COL, ones_d, st1);
            umma_commit(dp_full);
          }
        }
        if (role_b) {
          if (!(ok = warp_wait(p_ready, j & 1, ctl))) break;
          tc_fence_after();
          if constexpr (!L::SHARED_X) {
            // d = 64: dQ_j first, so the drain starts while dK_j runs
            if (j > 0) {
              if (!(ok = warp_wait(dq_free, (j - 1) & 1, ctl))) break;
              tc_fence_after();
            }
            const uint64_t ds_mn = sdesc_add(ds_mn0, (j % L::DS_BUFS) * L::DS_BYTES);
#pragma unroll
            for (int kk = 0; kk < kTileRows / 16; ++kk)
              umma_ss(tmem + L::DQ_COL, sdesc_add(ds_mn, kk * 2048), sdesc_add(k_mn, kk * 2048),
                      idesc_dq, kk > 0 ? 1u : 0u);
            umma_commit(dq_full);
          }
          // dK += dS^T Q_j (d = 64: dS^T read from shared memory, K-major)
          const uint64_t ds_kmaj = sdesc_add(ds_kmaj0, (j % L::DS_BUFS) * L::DS_BYTES);
#pragma unroll
          for (int kk = 0; kk < QN / 16; ++kk) {
            if constexpr (L::SHARED_X)
              umma_ts(tmem + L::DK_COL, tmem + dst_col(kk), sdesc_add(q_mn, kk * 2048),
                      idesc_tn, (j > 0 || kk > 0) ? 1u : 0u);
            else
              umma_ss(tmem + L::DK_COL, sdesc_add(ds_kmaj, (kk >> 2) * L::KREGION + (kk & 3) * 32),
                      sdesc_add(q_mn, kk * 2048), idesc_tn, (j > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(&q_empty[st]);
          if constexpr (!L::SHARED_X) umma_commit(&ds_free[j % L::DS_BUFS]);
        }
        if (L::SHARED_X && more) {
          // X is free once dV/dK have read P^T/dS^T (issue order): S^T of the
          // next step, then its dP^T once the P/dS warps have read that S^T
          if (!(ok = warp_wait(&q_full[st1], ph1, ctl))) break;
          tc_fence_after();
          issue_kmajor(L::S_COL, k_kmaj, sdesc_add(q_kmaj0, st1 * L::QSTRIDE));
            add_bias(L::S_COL, ones_l, st1);
          umma_commit(s_full);
          if (!(ok = warp_wait(s_free, (j + 1) & 1, ctl))) break;
          if (!(ok = warp_wait(&do_full[st1], ph1, ctl))) break;
          tc_fence_after();
          issue_kmajor(L::DP_COL, v_kmaj, sdesc_add(do_kmaj0, st1 * L::QTILE));
            add_bias(L::DP_COL, ones_d, st1);
          umma_commit(dp_full);
        }
        if (L::SHARED_X && role_b) {
          // dQ of this step, once the drain has read the previous one
          if (j > 0) {
            if (!(ok = warp_wait(dq_free, (j - 1) & 1, ctl))) break;
            tc_fence_after();
          }
          const uint64_t ds_mn = sdesc_add(ds_mn0, (j % L::DS_BUFS) * L::DS_BYTES);
#pragma unroll
          for (int kk = 0; kk < kTileRows / 16; ++kk) {
            if constexpr (L::DQT)   // A = K^T (MN-major over d), B = dS^T (MN-major over queries)
              umma_ss(tmem + L::DQ_COL, sdesc_add(k_mn, kk * 2048), sdesc_add(ds_mn, kk * 2048),
                      idesc_dq, kk > 0 ? 1u : 0u);
            else                    // A = dS (MN-major over queries), B = K (MN-major over d)
              umma_ss(tmem + L::DQ_COL, sdesc_add(ds_mn, kk * 2048), sdesc_add(k_mn, kk * 2048),
                      idesc_dq, kk > 0 ? 1u : 0u);
          }
          umma_commit(dq_full);
          umma_commit(&ds_free[j % L::DS_BUFS]);
        }
      }
      if (ok) umma_commit(dkv_full);  // one arrival per issuing warp
    }
  }
  } else if (warp < 8) {
    regs_inc<L::REGS_PDS>();
    // ------------------------------------------------------------ P / dS (thread = key row)
    const auto [k0, m_begin, n_q, q_rot] = sweep();
    const int wg = warp >> 2;            // query columns [CW wg, CW wg + CW)
    const int wq = warp & 3;             // TMEM lane quadrant
    const int j_local = wq * 32 + lane;
    const int krow = k0 + j_local;
    const bool k_valid = krow < p.N;
    const int q_start = k_valid ? (krow / p.T) * p.T : 0x7fffffff;  // first query seeing this key
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    const uint32_t s_addr = lane_base + L::S_COL + CW * wg;
    const uint32_t dp_addr = lane_base + L::DP_COL + CW * wg;
    // P^T / dS^T destinations: within this warpgroup's own 64 X columns
    // (d = 128), or in the separate P^T and dS^T blocks (d = 64)
    const uint32_t pds_p = lane_base + (L::SHARED_X ? L::PDS_COL + 64 * wg : L::PDS_COL + 32 * wg);
    const uint32_t pds_s = L::SHARED_X ? pds_p + 32 : pds_p + QN / 2;
    const float sl2 = p.scale_log2;
    // this thread's dS^T row segment: region (CW wg) / 64, chunks from (CW wg % 64) / 8
    const int c0 = CW * wg;
    const int ds_off = (c0 >> 6) * L::KREGION + j_local * 128;
    const int chunk0 = (c0 & 63) >> 3;
    const int sw = j_local & 7;
    bool ok = true;
    for (int j = 0; j < n_q; ++j) {
      const int st = j % NS;
      const int q0 = (m_begin + (j + q_rot) % n_q) * QN;
      const float* lse2 = sLSE + st * QN + c0;
      const float* delta = sDelta + st * QN + c0;
      if (!(ok = warp_wait(s_full, j & 1, ctl))) break;
      tc_fence_after();
      // d = 128: the step's LSE row (16 bytes per load), read once S^T is in
      // registers (d = 64: the MMA has already subtracted LSE / scale)
      float2 nl[CW / 2];
      auto load_lse = [&]() {
#pragma unroll
        for (int c = 0; c < CW / 4; ++c) {
          const float4 v = reinterpret_cast<const float4*>(lse2)[c];
          nl[2 * c] = make_float2(-v.x, -v.y);
          nl[2 * c + 1] = make_float2(-v.z, -v.w);
        }
      };
      float pr[CW];
      {
        uint32_t r[CW / 32][32];
#pragma unroll
        for (int h = 0; h < CW / 32; ++h) tmem_ld32(s_addr + 32 * h, r[h]);
        tmem_wait_ld();
#pragma unroll
        for (int h = 0; h < CW / 32; ++h)
#pragma unroll
          for (int k = 0; k < 32; ++k) pr[32 * h + k] = __uint_as_float(r[h][k]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free);
      const int lim = q_start - q0 - c0;  // columns c < lim are masked
      if constexpr (!L::FOLD) load_lse();
      const float2 sl2x2 = make_float2(sl2, sl2);
#pragma unroll
      for (int c = 0; c < CW / 2; ++c) {
        // d = 64: the MMA already subtracted LSE/scale
        const float2 x = L::FOLD ? mul2(make_float2(pr[2 * c], pr[2 * c + 1]), sl2x2)
                                 : fma2(make_float2(pr[2 * c], pr[2 * c + 1]), sl2x2, nl[c]);
        pr[2 * c] = ex2_approx(x.x);
        pr[2 * c + 1] = ex2_approx(x.y);
      }
      if (__any_sync(0xffffffffu, lim > 0)) {
#pragma unroll
        for (int c = 0; c < CW; ++c)
          if (c < lim) pr[c] = 0.f;
      }
      uint32_t dk[CW / 2];
      uint32_t pk[L::SHARED_X ? CW / 2 : 1];  // d = 128: P^T packed alongside dS^T
      // d = 64: P^T (bf16 pairs) -> TMEM right away, so that dV_j starts
      // while dS_j is computed.  (d = 128: X still holds dP^T_j; P^T is stored
      // with dS^T at the end of the step, which measured faster there.)
      auto store_pt = [&]() {
        uint32_t pe[CW / 2];
#pragma unroll
        for (int c = 0; c < CW / 2; ++c) pe[c] = pack_bf16x2(pr[2 * c], pr[2 * c + 1]);
        tmem_st32(pds_p, pe);
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(pt_ready);
      };
      if constexpr (!L::SHARED_X) {
        if (j > 0) {  // dV_{j-1} has read P^T_{j-1}
          if (!(ok = warp_wait(pt_free, (j - 1) & 1, ctl))) break;
          tc_fence_after();
        }
        store_pt();
      }
      if (!(ok = warp_wait(dp_full, j & 1, ctl))) break;
      tc_fence_after();
      // d = 128: the step's D row came with dO, which dP^T_j has read
#pragma unroll
      for (int h = 0; h < CW / 32; ++h) {
        uint32_t r[32];
        tmem_ld32(dp_addr + 32 * h, r);
        tmem_wait_ld();
        if (!L::SHARED_X && h == CW / 32 - 1) {
          // dP^T is in registers: its columns can take the next step's dP^T
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(dp_free);
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          // d = 64: the MMA already subtracted D
          const float4 dv = L::FOLD ? make_float4(0.f, 0.f, 0.f, 0.f)
                                    : reinterpret_cast<const float4*>(delta)[8 * h + k];
          const int c = 32 * h + 4 * k;
          // dS = P (dP - D), two columns per instruction
          const float2 dp0 = make_float2(__uint_as_float(r[4 * k]), __uint_as_float(r[4 * k + 1]));
          const float2 dp1 = make_float2(__uint_as_float(r[4 * k + 2]), __uint_as_float(r[4 * k + 3]));
          const float2 t0 = L::FOLD ? dp0 : add2(dp0, make_float2(-dv.x, -dv.y));
          const float2 t1 = L::FOLD ? dp1 : add2(dp1, make_float2(-dv.z, -dv.w));
          const float2 s0 = mul2(make_float2(pr[c], pr[c + 1]), t0);
          const float2 s1 = mul2(make_float2(pr[c + 2], pr[c + 3]), t1);
          dk[16 * h + 2 * k] = pack_bf16x2(s0.x, s0.y);
          dk[16 * h + 2 * k + 1] = pack_bf16x2(s1.x, s1.y);
          if constexpr (L::SHARED_X) {
            pk[16 * h + 2 * k] = pack_bf16x2(pr[c], pr[c + 1]);
            pk[16 * h + 2 * k + 1] = pack_bf16x2(pr[c + 2], pr[c + 3]);
          }
        }
      }
      // dS^T row segment -> shared memory (swizzled like a TMA 128-byte tile)
      const int buf = j % L::DS_BUFS;
      if (j >= L::DS_BUFS &&
          !(ok = warp_wait(&ds_free[buf], ((j / L::DS_BUFS) - 1) & 1, ctl)))
        break;
      uint8_t* ds_row = sDS + buf * L::DS_BYTES + ds_off;
#pragma unroll
      for (int q = 0; q < CW / 8; ++q)
        *reinterpret_cast<uint4*>(ds_row + (((chunk0 + q) ^ sw) << 4)) =
            make_uint4(dk[4 * q], dk[4 * q + 1], dk[4 * q + 2], dk[4 * q + 3]);
      // d = 128: P^T and dS^T -> TMEM (the dK and dV A operands)
      if constexpr (L::SHARED_X) {
        tmem_st32(pds_p, pk);
        tmem_st32(pds_s, dk);
      }
      fence_proxy_async_smem();
      if constexpr (L::SHARED_X) tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (L::SHARED_X) mbar_arrive(pt_ready);
        mbar_arrive(p_ready);
      }
    }
    // ---- epilogue: warpgroup 0 writes dK (x scale), warpgroup 1 writes dV
    // (zeros if a wait gave up: the rows get a defined value either way)
    const bool have = ok && warp_wait(dkv_full, 0, ctl);
    tc_fence_after();
    {
      const uint32_t col0 = wg == 0 ? L::DK_COL : L::DV_COL;
      const float mul = have ? (wg == 0 ? p.scale : 1.f) : 0.f;
      __nv_bfloat16* out = wg == 0 ? p.dk : p.dv;
      // the caller's rows hold d_io <= D columns (multiples of 8); only the
      // 128-wide kernel serves padded head dims
      const int d_io = (D == 64) ? D : p.d_io;
      const size_t row_off = (static_cast<size_t>(head()) * p.N + krow) * d_io;
#pragma unroll
      for (int c = 0; c < (DM + 31) / 32; ++c) {  // the chunks holding the DM columns
        uint32_t r[32];
        if (have) {
          tmem_ld32(lane_base + col0 + 32 * c, r);
          tmem_wait_ld();
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k) r[k] = 0u;
        }
        if (k_valid && 32 * c < d_io) {
          const int n16 = min(4, (d_io - 32 * c) / 8);
          uint4* dst = reinterpret_cast<uint4*>(out + row_off + 32 * c);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (k < n16) dst[k] = make_uint4(pack_bf16x2(__uint_as_float(r[8 * k]) * mul, __uint_as_float(r[8 * k + 1]) * mul),
                                pack_bf16x2(__uint_as_float(r[8 * k + 2]) * mul, __uint_as_float(r[8 * k + 3]) * mul),
                                pack_bf16x2(__uint_as_float(r[8 * k + 4]) * mul, __uint_as_float(r[8 * k + 5]) * mul),
                                pack_bf16x2(__uint_as_float(r[8 * k + 6]) * mul, __uint_as_float(r[8 * k + 7]) * mul));
        }
      }
    }
  } else {
    regs_dec<L::REGS_DRAIN>();
    // ------------------------------------------------------------ dQ drain
    const int wq = warp & 3;
    const int bh = head();
    const auto [k0, m_begin, n_q, q_rot] = sweep();
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    for (int j = 0; j < n_q; ++j) {
      const int q0 = (m_begin + (j + q_rot) % n_q) * QN;
      if (!warp_wait(dq_full, j & 1, ctl)) break;
      tc_fence_after();
      if constexpr (L::DQT) {
        // lanes = head-dim columns, TMEM columns = the QN query rows; one warp
        // instruction reduces 32 consecutive head-dim columns of one row
        float* dst = p.dq_acc + (static_cast<size_t>(bh) * p.N_pad + q0) * D + wq * 32 + lane;
        // head-dim columns past the caller's hold zeros: no reductions for them
        const bool col_ok = wq * 32 + lane < p.d_io;
#pragma unroll
        for (int half = 0; half < QN / 64; ++half) {
          uint32_t r0[32], r1[32];
          tmem_ld32(lane_base + L::DQ_COL + 64 * half, r0);
          tmem_ld32(lane_base + L::DQ_COL + 64 * half + 32, r1);
          tmem_wait_ld();
          if (half == QN / 64 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(dq_free);
          }
          if (col_ok) {
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              red_add(dst + static_cast<size_t>(64 * half + c) * D, __uint_as_float(r0[c]));
              red_add(dst + static_cast<size_t>(64 * half + c + 32) * D, __uint_as_float(r1[c]));
            }
          }
        }
      } else {
        // lanes = query rows: the warp's 32 x D block goes to shared memory as
        // 32-column boxes with the 128-byte swizzle (16-byte chunk c of row r
        // at c ^ (r mod 8): conflict-free), and one lane hands each box to the
        // TMA unit as a reduce-add into dQacc
        static_assert(D == 64, "the drain below covers two 32-column boxes");
        uint8_t* stg = smem + L::OFF_STG + wq * 4096;
        uint32_t r[2][32];
        tmem_ld32(lane_base + L::DQ_COL, r[0]);
        tmem_ld32(lane_base + L::DQ_COL + 32, r[1]);
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(dq_free);  // dQ_j is in registers
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          if (lane == 0) bulk_wait_read_all();  // the box buffer was read by the TMA unit
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 8; ++i)
            *reinterpret_cast<uint4*>(stg + lane * 128 + ((i ^ (lane & 7)) << 4)) =
                make_uint4(r[c][4 * i], r[c][4 * i + 1], r[c][4 * i + 2], r[c][4 * i + 3]);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_reduce_add_3d(&tm_dq, stg, 32 * c, q0 + wq * 32, bh);
            bulk_commit_group();
          }
        }
      }
    }
    // every reduce-add has completed before the CTA's shared memory goes away
    if constexpr (!L::DQT) {
      if (lane == 0) bulk_wait_all();
      __syncwarp();
    }

  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 13) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// D_i = <dO_i, O_i>, LSE2_i = LSE_i log2(e) for i < N; padding rows get
// D = 0, LSE2 = +inf (so their P is exactly 0).  Also zeroes dQacc.  A group
// of D / 8 lanes covers one row with 16-byte loads and stores (4 rows per
// warp at d = 64, 2 at d = 128).
template <int D>
__global__ void __launch_bounds__(256) bwd_pre_kernel(const __nv_bfloat16* __restrict__ o,
                                                      const __nv_bfloat16* __restrict__ dout,
                                                      const float* __restrict__ lse,
                                                      float* __restrict__ lse2,
                                                      float* __restrict__ delta,
                                                      float* __restrict__ dq_acc,
                                                      float* __restrict__ bias, float inv_scale,
                                                      int BH, int N, int N_pad, int d_io_arg) {
  const int d_io = (D == 64) ? D : d_io_arg;  // padded head dims use the 128-wide kernels
  constexpr int G = D / 8;                     // lanes per row (8 bf16 = 16 bytes each)
  const int lane = threadIdx.x & 31;
  const long long gr = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) / G;  // padded row
  const int sub = lane % G;
  // (the grid covers whole rows; lanes past the end stay for the shuffles)
  const bool valid = gr < static_cast<long long>(BH) * N_pad;
  const int bh = static_cast<int>(gr / N_pad);
  const int i = static_cast<int>(gr % N_pad);
  if (valid) {  // dQacc row: D fp32 = 2 D / 8 float4 stores, G lanes
    float4* acc = reinterpret_cast<float4*>(dq_acc + gr * D);
#pragma unroll
    for (int k = 0; k < 2; ++k) acc[sub + k * G] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  float sum = 0.f;
  if (valid && i < N && 8 * sub < d_io) {  // d_io is a multiple of 8
    const size_t off = (static_cast<size_t>(bh) * N + i) * d_io + 8 * sub;
    const uint4 a = *reinterpret_cast<const uint4*>(o + off);
    const uint4 b = *reinterpret_cast<const uint4*>(dout + off);
    const uint32_t av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      sum = fmaf(__uint_as_float(av[k] << 16), __uint_as_float(bv[k] << 16), sum);
      sum = fmaf(__uint_as_float(av[k] & 0xffff0000u), __uint_as_float(bv[k] & 0xffff0000u), sum);
    }
  }
#pragma unroll
  for (int s = G / 2; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
  if (valid && sub == 0) {
    delta[gr] = sum;
    lse2[gr] = (i < N) ? lse[static_cast<size_t>(bh) * N + i] * 1.4426950408889634f : INFINITY;
    if (bias != nullptr) {
      // -LSE/scale and -D, each as a tf32 part (low 13 mantissa bits cleared)
      // and the fp32 remainder; padding rows get -1e30, so their P is 0
      const float lb = (i < N) ? -lse[static_cast<size_t>(bh) * N + i] * inv_scale : -1e30f;
      const float lh = __uint_as_float(__float_as_uint(lb) & 0xffffe000u);
      const float dh = __uint_as_float(__float_as_uint(-sum) & 0xffffe000u);
      float4* row = reinterpret_cast<float4*>(bias + gr * 8);
      row[0] = make_float4(lh, lb - lh, dh, -sum - dh);
      row[1] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(256) bwd_post_kernel(const float* __restrict__ dq_acc,
                                                       __nv_bfloat16* __restrict__ dq, float scale,
                                                       int BH, int N, int N_pad, int d_io_arg) {
  const int d_io = (D == 64) ? D : d_io_arg;  // padded head dims use the 128-wide kernels
  const size_t idx = (static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x);  // 4 elements
  const size_t total = static_cast<size_t>(BH) * N * d_io / 4;
  if (idx >= total) return;
  const size_t e = idx * 4;  // element of dq [BH, N, d_io]
  const size_t row = e / d_io;  // over BH * N
  const int c = static_cast<int>(e % d_io);
  const size_t bh = row / N;
  const size_t i = row % N;
  const float4 v = *reinterpret_cast<const float4*>(dq_acc + (bh * N_pad + i) * D + c);
  uint2 out;
  out.x = pack_bf16x2(v.x * scale, v.y * scale);
  out.y = pack_bf16x2(v.z * scale, v.w * scale);
  *reinterpret_cast<uint2*>(dq + e) = out;
}

template <int D, int DM>
cudaError_t launch_bwd_main_t(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                              const CUtensorMap& tdo, const CUtensorMap& tdq,
                              const CUtensorMap& tbias, const BwdParams& p, cudaStream_t s) {
  using L = BwdLayout<D, DM>;
  static bool attr_set = false;
  if (!attr_set) {
    // The in-kernel register re-split assumes the launch register count; with
    // any other count its setmaxnreg.inc could never be satisfied, so refuse.
    cudaFuncAttributes fa;
    cudaError_t e0 = cudaFuncGetAttributes(&fa, bca_bwd_kernel<D, DM>);
    if (e0 != cudaSuccess) return e0;
    if (fa.numRegs != L::REGS_LAUNCH) return cudaErrorInvalidKernelImage;
    cudaError_t e = cudaFuncSetAttribute(bca_bwd_kernel<D, DM>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, L::BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const unsigned grid = static_cast<unsigned>(p.BH) * (p.N_pad / kTileRows);
  bca_bwd_kernel<D, DM><<<grid, L::THREADS, L::BYTES, s>>>(tq, tk, tv, tdo, tdq, tbias, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_bwd_pre(int d, int d_io, const __nv_bfloat16* o, const __nv_bfloat16* dout,
                           const float* lse, float* lse2, float* delta, float* dq_acc,
                           float* bias, float inv_scale, int BH, int N, int N_pad, cudaStream_t s) {
  const size_t threads = static_cast<size_t>(BH) * N_pad * (d / 8);  // d / 8 lanes per row
  const unsigned grid = static_cast<unsigned>((threads + 255) / 256);
  if (d == 64)
    bwd_pre_kernel<64><<<grid, 256, 0, s>>>(o, dout, lse, lse2, delta, dq_acc, bias, inv_scale, BH, N, N_pad, d_io);
  else
    bwd_pre_kernel<128><<<grid, 256, 0, s>>>(o, dout, lse, lse2, delta, dq_acc, nullptr, 0.f, BH, N, N_pad, d_io);
  return cudaGetLastError();
}

cudaError_t launch_bwd_main(int d, int dm, const CUtensorMap& tq, const CUtensorMap& tk,
                            const CUtensorMap& tv, const CUtensorMap& tdo, const CUtensorMap& tdq,
                            const CUtensorMap& tbias, const BwdParams& p, cudaStream_t s) {
  if (d == 64) return launch_bwd_main_t<64, 64>(tq, tk, tv, tdo, tdq, tbias, p, s);
  if (dm == 80) return launch_bwd_main_t<128, 80>(tq, tk, tv, tdo, tdq, tbias, p, s);
  return launch_bwd_main_t<128, 128>(tq, tk, tv, tdo, tdq, tbias, p, s);
}

cudaError_t launch_bwd_post(int d, int d_io, const float* dq_acc, __nv_bfloat16* dq, float scale,
                            int BH, int N, int N_pad, cudaStream_t s) {
  const size_t total = static_cast<size_t>(BH) * N * d_io / 4;
  const unsigned grid = static_cast<unsigned>((total + 255) / 256);
  if (total == 0) return cudaSuccess;
  if (d == 64)
    bwd_post_kernel<64><<<grid, 256, 0, s>>>(dq_acc, dq, scale, BH, N, N_pad, d_io);
  else
    bwd_post_kernel<128><<<grid, 256, 0, s>>>(dq_acc, dq, scale, BH, N, N_pad, d_io);
  return cudaGetLastError();
}

}  // namespace mw
