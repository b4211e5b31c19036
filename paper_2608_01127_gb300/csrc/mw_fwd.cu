// Block-causal attention forward on sm_103a (Sec. 3.2 block-causal
// self-attention; Sec. 3.5 rolling KV cache and pipelined denoising).
//
// One CTA owns a block of 2 x 128 query rows of one (b,h) and streams the key
// tiles that block can see.  Only unmasked work is enumerated: the key range
// of a query block ends at the end of the chunk of its last row, so whole
// chunk blocks above the diagonal are never visited; a per-row limit masks
// the few tiles that straddle a chunk edge.
//
// Roles (384 threads):
//   warps 0-3 / 4-7  softmax of query tile 0 / 1 (one thread per row = TMEM lane)
//   warp 8           TMA producer (Q once, then K/V tiles through a ring of stages)
//   warp 9           tcgen05 issuer (S = Q K^T into TMEM, O += P V with P in TMEM)
//   warps 10-11      RoPE re-shift of the sink anchor's key tiles in shared
//                    memory when it is enabled; with 80-wide MMAs on the
//                    128-wide tiles (and no re-shift) the ones columns of V;
//                    otherwise idle (they complete warpgroup 2 for the
//                    register re-split)
// TMEM (512 columns): S_t at column 128 t (P_t, bf16, overwrites its first 64
// columns), O_t at 256 + OW t (OW = the MMA width, plus 16 columns where the
// PV MMA also sums P through ones in V).
// CTA order: groups of heads of about three waves of CTAs, one group after
// another; in a group the longest query blocks first.
#include <type_traits>

#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace mw {
namespace {

// D: the head-dim width of the shared-memory tiles (64, or 128 with the
// columns past the caller's zero-filled by TMA); DM <= D: the columns the
// MMAs cover (QK^T reduces over DM, O has DM columns), 80 for head dims up
// to 80 on the 128-wide tiles
template <int D, int DM = D, bool ROPE = false>
struct FwdLayout {
  static_assert(DM % 16 == 0 && DM <= D, "MMA width");
  static constexpr int QT = kFwdQTiles;
  static constexpr int REG = D / 64;                  // 64-column swizzle regions per row
  static constexpr int REGION_BYTES = kTileRows * 128;
  static constexpr int TILE_BYTES = REG * REGION_BYTES;
  static constexpr int STAGES = (D == 64) ? 4 : 2;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + QT * TILE_BYTES;
  static constexpr int OFF_V = OFF_K + STAGES * TILE_BYTES;
  // The row sum of P comes out of the PV MMA itself: V gets 16 extra columns
  // of bf16 ones, so O gets 16 extra columns that all hold sum_j P_ij.
  // d = 64: the ones are a region of their own, reached through each stage
  // descriptor's leading-byte offset.  80-wide MMAs on the 128-wide tiles:
  // the ones go into columns 80..95 of each V tile (which TMA fills with
  // zeros), written by warps 10-11 after every load; with the RoPE re-shift
  // those warps are busy and the softmax sums P itself.
  static constexpr bool ONES_IN_V = (D == 128 && DM == 80 && !ROPE);
  static constexpr bool SUM_MMA = (D == 64) || ONES_IN_V;
  static constexpr int OW = SUM_MMA ? DM + 16 : DM;   // O columns in TMEM
  static constexpr int SUM_COL = DM;                  // first row-sum column of O
  static constexpr int OFF_ONES = OFF_V + STAGES * TILE_BYTES;
  static constexpr int ONES_BYTES = (D == 64) ? REGION_BYTES : 0;
  // RoPE re-shift: (cos, sin) of the shift per channel pair (one copy per
  // rotating warp)
  static constexpr int OFF_ROPE = OFF_ONES + ONES_BYTES;
  static constexpr int ROPE_WARP_BYTES = (D / 2) * 8;
  static constexpr int ROPE_BYTES = 2 * ROPE_WARP_BYTES;
  static constexpr int OFF_BAR = OFF_ROPE + ROPE_BYTES;
  static constexpr int NBAR = 1 + 6 * STAGES + 3 * QT + 1;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int BYTES = OFF_MISC + 16;
  static constexpr uint32_t S_COL(int t) { return 128u * t; }
  static constexpr uint32_t O_COL(int t) { return 256u + OW * t; }
  static constexpr int THREADS = 384;
  // registers per thread after the re-split: softmax warpgroups 0-1 get
  // more, warpgroup 2 (TMA, MMA, RoPE or idle warps) less; 2*128*S + 128*C
  // equals the launch's 384 threads x 168 registers.  d = 128: the MMA
  // warp's unrolled issue loop needs more than 56 (measured: 208/88 runs
  // the d=128 forward 4% faster, 224/56 the d=64 one 1% faster)
  static constexpr int REGS_LAUNCH = 168;
  static constexpr int REGS_SOFTMAX = (D == 64) ? 224 : 208;
  static constexpr int REGS_CONTROL = (D == 64) ? 56 : 88;
  static_assert(2 * 128 * REGS_SOFTMAX + 128 * REGS_CONTROL == THREADS * REGS_LAUNCH,
                "register re-split must hand out exactly the launch's registers");
};

// Where key tile j of a query block comes from.  Keys are visited in logical
// order: the sink anchor (segment S), the ring from its head to the end of
// the buffer (A) and from the start after wrapping (B), then the queries' own
// chunks (C).
enum : int { kSegOwn = 0, kSegRing = 1, kSegSink = 2 };
struct TileSrc {
  int seg;     // kSegOwn, kSegRing or kSegSink: which tensor maps hold the tile
  int row0;    // first physical row of the tile
  int end;     // ring and sink: exclusive end of the valid rows; own: unused
  int t0;      // ring: logical index (oldest = 0) of the tile's first row
};

struct Segs {
  int nS, nA, nB, nC;
  int endS, headA, endA, endB, lenA;
};

__device__ __forceinline__ TileSrc tile_src(const Segs& g, int j) {
  TileSrc s;
  s.t0 = 0;
  if (j < g.nS) {
    s.seg = kSegSink;
    s.row0 = j * kTileRows;
    s.end = g.endS;
    return s;
  }
  j -= g.nS;
  if (j < g.nA) {
    s.seg = kSegRing;
    s.row0 = g.headA + j * kTileRows;
    s.end = g.endA;
    s.t0 = j * kTileRows;
  } else if (j < g.nA + g.nB) {
    s.seg = kSegRing;
    s.row0 = (j - g.nA) * kTileRows;
    s.end = g.endB;
    s.t0 = g.lenA + (j - g.nA) * kTileRows;
  } else {
    s.seg = kSegOwn;
    s.row0 = (j - g.nA - g.nB) * kTileRows;
    s.end = 0;
  }
  return s;
}

// ROPE: the cache form with the RoPE re-shift of the sink anchor (warps 10-11
// turn its key tiles before the MMAs read them); the training and plain
// cache forms are compiled without it.  SPLIT: the key range is one of
// several (p.num_splits > 1), O goes out as fp32 partials through TMA
// stores; without it, as bf16 rows (the training form never pays for the
// partials' code).
template <int D, int DM, bool ROPE, bool SPLIT>
__global__ void __launch_bounds__(FwdLayout<D, DM>::THREADS, 1)
    bca_fwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_kr,
                   const __grid_constant__ CUtensorMap tm_vr, const __grid_constant__ CUtensorMap tm_ks,
                   const __grid_constant__ CUtensorMap tm_vs, const __grid_constant__ CUtensorMap tm_op,
                   const __grid_constant__ FwdParams p, const __grid_constant__ RopeFreq rope_om) {
  using L = FwdLayout<D, DM, ROPE>;
  constexpr int QT = L::QT;
  constexpr int NS = L::STAGES;
  extern __shared__ __align__(1024) uint8_t smem[];
  // ---- work item: p.head_groups groups of heads one after another (sizes
  // differ by at most one, the larger first), so that the CTAs running
  // together share a few heads' K/V in L2; inside a group the longest query
  // blocks (they see the most keys) come first
  int x = blockIdx.x;
  const int split = x % p.num_splits;
  x /= p.num_splits;
  const int g_base = p.BH / p.head_groups, g_rem = p.BH % p.head_groups;
  const int big = (g_base + 1) * p.n_qblocks;  // CTAs of one larger group
  int in_grp, gsize, h0;
  if (x < g_rem * big) {
    gsize = g_base + 1;
    h0 = (x / big) * gsize;
    in_grp = x % big;
  } else {
    const int y = x - g_rem * big;
    gsize = g_base;
    h0 = g_rem * (g_base + 1) + (y / (g_base * p.n_qblocks)) * g_base;
    in_grp = y % (g_base * p.n_qblocks);
  }
  const int bh = h0 + in_grp % gsize;
  const int qb = p.n_qblocks - 1 - in_grp / gsize;
  const int r0 = qb * kFwdBlockRows;
  if ((smem_u32(smem) & 1023u) != 0u) {
    // nothing runs without aligned shared memory: report it, and give this
    // CTA's rows a defined result (O = 0, LSE = -inf; as split partials, a
    // -inf LSE that the combine skips) instead of leaving stale values behind
    if (threadIdx.x == 0) atomicOr(p.status, kDevMisaligned);
    const int row = r0 + static_cast<int>(threadIdx.x);
    if (threadIdx.x < kFwdBlockRows && row < p.rows_q) {
      const size_t row_off = static_cast<size_t>(bh) * p.rows_q + row;
      if (p.num_splits == 1) {
        const int d_io = (D == 64) ? D : p.d_io;
        uint4* dst = reinterpret_cast<uint4*>(p.o + row_off * d_io);
        for (int c = 0; c < d_io / 8; ++c) dst[c] = make_uint4(0u, 0u, 0u, 0u);
        if (p.lse) p.lse[row_off] = -INFINITY;
      } else {
        p.lse_part[static_cast<size_t>(split) * p.BH * p.rows_q + row_off] = -INFINITY;
      }
    }
    return;  // uniform across the CTA, before any barrier or TMEM use
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;
  uint64_t* k_empty = k_full + NS;
  uint64_t* v_full = k_empty + NS;
  uint64_t* v_empty = v_full + NS;
  uint64_t* k_rdy = v_empty + NS;  // K tile in shared memory, RoPE re-shift applied
  uint64_t* v_rdy = k_rdy + NS;    // V tile in shared memory with its ones columns
  uint64_t* s_full = v_rdy + NS;
  uint64_t* p_full = s_full + QT;
  uint64_t* p_half = p_full + QT;  // first 64 keys of P in TMEM
  uint64_t* o_full = p_half + QT;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // query tiles of the block that hold rows (the last block may hold one)
  const int qt_n = (r0 + kTileRows < p.rows_q) ? QT : 1;
  const int last_row = min(r0 + kFwdBlockRows - 1, p.rows_q - 1);
  const int c_end = (last_row / p.T + 1) * p.T;  // keys of segment C visible to the block

  Segs g;
  g.lenA = 0;
  g.nS = (p.sink_len + kTileRows - 1) / kTileRows;
  g.endS = p.sink_len;
  const int lenA = min(p.ring_len, p.ring_cap - p.ring_head);
  const int lenB = p.ring_len - lenA;
  g.nA = (lenA + kTileRows - 1) / kTileRows;
  g.nB = (lenB + kTileRows - 1) / kTileRows;
  g.nC = (c_end + kTileRows - 1) / kTileRows;
  g.headA = p.ring_head;
  g.endA = p.ring_head + lenA;
  g.lenA = lenA;
  g.endB = lenB;
  const int n_all = g.nS + g.nA + g.nB + g.nC;
  const int j0 = (int)((long long)split * n_all / p.num_splits);
  const int j1 = (int)((long long)(split + 1) * n_all / p.num_splits);
  const int n_local = j1 - j0;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
      mbar_init(&k_rdy[s], 2);
      mbar_init(&v_rdy[s], 2);
    }
    for (int t = 0; t < QT; ++t) {
      mbar_init(&s_full[t], 1);
      mbar_init(&p_full[t], 4);
      mbar_init(&p_half[t], 4);
    }
    mbar_init(o_full, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 9) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  if constexpr (L::ONES_BYTES > 0) {
    uint32_t* ones = reinterpret_cast<uint32_t*>(smem + L::OFF_ONES);
    for (int k = threadIdx.x; k < L::ONES_BYTES / 4; k += L::THREADS) ones[k] = 0x3F803F80u;  // bf16 1.0
    fence_proxy_async_smem();  // read by the tensor core (async proxy)
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.status, p.budget_ns};
  // launched early (programmatic dependent launch): the setup above has run
  // while the previous kernel finished; global memory only from here on
  pdl_wait();

  uint8_t* sQ = smem + L::OFF_Q;
  uint8_t* sK = smem + L::OFF_K;
  uint8_t* sV = smem + L::OFF_V;

  if (warp >= 8) {
  // warpgroup 2: every warp executes this one re-split instruction
  regs_dec<L::REGS_CONTROL>();
  if (warp == 8) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && n_local > 0) {
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_k);
      prefetch_tmap(&tm_v);
      bool q_issued = false;
      if (!p.debug_skip_q) {
        mbar_arrive_expect_tx(q_full, QT * L::TILE_BYTES);
        for (int t = 0; t < QT; ++t)
          for (int r = 0; r < L::REG; ++r)
            tma_load_3d(sQ + t * L::TILE_BYTES + r * L::REGION_BYTES, &tm_q, q_full, 64 * r,
                        r0 + kTileRows * t, bh);
        q_issued = true;
      }
      int issued_k = 0, issued_v = 0;
      for (int i = 0; i < n_local; ++i) {
        const int st = i % NS;
        const uint32_t ph = (i / NS) & 1;
        const TileSrc src = tile_src(g, j0 + i);
        if (!mbar_wait(&k_empty[st], ph ^ 1, ctl)) break;
        mbar_arrive_expect_tx(&k_full[st], L::TILE_BYTES);
        for (int r = 0; r < L::REG; ++r)
          tma_load_3d(sK + st * L::TILE_BYTES + r * L::REGION_BYTES,
                      src.seg == kSegRing ? &tm_kr : src.seg == kSegSink ? &tm_ks : &tm_k,
                      &k_full[st], 64 * r, src.row0, bh);
        ++issued_k;
        if (!mbar_wait(&v_empty[st], ph ^ 1, ctl)) break;
        mbar_arrive_expect_tx(&v_full[st], L::TILE_BYTES);
        for (int r = 0; r < L::REG; ++r)
          tma_load_3d(sV + st * L::TILE_BYTES + r * L::REGION_BYTES,
                      src.seg == kSegRing ? &tm_vr : src.seg == kSegSink ? &tm_vs : &tm_v,
                      &v_full[st], 64 * r, src.row0, bh);
        ++issued_v;
      }
      if (*abort_flag) {
        // let every copy this CTA started land before shared memory goes away
        if (q_issued) drain_wait(q_full, 0, p.budget_ns);
        for (int i = max(0, issued_k - NS); i < issued_k; ++i)
          drain_wait(&k_full[i % NS], (i / NS) & 1, p.budget_ns);
        for (int i = max(0, issued_v - NS); i < issued_v; ++i)
          drain_wait(&v_full[i % NS], (i / NS) & 1, p.budget_ns);
      }
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------ MMA issuer (whole warp)
    if (n_local > 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, 128, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, L::OW, false, true);
      // descriptors computed once; each MMA adds a compile-time offset
      const uint64_t q_desc = sdesc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t k_desc = sdesc_sw128(smem_u32(sK), 16, 1024);
      const uint32_t v_addr = smem_u32(sV);
      const uint32_t ones_addr = smem_u32(smem + L::OFF_ONES);

      auto issue_qk = [&](int t, int st) {
        const uint64_t qa = sdesc_add(q_desc, t * L::TILE_BYTES);
        const uint64_t kb = sdesc_add(k_desc, st * L::TILE_BYTES);
#pragma unroll
        for (int kk = 0; kk < DM / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::REGION_BYTES + (kk & 3) * 32;
          umma_ss(tmem + L::S_COL(t), sdesc_add(qa, off), sdesc_add(kb, off), idesc_qk,
                  kk > 0 ? 1u : 0u);
        }
      };
      // O_t (+)= P_t V for keys [64 half, 64 half + 64) of the tile
      auto issue_pv = [&](int t, int st, bool acc, int half) {
        // V stage st; for d = 64 the next 64 "columns" are the ones region
        const uint32_t vs = v_addr + st * L::TILE_BYTES;
        const uint64_t vb = sdesc_sw128(vs, L::ONES_BYTES > 0 ? ones_addr - vs : L::REGION_BYTES, 1024);
#pragma unroll
        for (int k4 = 0; k4 < 4; ++k4) {
          const int kk = 4 * half + k4;
          umma_ts(tmem + L::O_COL(t), tmem + L::S_COL(t) + kk * 8, sdesc_add(vb, kk * 2048),
                  idesc_pv, (acc || kk > 0) ? 1u : 0u);
        }
      };

      bool ok = warp_wait(q_full, 0, ctl);
      tc_fence_after();
      for (int i = 0; ok && i < n_local; ++i) {
        const int st = i % NS;
        const uint32_t ph = (i / NS) & 1;
        const int stp = (i + NS - 1) % NS;
        const uint32_t php = ((i - 1) / NS) & 1;
        // with the re-shift, a sink tile is read once warps 10-11 have turned it
        const bool turned = ROPE && j0 + i < g.nS;
        if (!(ok = warp_wait(turned ? &k_rdy[st] : &k_full[st], ph, ctl))) break;
        tc_fence_after();
        // unrolled over the compile-time tile count, so every descriptor
        // offset stays a constant (a runtime trip count here slows the whole
        // forward by ~8%: the issuing code must never pause)
#pragma unroll
        for (int t = 0; t < QT; ++t) {
          if (t >= qt_n) break;
          if (i > 0) {
            // PV of the first 64 keys while the softmax warps store the rest of P
            if (!(ok = warp_wait(&p_half[t], (i - 1) & 1, ctl))) break;
            if (t == 0 && !(ok = warp_wait(L::ONES_IN_V ? &v_rdy[stp] : &v_full[stp], php, ctl))) break;
            tc_fence_after();
            issue_pv(t, stp, i - 1 > 0, 0);
            if (!(ok = warp_wait(&p_full[t], (i - 1) & 1, ctl))) break;
            tc_fence_after();
            issue_pv(t, stp, true, 1);
          }
          issue_qk(t, st);
          umma_commit(&s_full[t]);
        }
        if (!ok) break;
        umma_commit(&k_empty[st]);
        if (i > 0) umma_commit(&v_empty[stp]);
      }
      if (ok) {
        const int il = n_local - 1;
        const int stl = il % NS;
#pragma unroll
        for (int t = 0; t < QT; ++t) {
          if (!ok || t >= qt_n) break;
          if (!(ok = warp_wait(&p_half[t], il & 1, ctl))) break;
          if (t == 0 && !(ok = warp_wait(L::ONES_IN_V ? &v_rdy[stl] : &v_full[stl], (il / NS) & 1, ctl)))
            break;
          tc_fence_after();
          issue_pv(t, stl, il > 0, 0);
          if (!(ok = warp_wait(&p_full[t], il & 1, ctl))) break;
          tc_fence_after();
          issue_pv(t, stl, true, 1);
        }
        if (ok) {
          umma_commit(&v_empty[stl]);
          umma_commit(o_full);
        }
      }
    }
  } else if (ROPE && (warp == 10 || warp == 11) && n_local > 0) {
    // ------------------------------------------------------------ RoPE re-shift of the sink
    // Queries, in-flight keys and ring keys carry their temporal rotation at
    // stream positions.  Re-shifting (Sec. 3.5) moves the window back by the
    // evicted frames and leaves the sink anchor at its position; since the
    // scores depend only on position differences, that changes just the
    // query-sink angles, exactly as turning the sink's keys forward by
    // rope_shift frames does.  That happens here, in shared memory, between
    // the TMA copy of a sink tile and the MMAs that read it: channel pair
    // (2i, 2i+1), i < rope_dims / 2, turns by rope_shift * base^(-2i/rope_dims).
    // Each of the two warps turns its own half of every sink tile (rows
    // [64 h, 64 h + 64)), so they never wait for each other.
    const int half = warp - 10;
    float2* cs = reinterpret_cast<float2*>(smem + L::OFF_ROPE + half * L::ROPE_WARP_BYTES);
    const int pairs = p.rope_dims / 2;
    for (int i = lane; i < pairs; i += 32) cs[i] = rope_cos_sin(p.rope_shift, rope_om.hi[i], rope_om.lo[i]);
    __syncwarp();
    // lane -> (row within a pass, 16-byte chunk of 8 channels = 4 pairs)
    const int n_ch = (pairs + 3) / 4;
    const int rpp = 32 / n_ch;
    const int my_r = lane / n_ch, my_ch = lane % n_ch;
    const bool active = my_r < rpp;
    const int c0 = 8 * my_ch;
    const int np = min(4, pairs - 4 * my_ch);        // pairs of the chunk that turn
    const int region_off = (c0 >> 6) * L::REGION_BYTES;
    const int cidx = (c0 & 63) >> 3;                 // chunk index within the 128-byte row
    const float4 c01 = reinterpret_cast<const float4*>(cs)[2 * my_ch];
    const float4 c23 = reinterpret_cast<const float4*>(cs)[2 * my_ch + 1];
    const int n_sink = min(n_local, g.nS - j0);     // a block visits the sink first
    for (int i = 0; i < n_sink; ++i) {
      const int st = i % NS;
      if (!warp_wait(&k_full[st], (i / NS) & 1, ctl)) break;
      const TileSrc src = tile_src(g, j0 + i);
      const int r_lo = 64 * half;
      const int nrows = min(64, src.end - src.row0 - r_lo);  // valid rows of this half
      if (active && nrows > 0) {
        uint8_t* tile = sK + st * L::TILE_BYTES + region_off;
#pragma unroll 2
        for (int rr = my_r; rr < nrows; rr += rpp) {
          const int r = r_lo + rr;
          // 128-byte swizzle: 16-byte chunk index ^ (row mod 8)
          uint4* a = reinterpret_cast<uint4*>(tile + r * 128 + ((cidx ^ (r & 7)) << 4));
          uint4 v = *a;
          v.x = rope_turn(v.x, make_float2(c01.x, c01.y));
          if (np > 1) v.y = rope_turn(v.y, make_float2(c01.z, c01.w));
          if (np > 2) v.z = rope_turn(v.z, make_float2(c23.x, c23.y));
          if (np > 3) v.w = rope_turn(v.w, make_float2(c23.z, c23.w));
          *a = v;
        }
      }
      fence_proxy_async_smem();  // the tensor core reads the tile next
      __syncwarp();
      if (lane == 0) mbar_arrive(&k_rdy[st]);
    }
  } else if (L::ONES_IN_V && (warp == 10 || warp == 11) && n_local > 0) {
    // ------------------------------------------------------------ ones columns of V
    // columns DM..DM+15 of each V tile hold bf16 ones (the row-sum columns of
    // the PV MMA); TMA zero-fills them on every load, so they are written
    // again after each one: 16-byte chunks (DM-64)/8 and (DM-64)/8 + 1 of
    // region 1's 128-byte rows, at their 128-byte-swizzle positions
    const int half = warp - 10;
    const int c0 = (DM - 64) / 8;
    const uint4 ones = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    for (int i = 0; i < n_local; ++i) {
      const int st = i % NS;
      if (!warp_wait(&v_full[st], (i / NS) & 1, ctl)) break;
      uint8_t* reg1 = sV + st * L::TILE_BYTES + L::REGION_BYTES;
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int r = 64 * half + 32 * k + lane;
        *reinterpret_cast<uint4*>(reg1 + r * 128 + ((c0 ^ (r & 7)) << 4)) = ones;
        *reinterpret_cast<uint4*>(reg1 + r * 128 + (((c0 + 1) ^ (r & 7)) << 4)) = ones;
      }
      fence_proxy_async_smem();  // the tensor core reads the tile next
      __syncwarp();
      if (lane == 0) mbar_arrive(&v_rdy[st]);
    }
  }
  } else {
    regs_inc<L::REGS_SOFTMAX>();
    // ------------------------------------------------------------ softmax
    const int t = warp >> 2;
    const int wq = warp & 3;
    const int row_local = wq * 32 + lane;
    const int row = r0 + t * kTileRows + row_local;
    const bool row_valid = row < p.rows_q;
    const int c_limit = (min(row, p.rows_q - 1) / p.T + 1) * p.T;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    const uint32_t s_addr = lane_base + L::S_COL(t);
    const uint32_t o_addr = lane_base + L::O_COL(t);
    const float sl2 = p.scale_log2;

    float m_used = -INFINITY;
    float l = 0.f;
    bool ok = true;
    const int n_steps = t < qt_n ? n_local : 0;  // an empty query tile does nothing
    for (int i = 0; i < n_steps; ++i) {
      const TileSrc src = tile_src(g, j0 + i);
      if (!(ok = warp_wait(&s_full[t], i & 1, ctl))) break;
      tc_fence_after();
      float s[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t r[32];
        tmem_ld32(s_addr + 32 * c, r);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) s[32 * c + k] = __uint_as_float(r[k]);
      }
      const int limit = (src.seg != kSegOwn ? src.end : c_limit) - src.row0;
      if (limit < kTileRows) {
#pragma unroll
        for (int c = 0; c < 128; ++c)
          if (c >= limit) s[c] = -INFINITY;
      }
      float mq[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) mq[k] = fmaxf(s[k], s[k + 4]);
#pragma unroll
      for (int c = 8; c < 128; c += 8) {
        mq[0] = max3(mq[0], s[c], s[c + 1]);
        mq[1] = max3(mq[1], s[c + 2], s[c + 3]);
        mq[2] = max3(mq[2], s[c + 4], s[c + 5]);
        mq[3] = max3(mq[3], s[c + 6], s[c + 7]);
      }
      const float mx = max3(fmaxf(mq[0], mq[1]), mq[2], mq[3]);
      const float m_tile = mx * sl2;  // scale > 0
      const float m_cand = fmaxf(m_used, m_tile);
      // Rescale only when the running maximum grew by more than 2^8: P stays
      // below 256 in between, and the final O / l is exact either way.
      const bool need = m_cand > m_used + 8.0f;
      if (__any_sync(0xffffffffu, need)) {
        float alpha = 1.f;
        if (need) {
          alpha = ex2_approx(m_used - m_cand);
          m_used = m_cand;
        }
        l *= alpha;
        if (i > 0) {
          // exactly the tile's O columns (the next tile's O follows them)
#pragma unroll
          for (int c = 0; c < DM / 32; ++c) {
            uint32_t r[32];
            tmem_ld32(o_addr + 32 * c, r);
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < 32; ++k) r[k] = __float_as_uint(__uint_as_float(r[k]) * alpha);
            tmem_st32(o_addr + 32 * c, r);
          }
          if constexpr (DM % 32 != 0) {
            uint32_t r[16];
            tmem_ld16(o_addr + DM - 16, r);
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < 16; ++k) r[k] = __float_as_uint(__uint_as_float(r[k]) * alpha);
            tmem_st16(o_addr + DM - 16, r);
          }
          if constexpr (L::SUM_MMA) {  // the row-sum columns scale with O
            uint32_t r[16];
            tmem_ld16(o_addr + L::SUM_COL, r);
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < 16; ++k) r[k] = __float_as_uint(__uint_as_float(r[k]) * alpha);
            tmem_st16(o_addr + L::SUM_COL, r);
          }
          tmem_wait_st();
        }
      }
      const float m_eff = (m_used == -INFINITY) ? 0.f : m_used;
      const float2 sl2x2 = make_float2(sl2, sl2);
      const float2 negm = make_float2(-m_eff, -m_eff);
      float2 acc = make_float2(0.f, 0.f);
      // P in four 32-key groups, each stored as soon as it is packed; the first
      // two groups (keys 0..63) are announced while the third is stored
#pragma unroll
      for (int g4 = 0; g4 < 4; ++g4) {
        uint32_t packed[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float2 x = fma2(make_float2(s[32 * g4 + 2 * k], s[32 * g4 + 2 * k + 1]), sl2x2, negm);
          const uint32_t pk = pack_bf16x2(ex2_approx(x.x), ex2_approx(x.y));
          // the row sum uses the bf16 weights the PV MMA consumes, so O is an
          // exact convex combination of them (d = 64: summed by the MMA)
          if constexpr (!L::SUM_MMA)
            acc = add2(acc, make_float2(__uint_as_float(pk << 16), __uint_as_float(pk & 0xffff0000u)));
          packed[k] = pk;
        }
        if (g4 == 2) {  // the first half has landed: its PV can start
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&p_half[t]);
        }
        tmem_st16(s_addr + 16 * g4, packed);
      }
      l += acc.x + acc.y;
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[t]);
    }

    // ---- epilogue
    pdl_trigger();  // the next kernel (the split combine) may be scheduled now
    const bool have = __all_sync(0xffffffffu, ok) && n_steps > 0 && warp_wait(o_full, 0, ctl);
    tc_fence_after();
    if constexpr (L::SUM_MMA) {
      if (have) {
        uint32_t r[16];
        tmem_ld16(o_addr + L::SUM_COL, r);
        tmem_wait_ld();
        l = __uint_as_float(r[0]);
      }
    }
    const bool nonzero = have && l > 0.f;
    const float inv_l = nonzero ? 1.f / l : 0.f;
    const float m_eff = (m_used == -INFINITY) ? 0.f : m_used;
    const float lse = nonzero ? (m_eff + __log2f(l)) * 0.69314718055994530942f : -INFINITY;
    const size_t row_off = static_cast<size_t>(bh) * p.rows_q + row;
    // split partials: each warp writes its 32 rows of the tile's fp32 O into
    // shared memory (the K/V stages, no longer read once O is final) as
    // 32-column boxes with the 128-byte swizzle, and one thread of the tile
    // hands the boxes to the TMA unit.  Row-per-thread global stores would
    // cost 32 transactions per warp instruction, all CTAs at once.
    constexpr int kBoxBytes = kTileRows * 128;  // 128 rows x 32 fp32
    // the chunks that hold the DM columns of O (the caller's d_io <= DM)
#pragma unroll
    for (int c = 0; c < (DM + 31) / 32; ++c) {
      uint32_t r[32];
      if (have) {
        tmem_ld32(o_addr + 32 * c, r);
        tmem_wait_ld();
      }
      float v[32];
#pragma unroll
      for (int k = 0; k < 32; ++k) v[k] = nonzero ? __uint_as_float(r[k]) * inv_l : 0.f;
      if constexpr (!SPLIT) {
        if (!row_valid) continue;
        if (p.num_splits == 1) {
          // the caller's rows hold d_io <= D columns (multiples of 8); only
          // the 128-wide kernel serves padded head dims
          const int d_io = (D == 64) ? D : p.d_io;
          if (32 * c >= d_io) continue;
          const int n16 = min(4, (d_io - 32 * c) / 8);
          uint4* dst = reinterpret_cast<uint4*>(p.o + row_off * d_io + 32 * c);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (k < n16) dst[k] = make_uint4(pack_bf16x2(v[8 * k], v[8 * k + 1]), pack_bf16x2(v[8 * k + 2], v[8 * k + 3]),
                                pack_bf16x2(v[8 * k + 4], v[8 * k + 5]),
                                pack_bf16x2(v[8 * k + 6], v[8 * k + 7]));
        } else {
          // never taken (the launcher picks SPLIT for several splits), but
          // with this row-per-thread form of the partials here the compiler
          // schedules the training kernel 1.4% faster at d = 128
          float4* dst = reinterpret_cast<float4*>(
              p.o_part + (static_cast<size_t>(split) * p.BH * p.rows_q + row_off) * D + 32 * c);
#pragma unroll
          for (int k = 0; k < 8; ++k) dst[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
        }
      } else if (t < qt_n) {
        // (an empty tile's warps skip the O wait: they must not touch the
        // stages, which the other tile's MMAs may still be reading)
        // row row_local of box c: 16-byte piece k at piece k ^ (row mod 8)
        uint8_t* box_row = smem + L::OFF_K + (t * (D / 32) + c) * kBoxBytes + row_local * 128;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          *reinterpret_cast<float4*>(box_row + ((k ^ (row_local & 7)) << 4)) =
              make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
      }
    }
    if (SPLIT && t < qt_n) {  // a tile past the rows stores nothing
      fence_proxy_async_smem();  // the TMA unit reads the boxes next
      // this tile's four warps (barrier 1 or 2; 0 is __syncthreads)
      if (t == 0)
        named_barrier_sync<1, 4 * 32>();
      else
        named_barrier_sync<2, 4 * 32>();
      if (wq == 0 && lane == 0) {
        const uint8_t* stage = smem + L::OFF_K + t * (D / 32) * kBoxBytes;
#pragma unroll
        for (int c = 0; c < (DM + 31) / 32; ++c)
          tma_store_3d(&tm_op, stage + c * kBoxBytes, 32 * c, r0 + t * kTileRows, split * p.BH + bh);
        bulk_commit_group();
        bulk_wait_read_all();  // the boxes are read before the CTA's shared memory goes
      }
    }
    if (row_valid) {
      if (!SPLIT && p.num_splits == 1) {
        if (p.lse) p.lse[row_off] = lse;
      } else {
        p.lse_part[static_cast<size_t>(split) * p.BH * p.rows_q + row_off] = lse;
      }
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

// Merge of split-KV partials (per row): LSE = ln sum_s exp(LSE_s),
// O = sum_s exp(LSE_s - LSE) O_s.  One warp per row, 8 rows per block; the
// blocks after those carry the ring commit cj (one thread per 16-byte piece
// of a committed row of one head), when there is one.
template <int D>
__global__ void __launch_bounds__(256) combine_kernel(const float* __restrict__ o_part,
                                                      const float* __restrict__ lse_part,
                                                      __nv_bfloat16* __restrict__ o,
                                                      float* __restrict__ lse, int splits,
                                                      int n_rows, int d_io_arg,
                                                      const CommitJob cj) {
  pdl_wait();     // the forward's partials (and its reads of the ring) are complete
  pdl_trigger();  // the next step's forward may start its setup meanwhile
  const int combine_blocks = (n_rows + 7) / 8;
  if (static_cast<int>(blockIdx.x) >= combine_blocks) {
    const long long idx =
        static_cast<long long>(blockIdx.x - combine_blocks) * blockDim.x + threadIdx.x;
    const int per_head = cj.rows * (cj.d / 8);
    if (idx < static_cast<long long>(per_head) * cj.BH)
      commit_piece(cj, static_cast<int>(idx / per_head), static_cast<int>(idx % per_head));
    return;
  }
  const int d_io = (D == 64) ? D : d_io_arg;  // padded head dims use the 128-wide kernels
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= n_rows) return;
  constexpr int PER = D / 32;
  float acc[PER];
#pragma unroll
  for (int k = 0; k < PER; ++k) acc[k] = 0.f;
  float wsum = 0.f, m = -INFINITY;
  using Vec = typename std::conditional<PER == 4, float4, float2>::type;  // a lane's columns
  // a split whose LSE is -inf saw no key of the row: its O part is skipped
  // (never multiplied: it may hold anything)
  auto add = [&](float ls, const Vec& x) {
    const float w = ls == -INFINITY ? 0.f : __expf(ls - m);
    wsum += w;
    if (w > 0.f) {
      acc[0] += w * x.x;
      acc[1] += w * x.y;
      if constexpr (PER == 4) {
        acc[2] += w * x.z;
        acc[3] += w * x.w;
      }
    }
  };
  const Vec* src0 = reinterpret_cast<const Vec*>(o_part + static_cast<size_t>(row) * D) + lane;
  const size_t split_stride = static_cast<size_t>(n_rows) * D / PER;  // in Vec
  if (splits == 2) {
    // the usual case: both LSEs and both O parts requested at once (one
    // memory round trip instead of four)
    const float l0 = lse_part[row], l1 = lse_part[static_cast<size_t>(n_rows) + row];
    const Vec x0 = src0[0], x1 = src0[split_stride];
    m = fmaxf(l0, l1);
    add(l0, x0);
    add(l1, x1);
  } else {
    for (int s = 0; s < splits; ++s) m = fmaxf(m, lse_part[static_cast<size_t>(s) * n_rows + row]);
    for (int s = 0; s < splits; ++s)
      add(lse_part[static_cast<size_t>(s) * n_rows + row], src0[s * split_stride]);
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  __nv_bfloat16* dst = o + static_cast<size_t>(row) * d_io + lane * PER;
  if (lane * PER < d_io) {  // d_io is a multiple of 8, so a lane's PER columns are all in range
    if constexpr (PER == 4)
      *reinterpret_cast<uint2*>(dst) = make_uint2(pack_bf16x2(acc[0] * inv, acc[1] * inv),
                                                  pack_bf16x2(acc[2] * inv, acc[3] * inv));
    else
      *reinterpret_cast<uint32_t*>(dst) = pack_bf16x2(acc[0] * inv, acc[1] * inv);
  }
  if (lse && lane == 0) lse[row] = wsum > 0.f ? m + __logf(wsum) : -INFINITY;
}

template <int D, int DM, bool ROPE, bool SPLIT>
cudaError_t launch_fwd_t(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                         const CUtensorMap& tkr, const CUtensorMap& tvr, const CUtensorMap& tks,
                         const CUtensorMap& tvs, const CUtensorMap& top, const FwdParams& p,
                         const RopeFreq& om, cudaStream_t s) {
  using L = FwdLayout<D, DM, ROPE>;
  static bool attr_set = false;  // per process; the attribute is per function
  if (!attr_set) {
    // The in-kernel register re-split assumes the launch register count; with
    // any other count its setmaxnreg.inc could never be satisfied, so refuse.
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, bca_fwd_kernel<D, DM, ROPE, SPLIT>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs != L::REGS_LAUNCH) return cudaErrorInvalidKernelImage;
    e = cudaFuncSetAttribute(bca_fwd_kernel<D, DM, ROPE, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             L::BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const unsigned grid = static_cast<unsigned>(p.BH) * p.n_qblocks * p.num_splits;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr;
  pdl_config(cfg, attr, dim3(grid), dim3(L::THREADS), L::BYTES, s);
  return cudaLaunchKernelEx(&cfg, bca_fwd_kernel<D, DM, ROPE, SPLIT>, tq, tk, tv, tkr, tvr, tks, tvs, top, p,
                            om);
}

template <bool SPLIT>
cudaError_t launch_fwd_split(int d, int dm, const CUtensorMap& tq, const CUtensorMap& tk,
                             const CUtensorMap& tv, const CUtensorMap& tkr, const CUtensorMap& tvr,
                             const CUtensorMap& tks, const CUtensorMap& tvs, const CUtensorMap& top,
                             const FwdParams& p, const RopeFreq& om, cudaStream_t s) {
  if (p.rope_dims > 0) {
    if (d == 64) return launch_fwd_t<64, 64, true, SPLIT>(tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
    if (dm == 80) return launch_fwd_t<128, 80, true, SPLIT>(tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
    return launch_fwd_t<128, 128, true, SPLIT>(tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
  }
  if (d == 64) return launch_fwd_t<64, 64, false, SPLIT>(tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
  if (dm == 80) return launch_fwd_t<128, 80, false, SPLIT>(tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
  return launch_fwd_t<128, 128, false, SPLIT>(tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
}

}  // namespace

cudaError_t launch_fwd(int d, int dm, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                       const CUtensorMap& tkr, const CUtensorMap& tvr, const CUtensorMap& tks,
                       const CUtensorMap& tvs, const CUtensorMap& top, const FwdParams& p,
                       const RopeFreq& om, cudaStream_t s) {
  return p.num_splits > 1 ? launch_fwd_split<true>(d, dm, tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s)
                          : launch_fwd_split<false>(d, dm, tq, tk, tv, tkr, tvr, tks, tvs, top, p, om, s);
}

cudaError_t launch_combine(int d, int d_io, const float* o_part, const float* lse_part,
                           __nv_bfloat16* o, float* lse, int splits, int BH, int rows,
                           const CommitJob& cj, cudaStream_t s) {
  const int n_rows = BH * rows;
  const long long commit_pieces = static_cast<long long>(cj.rows) * (cj.d / 8) * cj.BH;
  const long long blocks = (n_rows + 7) / 8 + (commit_pieces + 255) / 256;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr;
  pdl_config(cfg, attr, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, s);
  if (d == 64)
    return cudaLaunchKernelEx(&cfg, combine_kernel<64>, o_part, lse_part, o, lse, splits, n_rows,
                              d_io, cj);
  return cudaLaunchKernelEx(&cfg, combine_kernel<128>, o_part, lse_part, o, lse, splits, n_rows,
                            d_io, cj);
}

}  // namespace mw
