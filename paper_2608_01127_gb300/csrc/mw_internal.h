// Internal interfaces between the C-ABI layer and the CUDA kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mw {

// Rows of one query tile / key tile (the tcgen05 M and N of S = Q K^T).
constexpr int kTileRows = 128;
// Query tiles that share one key/value stream inside a forward CTA.
constexpr int kFwdQTiles = 2;
constexpr int kFwdBlockRows = kTileRows * kFwdQTiles;
constexpr int kMaxSplits = 16;

// Query rows per step of the backward key-tile kernel.
__host__ __device__ constexpr int bwd_q_rows(int) { return 128; }

// Forward over one (b,h) query block against up to three key segments:
//   A: ring rows [head, head + lenA)        (committed history, all visible)
//   B: ring rows [0, lenB)                  (the part after the wrap)
//   C: the queries' own rows [0, rows_q)    (chunk-causal: key < (chunk(i)+1) T)
// Training uses C only (ring_len = 0).
// RoPE frequencies omega_i = base^(-2i / rope_dims), i < rope_dims / 2,
// computed in fp64 on the host and handed over as two floats (hi + lo), so
// that frame * omega keeps its low bits for frames up to 2^24.
constexpr int kMaxRopePairs = 64;  // head dims up to 128
struct RopeFreq {
  float hi[kMaxRopePairs];
  float lo[kMaxRopePairs];
};

struct FwdParams {
  int BH;
  int rows_q;       // query rows (= rows of segment C) per (b,h)
  int d_io;         // head dim of the caller's tensors (<= the kernel's D; the
                    // TMA maps zero-fill the columns in between)
  int T;            // chunk length in tokens
  int n_qblocks;    // ceil(rows_q / kFwdBlockRows)
  int head_groups;  // the heads are scheduled in this many groups (1..BH)
  int ring_cap;
  int ring_head;
  int ring_len;
  int sink_len;     // tokens of the sink anchor, visited before the ring
  // RoPE re-shift (0 rope_dims: off): the sink anchor's keys turn forward by
  // rope_shift frames as they are read (the frequencies are a kernel
  // parameter of their own)
  int rope_dims;
  int rope_shift;
  int num_splits;   // 1: write bf16 O + LSE; >1: fp32 partials for the combine
  float scale_log2; // softmax scale * log2(e)
  __nv_bfloat16* o;
  float* lse;       // nullable
  float* o_part;    // [splits, BH, rows_q, d]
  float* lse_part;  // [splits, BH, rows_q]
  unsigned* status;
  unsigned long long budget_ns;
  int debug_skip_q;  // test hook: never load Q, so the MMA warp's wait expires
};

struct BwdParams {
  int BH;
  int head_groups;  // CTA order: groups of heads one after another
  int N;            // tokens per (b,h)
  int N_pad;        // N rounded up to kTileRows
  int d_io;         // head dim of the caller's tensors (<= the kernel's D)
  int T;
  float scale_log2;
  float scale;
  const float* lse2;   // [BH, N_pad]  LSE * log2(e); +inf on padding rows
  const float* delta;  // [BH, N_pad]  rowsum(dO * O); 0 on padding rows
  float* dq_acc;       // [BH, N_pad, d] fp32
  __nv_bfloat16* dk;
  __nv_bfloat16* dv;
  unsigned* status;
  unsigned long long budget_ns;
  int debug_skip_q;  // test hook: never load Q, so the first S^T wait expires
};

// A ring commit (Sec. 3.5): rows [0, rows) of each head of k_src / v_src
// ([B,H,src_rows,d], src_rows >= rows) go to ring rows (slot + r) mod cap of
// k_cache / v_cache ([B,H,cap,d]).  rows == 0: nothing to do.
struct CommitJob {
  __nv_bfloat16* kc = nullptr;
  __nv_bfloat16* vc = nullptr;
  const __nv_bfloat16* ks = nullptr;
  const __nv_bfloat16* vs = nullptr;
  int cap = 1, slot = 0, rows = 0, src_rows = 0, d = 0, BH = 0;
};

// One 16-byte piece of a commit: piece `idx` of head bh (row idx / (d/8),
// 16-byte column chunk idx % (d/8)) of K and of V.
__device__ __forceinline__ void commit_piece(const CommitJob& j, int bh, int idx) {
  const int pieces = j.d / 8;
  const int piece = idx % pieces;
  const int r = idx / pieces;
  int dst = j.slot + r;
  if (dst >= j.cap) dst -= j.cap;  // slot < cap and rows <= cap
  const size_t so = (static_cast<size_t>(bh) * j.src_rows + r) * j.d + piece * 8;
  const size_t dso = (static_cast<size_t>(bh) * j.cap + dst) * j.d + piece * 8;
  *reinterpret_cast<uint4*>(j.kc + dso) = *reinterpret_cast<const uint4*>(j.ks + so);
  *reinterpret_cast<uint4*>(j.vc + dso) = *reinterpret_cast<const uint4*>(j.vs + so);
}

// Programmatic dependent launch of the forward, the split combine and the
// commit (option "pdl", on by default): each may start while the previous
// kernel in the stream finishes and waits in-kernel before touching global
// memory.  pdl_config fills `cfg` (and its one attribute `attr`).
extern int g_pdl_enabled;
inline void pdl_config(cudaLaunchConfig_t& cfg, cudaLaunchAttribute& attr, dim3 grid, dim3 block,
                       size_t smem, cudaStream_t s) {
  cfg = cudaLaunchConfig_t{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = g_pdl_enabled ? 1 : 0;
}

// Launchers (return cudaGetLastError() of the launch).
// tkr/tvr: ring buffer maps; tks/tvs: sink anchor maps (any valid map when
// the segment is empty)
// d: tile width (64 or 128); dm: MMA width (d, or 80 on the 128-wide tiles
// for head dims up to 80)
// top: the fp32 split partials p.o_part as [splits * BH][rows_q][d] with
// 32-column boxes (any valid map when p.num_splits == 1)
cudaError_t launch_fwd(int d, int dm, const CUtensorMap& tq, const CUtensorMap& tk,
                       const CUtensorMap& tv, const CUtensorMap& tkr, const CUtensorMap& tvr, const CUtensorMap& tks,
                       const CUtensorMap& tvs, const CUtensorMap& top, const FwdParams& p,
                       const RopeFreq& rope_om, cudaStream_t s);
// d: the kernels' head dim (64 or 128); d_io: the caller's (a multiple of 8, <= d)
// The combine's launch also carries the ring commit `cj` (if cj.rows > 0)
// in blocks of its own: both only run once the forward has finished, and
// they touch disjoint memory.
cudaError_t launch_combine(int d, int d_io, const float* o_part, const float* lse_part,
                           __nv_bfloat16* o, float* lse, int splits, int BH, int rows,
                           const CommitJob& cj, cudaStream_t s);
// bias (d = 64, else null): per padded row 8 floats (hi, lo of -LSE/scale;
// hi, lo of -D; 4 zeros), the B operand of the tf32 MMAs that add those
// per-query terms to S^T and dP^T
cudaError_t launch_bwd_pre(int d, int d_io, const __nv_bfloat16* o, const __nv_bfloat16* dout,
                           const float* lse, float* lse2, float* delta, float* dq_acc,
                           float* bias, float inv_scale, int BH, int N, int N_pad, cudaStream_t s);
// tdq: f32 map over dQacc [BH, N_pad, d] with 32 x 32 boxes (128-byte
// swizzle), the target of the d = 64 kernel's TMA reduce-adds
// dm: MMA width as for launch_fwd
// tbias (d = 64): f32 map over the bias rows [BH, N_pad, 8], 8 x 128 boxes,
// 32-byte swizzle (d = 128: any map, unused)
cudaError_t launch_bwd_main(int d, int dm, const CUtensorMap& tq, const CUtensorMap& tk,
                            const CUtensorMap& tv, const CUtensorMap& tdo, const CUtensorMap& tdq,
                            const CUtensorMap& tbias, const BwdParams& p, cudaStream_t s);
cudaError_t launch_bwd_post(int d, int d_io, const float* dq_acc, __nv_bfloat16* dq, float scale,
                            int BH, int N, int N_pad, cudaStream_t s);
// d: any multiple of 8 (rows are copied in 16-byte pieces)
cudaError_t launch_commit(const CommitJob& j, cudaStream_t s);
// QKV split + temporal RoPE: qkv [B, N, 3, H, d] -> q, k, v [B, H, N, d]
// (d a multiple of 8; rope_dims = 0 is a plain split)
cudaError_t launch_qkv_rope(const __nv_bfloat16* qkv, __nv_bfloat16* q, __nv_bfloat16* k,
                            __nv_bfloat16* v, int B, int N, int H, int d, int rope_dims,
                            const RopeFreq& omega, int per_frame, int first_frame,
                            cudaStream_t s);

}  // namespace mw
