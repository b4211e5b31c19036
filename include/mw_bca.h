/*
 * mw_bca.h -- C ABI of the GB300 (sm_103a) block-causal attention library.
 *
 * The operation (paper Sec. 3.2, "Block-Causal Video DiT"): the token
 * sequence of a video is cut into temporally ordered chunks of T_chunk tokens;
 * a token attends bidirectionally to every token of its own chunk and causally
 * to all tokens of earlier chunks, never to later chunks.  With
 * chunk(i) = floor(i / T_chunk):
 *
 *     s_ij  = scale * <q_i, k_j>               for chunk(j) <= chunk(i)
 *     LSE_i = ln sum_j exp(s_ij),   P_ij = exp(s_ij - LSE_i),   O_i = sum_j P_ij v_j
 *
 * Streaming inference (Sec. 3.5): finished chunks' keys/values are committed
 * once to a rolling KV cache -- a FIFO of fixed capacity held here as a ring
 * buffer -- and the chunks still being denoised (the in-flight / active
 * window, "pipelined denoising") attend to the whole committed history and,
 * chunk-causally, to the in-flight chunks before them and to themselves.
 *
 * Conventions shared by every entry point
 *   - Tensors are DEVICE pointers to contiguous row-major arrays
 *     [B, H, rows, d] of bf16 (raw 16-bit bfloat16 bits; nv_bfloat16 in CUDA),
 *     16-byte aligned.  LSE arrays are fp32 [B, H, rows].  The caller owns every
 *     buffer; the library keeps no pointer after a call returns.
 *   - d is a multiple of 8 from 64 to 128.  The kernels are built for 64
 *     and 128 (the head dims of most of the paper's model table, Sec. 4.1);
 *     a head dim in between (the 0.5B layout's 72) runs on the 128-wide
 *     kernels, whose loads fill the missing columns with zeros.  Anything
 *     else returns MW_ERR_UNSUPPORTED.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Every call
 *     validates its arguments on the host, then enqueues kernels on `stream`
 *     and returns without synchronising.  Outputs are ready when the stream
 *     reaches that point.
 *   - Outputs must not overlap inputs.
 *   - Errors: invalid arguments are rejected before anything is enqueued
 *     (MW_ERR_INVALID_ARG / MW_ERR_UNSUPPORTED / MW_ERR_WORKSPACE) and
 *     mw_last_error() describes why; a failed launch returns MW_ERR_CUDA.
 *     No entry point aborts, exits, throws or traps.  Every wait inside the
 *     kernels is bounded; a wait that runs out sets a bit in a per-device
 *     status word that mw_device_status() reports as MW_ERR_TIMEOUT.
 *   - The library allocates no device memory of its own except a 4-byte
 *     status word per device (a static device variable).
 */
#ifndef MW_BCA_H
#define MW_BCA_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MW_OK = 0,
  MW_ERR_INVALID_ARG = 1,  /* null pointer, bad size, misalignment, bad ring state */
  MW_ERR_UNSUPPORTED = 2,  /* valid but not implemented (d outside 64..128 or not a multiple of 8) */
  MW_ERR_CUDA = 3,         /* a CUDA runtime / driver call failed */
  MW_ERR_TIMEOUT = 4,      /* a kernel's bounded wait expired (mw_device_status) */
  MW_ERR_WORKSPACE = 5     /* workspace missing or smaller than *_workspace_size() */
} mw_status;

/*
 * Block-causal attention forward (Sec. 3.2) over N = n_chunks * T_chunk tokens.
 *   q, k, v : [B, H, N, d] bf16 (inputs, after any positional rotation)
 *   o       : [B, H, N, d] bf16 output
 *   lse     : [B, H, N] fp32 output, natural-log LSE_i of the scaled logits;
 *             may be NULL when the backward pass is not needed
 *   scale   : softmax scale (> 0), usually 1/sqrt(d)
 * B, H, n_chunks, T_chunk >= 1.  Only the visible (query chunk, key chunk)
 * blocks are computed; blocks above the chunk diagonal are never visited.
 */
mw_status mw_bca_fwd(const void* q, const void* k, const void* v, void* o, float* lse, int B,
                     int H, int n_chunks, int T_chunk, int d, float scale, void* stream);

/* Bytes of device workspace mw_bca_bwd needs (fp32 dQ accumulator plus two
 * fp32 row vectors, each padded to a multiple of 128 rows).  0 on bad sizes. */
size_t mw_bca_bwd_workspace_size(int B, int H, int n_chunks, int T_chunk, int d);

/*
 * The CTA order the backward key-tile kernel takes for these sizes: the
 * number of head groups its key tiles run in, one after another (B*H = one
 * head after another).  Host-side planning only, no device work: with
 * sm_count > 0 it plans for that many SMs, else for the current device.
 * The heads form groups of nearly equal size, and in a group the key tiles
 * of all its heads run side by side, the first (longest) ones first.  The
 * groups are taken where a list-scheduling model of the launch ends at least
 * 1% before head by head (launches of up to 2^18 CTAs; larger ones and head
 * dims over 80 always run head by head); the
 * option "bwd_group_heads" overrides the choice.  Returns -1 on invalid
 * sizes (mw_last_error says why).
 */
int mw_bca_bwd_head_groups(int B, int H, int n_chunks, int T_chunk, int d, int sm_count);

/*
 * Backward of mw_bca_fwd: the analytic gradient of sum(O * dO) with respect
 * to q, k, v (training in bf16 mixed precision, Sec. 4.1), P recomputed from
 * the saved LSE.
 *   q, k, v, o : forward inputs and output, [B, H, N, d] bf16
 *   lse        : forward LSE [B, H, N] fp32 (required)
 *   dout       : upstream gradient dO [B, H, N, d] bf16
 *   dq, dk, dv : gradients, [B, H, N, d] bf16 outputs
 *   workspace  : device scratch of ws_bytes >= mw_bca_bwd_workspace_size(),
 *                256-byte aligned, caller-owned; contents on entry ignored
 * dQ is accumulated in fp32 with atomic adds, so its bits can differ from run
 * to run in the last place; dK and dV are deterministic.
 */
mw_status mw_bca_bwd(const void* q, const void* k, const void* v, const void* o, const float* lse,
                     const void* dout, void* dq, void* dk, void* dv, void* workspace,
                     size_t ws_bytes, int B, int H, int n_chunks, int T_chunk, int d, float scale,
                     void* stream);

/*
 * mw_bca_bwd split into its three stages, with the same arguments:
 *   stage 1: D_i = <dO_i, O_i>, LSE_i * log2(e) and a zeroed fp32 dQ
 *            accumulator, all in the workspace;
 *   stage 2: the key-tile kernel: dK, dV, and dQ accumulated in the workspace;
 *   stage 3: dQ = scale * accumulator, converted to bf16.
 * Stages 1, 2, 3 enqueued in order on one stream with the same workspace equal
 * mw_bca_bwd; stage 0 runs all three.  Arguments a stage does not read may be
 * NULL (stage 1 reads o, lse, dout; stage 2 q, k, v, dout, dk, dv; stage 3 dq),
 * the workspace is always required.  Lets a caller time or interleave stages.
 */
mw_status mw_bca_bwd_stage(int stage, const void* q, const void* k, const void* v, const void* o,
                           const float* lse, const void* dout, void* dq, void* dk, void* dv,
                           void* workspace, size_t ws_bytes, int B, int H, int n_chunks,
                           int T_chunk, int d, float scale, void* stream);

/* Bytes of device workspace mw_bca_cache_fwd needs for these sizes on the
 * current device (split-KV partials; 0 when no split is used). */
size_t mw_bca_cache_workspace_size(int B, int H, int n_q_chunks, int T_chunk, int d,
                                   int cache_len);

/*
 * Forward of W = n_q_chunks in-flight chunks against the rolling KV cache
 * (Sec. 3.5: streaming inference with a structured rolling KV cache and
 * pipelined denoising).
 *   q, k_new, v_new : [B, H, W*T_chunk, d] bf16, the in-flight chunks in
 *                     temporal order
 *   k_cache, v_cache: ring buffers [B, H, cache_cap, d] bf16 of committed
 *                     tokens.  Logical token t (t = 0 the oldest) lives at
 *                     physical row (cache_head + t) mod cache_cap, for
 *                     0 <= t < cache_len; other rows are ignored.
 *   o               : [B, H, W*T_chunk, d] bf16 output
 *   lse             : [B, H, W*T_chunk] fp32 output or NULL
 *   workspace       : >= mw_bca_cache_workspace_size() bytes (may be NULL
 *                     when that size is 0), 256-byte aligned
 * In-flight chunk j sees all cache_len cached tokens and in-flight chunks
 * 0..j.  0 <= cache_head < cache_cap, 0 <= cache_len <= cache_cap.
 */
mw_status mw_bca_cache_fwd(const void* q, const void* k_new, const void* v_new,
                           const void* k_cache, const void* v_cache, int cache_cap,
                           int cache_head, int cache_len, void* o, float* lse, void* workspace,
                           size_t ws_bytes, int B, int H, int n_q_chunks, int T_chunk, int d,
                           float scale, void* stream);

/*
 * The same forward with a sink anchor ahead of the ring (Sec. 3.5, structured
 * rolling KV cache: the initial clean context is retained permanently as a
 * sink anchor that occupies the first position and never takes part in the
 * FIFO eviction).
 *   k_sink, v_sink  : [B, H, sink_len, d] bf16 (may be NULL when sink_len is 0)
 * In-flight chunk j sees the sink_len sink tokens, all cache_len cached
 * tokens and in-flight chunks 0..j.  0 <= sink_len <= 2^24; every other
 * argument is as for mw_bca_cache_fwd, which is this call with sink_len 0.
 * The workspace is mw_bca_cache_workspace_size(B, H, n_q_chunks, T_chunk, d,
 * sink_len + cache_len) bytes.
 */
mw_status mw_bca_cache_fwd_sink(const void* q, const void* k_new, const void* v_new,
                                const void* k_sink, const void* v_sink, int sink_len,
                                const void* k_cache, const void* v_cache, int cache_cap,
                                int cache_head, int cache_len, void* o, float* lse,
                                void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                                int T_chunk, int d, float scale, void* stream);

/*
 * The same forward with RoPE re-shifting (Sec. 3.5, RoPE re-shifting: after
 * each cache update the retained keys are re-indexed from the start of the
 * window by subtracting the temporal offset of the evicted chunks, so that
 * positions stay in the trained range; the sink anchor keeps the first
 * position and is excluded).
 *   The inputs carry their temporal rotation: queries, in-flight keys and the
 *   ring's keys at their stream positions (each key rotated once, when its
 *   chunk was projected, e.g. by mw_qkv_rope_split, and committed as it
 *   is), the sink's keys at the sink's own position(s).  shift_frames frames
 *   have been evicted.  Re-indexing moves the queries and every non-sink key
 *   back by the same offset, which leaves their mutual scores unchanged (RoPE
 *   scores depend on position differences only); what it changes are the
 *   query-sink scores.  This call computes exactly that: the sink's keys turn
 *   forward by shift_frames frames as they are read, rounded to bf16 before
 *   QK^T, and nothing else is rotated:
 *     channel pair (2i, 2i+1), 0 <= i < rope_dims / 2, turns by
 *     shift_frames * rope_base^(-2i / rope_dims):  (x, y) -> (x cos - y sin, x sin + y cos)
 *   Without a sink, or with shift_frames 0, the result is that of
 *   mw_bca_cache_fwd_sink.  The paper states neither the channel layout nor
 *   the frequencies of its RoPE, so they are arguments.
 *   rope_dims    : even, 0 <= rope_dims <= d (0: no rotation)
 *   rope_base    : > 1
 *   shift_frames : frames evicted so far, 0 <= shift_frames <= 2^24 (the
 *                  angle reduction is exact up to there)
 * Every other argument is as for mw_bca_cache_fwd_sink.
 */
mw_status mw_bca_cache_fwd_rope(const void* q, const void* k_new, const void* v_new,
                                const void* k_sink, const void* v_sink, int sink_len,
                                const void* k_cache, const void* v_cache, int cache_cap,
                                int cache_head, int cache_len, int rope_dims, float rope_base,
                                int shift_frames, void* o, float* lse,
                                void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                                int T_chunk, int d, float scale, void* stream);

/*
 * Commit of finished tokens into the ring (Sec. 3.5: once a chunk reaches the
 * data endpoint its keys/values go to the cache and are never modified).
 * Copies rows r = 0..rows-1 of k_src / v_src ([B, H, rows, d] bf16) to
 * physical ring rows (slot_start + r) mod cache_cap of k_cache / v_cache
 * ([B, H, cache_cap, d] bf16).  FIFO bookkeeping stays with the caller:
 * append at slot (head + len) mod cap, and when the ring is full advance head
 * by the rows written (the oldest tokens are the ones overwritten).
 * 0 <= slot_start < cache_cap, 1 <= rows <= cache_cap.
 */
mw_status mw_bca_cache_commit(void* k_cache, void* v_cache, int cache_cap, int slot_start,
                              const void* k_src, const void* v_src, int rows, int B, int H, int d,
                              void* stream);

/*
 * One streaming step (Sec. 3.5): the in-flight chunks attend to the ring as
 * in mw_bca_cache_fwd, then the oldest commit_rows rows of k_new / v_new
 * (the chunk that reached the data endpoint) are committed to ring rows
 * (commit_slot + r) mod cache_cap, exactly as mw_bca_cache_commit would.
 * The commit runs after the forward has read the ring (stream order), so
 * commit_slot may be the slot of the tokens it evicts; when the forward
 * splits its key range, the commit shares one launch with the split
 * combine.  The result equals mw_bca_cache_fwd followed by
 * mw_bca_cache_commit, bit for bit.
 *   k_cache, v_cache : written ([B,H,cache_cap,d])
 *   commit_rows      : 0 <= commit_rows <= min(cache_cap, n_q_chunks*T_chunk)
 *                      (0: no commit, i.e. mw_bca_cache_fwd)
 *   commit_slot      : 0 <= commit_slot < cache_cap
 * Every other argument, the workspace and the errors are as for
 * mw_bca_cache_fwd.
 */
mw_status mw_bca_cache_step(const void* q, const void* k_new, const void* v_new, void* k_cache,
                            void* v_cache, int cache_cap, int cache_head, int cache_len,
                            int commit_slot, int commit_rows, void* o, float* lse,
                            void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                            int T_chunk, int d, float scale, void* stream);

/*
 * QKV split with temporal RoPE (the input side of the attention: Sec. 3.2
 * runs block-causal attention over the latent tokens; Sec. 3.5 gives keys
 * temporal positions that the rolling cache re-shifts).  The fused QKV
 * projection leaves each token's heads interleaved; this writes them
 * head-major for the attention calls and rotates Q and K on the way:
 *   qkv     : [B, N, 3, H, d] bf16 (index 0 = Q, 1 = K, 2 = V), read only
 *   q, k, v : [B, H, N, d] bf16 outputs, written whole; must not overlap qkv
 * Token t sits at frame first_frame + t / tokens_per_frame; channel pair
 * (2i, 2i+1), 0 <= i < rope_dims / 2, of its query and key turns by
 *     frame * rope_base^(-2i / rope_dims):  (x, y) -> (x cos - y sin, x sin + y cos)
 * computed in fp32 and rounded to bf16 (V and the other channels are copied
 * bit for bit).  mw_bca_cache_fwd_rope turns ring keys on read with the same
 * arithmetic, so a key turned here to frame f equals an un-rotated ring key
 * turned there to frame f.  rope_dims = 0 is a plain split (rope_base,
 * tokens_per_frame and first_frame are then ignored).
 *   d                : a multiple of 8 from 64 to 128
 *   1 <= N <= 2^24, B * H * N <= 2^31
 *   rope_dims        : even, 0 <= rope_dims <= d
 *   rope_base        : > 1 (the frequencies base^(-2i/rope_dims) of this float
 *                      value are formed in fp64, and the angles reduced so
 *                      that they stay exact to ~1e-6 rad at every frame)
 *   tokens_per_frame : >= 1
 *   first_frame      : >= 0, and first_frame + (N - 1) / tokens_per_frame <= 2^24
 * Errors: MW_ERR_INVALID_ARG (NULL or misaligned pointer, bad sizes),
 * MW_ERR_UNSUPPORTED (d), MW_ERR_CUDA (launch).  Asynchronous on `stream`.
 */
mw_status mw_qkv_rope_split(const void* qkv, void* q, void* k, void* v, int B, int N, int H,
                            int d, int rope_dims, float rope_base, int tokens_per_frame,
                            int first_frame, void* stream);

/* Size of the library's static scratch array used by
 * mw_bca_cache_fwd_noalloc (64 MiB on every device that loads the library). */
#define MW_NOALLOC_SCRATCH_BYTES (64u << 20)

/*
 * mw_bca_cache_fwd without a workspace argument, for callers that cannot
 * allocate device memory: hosts that hand the library only their input and
 * output buffers (plugin-style integrations with no allocator), and real-time
 * streaming loops that must never call cudaMalloc / cudaFree because those
 * calls can synchronise the device and stall the stream.  This entry point
 * allocates nothing.  The split-KV partials it needs live in a fixed scratch
 * array of MW_NOALLOC_SCRATCH_BYTES that the library declares as a static
 * device variable; every GPU that loads the library holds that array until
 * the process exits.  The paper has no counterpart: this is an
 * integration convenience, not part of the method.
 *   Arguments, layouts and results are exactly those of mw_bca_cache_fwd
 *   (same kernels, same split plan), minus workspace / ws_bytes.
 *   When the partials for these sizes would exceed MW_NOALLOC_SCRATCH_BYTES
 *   the call returns MW_ERR_WORKSPACE, enqueues nothing, and mw_last_error()
 *   names the bytes needed; use mw_bca_cache_fwd with a caller workspace
 *   instead.
 *   The first call on a device looks up the array's device address
 *   (cudaGetSymbolAddress, once per device, with that device current); make
 *   that first call before any stream capture.
 *   All calls share the one array and it keeps the last call's contents.
 *   Each call writes every partial it later reads, so nothing has to start at
 *   zero; a kernel that cannot run (mw_device_status then reports it) writes
 *   its rows as O = 0, LSE = -inf rather than leaving an earlier call's
 *   partials to be merged.  Calls whose kernels overlap on the GPU (different
 *   streams, or different host threads without ordering) race on the array:
 *   serialise them, e.g. on one stream.
 */
mw_status mw_bca_cache_fwd_noalloc(const void* q, const void* k_new, const void* v_new,
                                   const void* k_cache, const void* v_cache, int cache_cap,
                                   int cache_head, int cache_len, void* o, float* lse, int B,
                                   int H, int n_q_chunks, int T_chunk, int d, float scale,
                                   void* stream);

/* Human-readable name of a status code (static string). */
const char* mw_status_string(mw_status s);

/* Message of the last failed call on this host thread ("" if none). */
const char* mw_last_error(void);

/*
 * Reads the status word of the current device after synchronising `stream`:
 * MW_ERR_TIMEOUT if any kernel since the last clear gave up a bounded wait,
 * MW_ERR_CUDA if the read itself failed, else MW_OK.  clear != 0 resets it.
 */
mw_status mw_device_status(void* stream, int clear);

/*
 * Tuning and test knobs (process-wide; not needed for normal use):
 *   "cache_splits"     split-KV count for mw_bca_cache_fwd, 0 = automatic
 *                      (the workspace size follows this setting)
 *   "wait_budget_ms"   time limit of every bounded wait inside the kernels
 *                      (default 2000)
 *   "debug_skip_q_load" non-zero: the forward and backward kernels never
 *                      load Q, so their first wait expires; for testing the
 *                      timeout path only
 *   "fwd_group_waves"  forward CTAs per head group, in multiples of the SM
 *                      count (default 3; 0 restores it): the query blocks of
 *                      a group's heads run together and share their K/V in L2
 *   "bwd_group_heads"  heads per group of the backward's CTA order, 0 =
 *                      automatic (groups sized by their work, Q/dO/dQ
 *                      bytes within 48 MB, taken where list scheduling
 *                      predicts a 1% shorter launch); 1 = one head after
 *                      another; head dims over 80 always run head by head
 *   "pdl"              0 launches the forward, the split combine and the
 *                      commit without programmatic dependent launch
 *                      (default 1)
 * Returns MW_ERR_INVALID_ARG for an unknown name or a negative value.
 */
mw_status mw_set_option(const char* name, long long value);

#ifdef __cplusplus
}
#endif

#endif /* MW_BCA_H */
