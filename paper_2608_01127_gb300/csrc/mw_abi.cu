// C ABI of the block-causal attention library (declared in include/mw_bca.h):
// host-side validation, TMA descriptor creation, split-KV planning and
// kernel launches.  Validation happens before any CUDA call, so argument
// errors are reported without touching the device.
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstdarg>
#include <cstdio>
#include <cmath>
#include <cstring>
#include <functional>
#include <map>
#include <mutex>
#include <queue>
#include <string>
#include <tuple>
#include <vector>

#include "mw_bca.h"
#include "mw_internal.h"
#include "mw_ptx.cuh"

namespace {

thread_local std::string g_last_error;

// Device status word (bit 0: a bounded wait expired; bit 1: misaligned
// shared memory).  One per device: a static device variable.
__device__ unsigned g_status_word;

constexpr int kMaxDevices = 64;
unsigned* g_status_ptr[kMaxDevices] = {};
std::mutex g_mutex;

long long g_opt_cache_splits = 0;
long long g_opt_budget_ms = 2000;
long long g_opt_skip_q = 0;
long long g_opt_group_waves = 3;
long long g_opt_bwd_group_heads = 0;

mw_status fail(mw_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

mw_status ok() {
  g_last_error.clear();
  return MW_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

mw_status check_ptr(const void* p, const char* name) {
  if (p == nullptr) return fail(MW_ERR_INVALID_ARG, "%s is NULL", name);
  if (!aligned16(p)) return fail(MW_ERR_INVALID_ARG, "%s is not 16-byte aligned", name);
  return MW_OK;
}

// Head dims: the kernels are built for 64 and 128; a head dim in between (a
// multiple of 8, e.g. 72) runs on the 128-wide tiles, whose TMA maps read
// the caller's d columns and fill the rest of each 128-column tile with
// zeros; up to 80 the MMAs themselves cover only 80 columns.
bool d_supported(int d) { return d >= 64 && d <= 128 && d % 8 == 0; }
int kernel_d(int d) { return d == 64 ? 64 : 128; }
// The columns the MMAs cover: head dims up to 80 on the 128-wide tiles run
// 80-wide MMAs (QK^T over 80 columns, 80 output columns), the rest use the
// tile width.
int mma_d(int d) { return d == 64 ? 64 : (d <= 80 ? 80 : 128); }

mw_status check_dims(int B, int H, int d) {
  if (B < 1 || H < 1) return fail(MW_ERR_INVALID_ARG, "B and H must be >= 1 (B=%d H=%d)", B, H);
  if (static_cast<long long>(B) * H > (1 << 20))
    return fail(MW_ERR_INVALID_ARG, "B*H=%lld exceeds 2^20", static_cast<long long>(B) * H);
  if (!d_supported(d))
    return fail(MW_ERR_UNSUPPORTED, "head dim d=%d (supported: multiples of 8 from 64 to 128)", d);
  return MW_OK;
}

mw_status check_rows(long long rows, const char* what) {
  if (rows < 1 || rows > (1 << 24))
    return fail(MW_ERR_INVALID_ARG, "%s=%lld out of range [1, 2^24]", what, rows);
  return MW_OK;
}

// B*H*rows (plus padding to whole tiles) bounds every grid and element index
// the launches derive: keep it within 2^31 tokens.
mw_status check_tokens(long long BH, long long rows) {
  const long long padded = (rows + 255) / 256 * 256;
  if (BH * padded > (1ll << 31))
    return fail(MW_ERR_INVALID_ARG, "B*H*rows=%lld exceeds 2^31 tokens", BH * rows);
  return MW_OK;
}

#define MW_TRY(expr)                 \
  do {                               \
    mw_status _s = (expr);           \
    if (_s != MW_OK) return _s;      \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

// 3-D map over [BH, rows, d] with the 128-byte swizzle the tcgen05
// descriptors and the drain's boxes use; rows past the end read as zero.
// bf16 operands: 64-column x box_rows boxes.  f32 (the dQ accumulator):
// 32-column x box_rows boxes.
mw_status encode_map(CUtensorMap* m, const void* ptr, int rows, int BH, int d, const char* name,
                     int box_rows, bool f32 = false) {
  auto fn = encode_fn();
  if (!fn) return fail(MW_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable (no CUDA driver?)");
  const cuuint64_t es = f32 ? 4 : 2;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows),
                        static_cast<cuuint64_t>(BH)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * es,
                           static_cast<cuuint64_t>(rows) * d * es};
  cuuint32_t box[3] = {f32 ? 32u : 64u, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                  const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(MW_ERR_CUDA, "cuTensorMapEncodeTiled(%s) failed: %d", name, (int)r);
  return MW_OK;
}

// Small per-thread cache of encoded maps: streaming callers pass the same
// buffers every step, and encoding is pure host work that depends only on
// (address, shape, box).
struct MapKey {
  const void* ptr;
  int rows, BH, d, box_rows;
  bool f32;
  bool operator==(const MapKey& o) const {
    return ptr == o.ptr && rows == o.rows && BH == o.BH && d == o.d && box_rows == o.box_rows &&
           f32 == o.f32;
  }
};
constexpr int kMapCache = 16;
thread_local MapKey t_map_keys[kMapCache];
thread_local CUtensorMap t_maps[kMapCache];
thread_local int t_map_next = 0;

mw_status make_map(CUtensorMap* m, const void* ptr, int rows, int BH, int d, const char* name,
                   int box_rows = mw::kTileRows, bool f32 = false) {
  const MapKey key{ptr, rows, BH, d, box_rows, f32};
  for (int i = 0; i < kMapCache; ++i) {
    if (t_map_keys[i].ptr != nullptr && t_map_keys[i] == key) {
      *m = t_maps[i];
      return MW_OK;
    }
  }
  MW_TRY(encode_map(m, ptr, rows, BH, d, name, box_rows, f32));
  const int slot = t_map_next;
  t_map_next = (t_map_next + 1) % kMapCache;
  t_map_keys[slot] = key;
  t_maps[slot] = *m;
  return MW_OK;
}

mw_status status_ptr(unsigned** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(MW_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(MW_ERR_CUDA, "device index %d too large", dev);
  std::lock_guard<std::mutex> lock(g_mutex);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_status_word);
    if (e != cudaSuccess) return fail(MW_ERR_CUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    g_status_ptr[dev] = static_cast<unsigned*>(p);
  }
  *out = g_status_ptr[dev];
  return MW_OK;
}

// SM count of the current device, queried once per device.
int sm_count() {
  static int cached[kMaxDevices] = {};
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 152;
  if (cached[dev] > 0) return cached[dev];
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    return 152;
  cached[dev] = n;
  return n;
}

unsigned long long budget_ns() { return static_cast<unsigned long long>(g_opt_budget_ms) * 1000000ull; }

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int ceil_div(long long a, long long b) { return static_cast<int>((a + b - 1) / b); }

// Split-KV count for the cache path: balances (query blocks x splits) CTAs
// over the SMs against the per-split key-tile count plus a fixed cost.
int plan_splits(int BH, int rows_q, int cache_len) {
  if (g_opt_cache_splits > 0) return static_cast<int>(g_opt_cache_splits);
  const int blocks = BH * ceil_div(rows_q, mw::kFwdBlockRows);
  const int tiles = ceil_div(cache_len, mw::kTileRows) + 1 + ceil_div(rows_q, mw::kTileRows);
  const int sms = sm_count();
  int best = 1;
  long long best_cost = LLONG_MAX;
  for (int s = 1; s <= mw::kMaxSplits && s <= tiles; ++s) {
    const long long waves = ceil_div(static_cast<long long>(blocks) * s, sms);
    const long long cost = waves * (ceil_div(tiles, s) + 3);
    if (cost < best_cost) {
      best_cost = cost;
      best = s;
    }
  }
  return best;
}

// Finish time of the last SM when CTAs of the given lengths start in the given
// order, each on the SM that frees first (the hardware's dispatch, modelled
// as list scheduling).
long long list_makespan(const std::vector<int>& order_work, int sms) {
  std::priority_queue<long long, std::vector<long long>, std::greater<long long>> free_at;
  for (int i = 0; i < sms; ++i) free_at.push(0);
  long long end = 0;
  for (int w : order_work) {
    const long long t = free_at.top() + w;
    free_at.pop();
    free_at.push(t);
    end = std::max(end, t);
  }
  return end;
}

// CTA lengths of the backward in its launch order for `groups` head groups
// (the kernel's decode: groups of nearly equal size, the larger first; in a
// group, key tile after key tile, each over the group's heads)
std::vector<int> bwd_order_work(const std::vector<int>& kt_work, int BH, int groups) {
  const int n_kt = static_cast<int>(kt_work.size());
  const int g_base = BH / groups, g_rem = BH % groups;
  std::vector<int> out;
  out.reserve(static_cast<size_t>(BH) * n_kt);
  for (int g = 0; g < groups; ++g) {
    const int gsize = g_base + (g < g_rem ? 1 : 0);
    for (int kt = 0; kt < n_kt; ++kt)
      for (int h = 0; h < gsize; ++h) out.push_back(kt_work[kt]);
  }
  return out;
}

// Head groups of the backward's CTA order.  A key tile's CTA runs one step
// per visible query tile, plus a fixed cost of about three.  Head by head
// (groups of one head), the last head's longest key tiles start near the end
// of the launch; grouping heads lets them start earlier.  The candidate:
// the last group holds at least twice the longest CTA's steps on every SM,
// and a group's Q, dO and fp32 dQ accumulator stay within 48 MB.  It is
// taken when list scheduling puts its end at least 1% before that of head
// by head (the grouped decode and its wider L2 footprint cost about that
// much where the tail is small).  Decisions are cached per shape.  The
// kernel variant with 128-wide MMAs always runs head by head.
int bwd_head_groups(int BH, int N_pad, int T, int qrows, int d_io, int D, int sms) {
  if (D == 128 && mma_d(d_io) == 128) return BH;  // that kernel variant runs head by head
  if (g_opt_bwd_group_heads > 0) return ceil_div(BH, std::min<long long>(BH, g_opt_bwd_group_heads));
  static std::mutex mu;
  static std::map<std::tuple<int, int, int, int, int, int, int>, int> cache;
  const auto key = std::make_tuple(BH, N_pad, T, qrows, d_io, D, sms);
  {
    std::lock_guard<std::mutex> lock(mu);
    const auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  constexpr int kFixed = 3;
  constexpr long long kGroupBytes = 48LL << 20;
  const int n_kt = N_pad / mw::kTileRows;
  const int n_qt = N_pad / qrows;
  std::vector<int> kt_work(n_kt);
  long long per_head = 0, longest = 0;
  for (int kt = 0; kt < n_kt; ++kt) {
    const long long first_q = static_cast<long long>(kt) * mw::kTileRows / T * T;
    kt_work[kt] = static_cast<int>(n_qt - first_q / qrows + kFixed);
    per_head += kt_work[kt];
    longest = std::max<long long>(longest, kt_work[kt]);
  }
  const long long head_bytes = static_cast<long long>(N_pad) * (4LL * d_io + 4LL * D + 32);
  const long long per_group = std::max(1LL, std::min<long long>(
      std::min<long long>(BH, kGroupBytes / head_bytes),
      (2 * longest * sms + per_head - 1) / per_head));
  int groups = BH;  // head by head
  const int candidate = ceil_div(BH, per_group);
  // (past ~256K CTAs the model's host time passes a few ms, and with that
  // many the tail of head-by-head order is a small share of the launch)
  if (candidate < BH && static_cast<long long>(BH) * n_kt <= (1LL << 18)) {
    const long long t_heads = list_makespan(bwd_order_work(kt_work, BH, BH), sms);
    const long long t_groups = list_makespan(bwd_order_work(kt_work, BH, candidate), sms);
    if (100 * t_groups <= 99 * t_heads) groups = candidate;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() >= 4096) cache.clear();  // bounded for callers that vary the sizes
  cache.emplace(key, groups);
  return groups;
}

size_t cache_ws_bytes(int splits, int BH, int rows_q, int d) {
  if (splits <= 1) return 0;
  const size_t o_part = static_cast<size_t>(splits) * BH * rows_q * d * sizeof(float);
  const size_t l_part = static_cast<size_t>(splits) * BH * rows_q * sizeof(float);
  return align256(o_part) + align256(l_part);
}

struct BwdWs {
  size_t dq_acc, lse2, delta, bias, total;
};

// d = 64 adds the bias rows of the MMA-folded LSE and D terms: 8 floats
// (32 bytes) per padded row
BwdWs bwd_ws_layout(int BH, int N_pad, int d) {
  BwdWs w;
  w.dq_acc = 0;
  w.lse2 = align256(static_cast<size_t>(BH) * N_pad * d * sizeof(float));
  w.delta = w.lse2 + align256(static_cast<size_t>(BH) * N_pad * sizeof(float));
  w.bias = w.delta + align256(static_cast<size_t>(BH) * N_pad * sizeof(float));
  w.total = w.bias + (d == 64 ? align256(static_cast<size_t>(BH) * N_pad * 8 * sizeof(float)) : 0);
  return w;
}

// 3-D map over the bias rows [BH, N_pad, 8] f32: 8 x box_rows boxes with the
// 32-byte swizzle the tf32 MMA descriptors read
mw_status encode_bias_map(CUtensorMap* m, const float* bias, int N_pad, int BH, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return fail(MW_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable (no CUDA driver?)");
  cuuint64_t dims[3] = {8, static_cast<cuuint64_t>(N_pad), static_cast<cuuint64_t>(BH)};
  cuuint64_t strides[2] = {32, static_cast<cuuint64_t>(N_pad) * 32};
  cuuint32_t box[3] = {8, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(bias), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(MW_ERR_CUDA, "cuTensorMapEncodeTiled(bias) failed: %d", (int)r);
  return MW_OK;
}

// Makes the device of `stream` current on the calling thread for the scope
// of one entry point (binding its primary context, which driver calls such
// as cuTensorMapEncodeTiled need on threads where nothing else did), and
// restores the caller's device afterwards.
class DeviceScope {
 public:
  explicit DeviceScope(cudaStream_t stream) {
    if (cudaGetDevice(&prev_) != cudaSuccess) prev_ = -1;
    int dev = prev_;
    // (cudaStreamGetDevice is not allowed on a stream under graph capture,
    // and a capturing stream belongs to the current device anyway)
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (stream != nullptr && cudaStreamIsCapturing(stream, &cs) == cudaSuccess &&
        cs == cudaStreamCaptureStatusNone && cudaStreamGetDevice(stream, &dev) != cudaSuccess)
      dev = prev_;
    if (dev < 0) dev = 0;
    err_ = cudaSetDevice(dev);
    dev_ = dev;
  }
  ~DeviceScope() {
    if (prev_ >= 0 && prev_ != dev_) cudaSetDevice(prev_);
  }
  mw_status status() const {
    if (err_ != cudaSuccess) return fail(MW_ERR_CUDA, "cudaSetDevice: %s", cudaGetErrorString(err_));
    return MW_OK;
  }

 private:
  int prev_ = -1, dev_ = 0;
  cudaError_t err_ = cudaSuccess;
};

mw_status launch_status(cudaError_t e, const char* what) {
  if (e != cudaSuccess) return fail(MW_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  return ok();
}

struct RopeArgs {
  int dims = 0;          // 0: off
  mw::RopeFreq omega{};
  int shift = 0;         // frames the sink anchor's keys turn forward
};

// omega_i = base^(-2i / dims) in fp64, split into float hi + lo
mw::RopeFreq rope_freq(int dims, float base) {
  mw::RopeFreq f{};
  for (int i = 0; i < dims / 2 && i < mw::kMaxRopePairs; ++i) {
    const double w = std::pow(static_cast<double>(base), -2.0 * i / dims);
    f.hi[i] = static_cast<float>(w);
    f.lo[i] = static_cast<float>(w - static_cast<double>(f.hi[i]));
  }
  return f;
}

mw_status fwd_common(const void* q, const void* k, const void* v, const void* kr, const void* vr,
                     int cap, int head, int len, const void* ks, const void* vs, int sink_len,
                     const RopeArgs& rope, void* o, float* lse, void* ws, size_t ws_bytes, int BH,
                     int rows_q, int T, int d, float scale, int splits,
                     const mw::CommitJob& commit, cudaStream_t stream) {
  DeviceScope scope(stream);
  MW_TRY(scope.status());
  unsigned* status = nullptr;
  MW_TRY(status_ptr(&status));
  CUtensorMap tq, tk, tv, tkr, tvr, tks, tvs;
  MW_TRY(make_map(&tq, q, rows_q, BH, d, "q"));
  MW_TRY(make_map(&tk, k, rows_q, BH, d, "k"));
  MW_TRY(make_map(&tv, v, rows_q, BH, d, "v"));
  if (len > 0) {
    MW_TRY(make_map(&tkr, kr, cap, BH, d, "k_cache"));
    MW_TRY(make_map(&tvr, vr, cap, BH, d, "v_cache"));
  } else {
    tkr = tk;
    tvr = tv;
  }
  if (sink_len > 0) {
    MW_TRY(make_map(&tks, ks, sink_len, BH, d, "k_sink"));
    MW_TRY(make_map(&tvs, vs, sink_len, BH, d, "v_sink"));
  } else {
    tks = tk;
    tvs = tv;
  }
  const int D = kernel_d(d);
  mw::FwdParams p{};
  p.BH = BH;
  p.rows_q = rows_q;
  p.d_io = d;
  p.T = T;
  p.n_qblocks = ceil_div(rows_q, mw::kFwdBlockRows);
  // head groups of about three waves of CTAs each: a group's K/V stay in L2
  // while its query blocks run, and the longest blocks of each group start
  // first; groups of (nearly) equal size keep the last one from ending late
  // (at d = 128, groups of four waves hold 8 heads' K/V, 76 MB, and miss L2
  // often enough to read 1.44x the algorithmic bytes, three waves 1.04x;
  // two waves, 0.95x, leave more group boundaries, which cost the cache
  // forward with a sink anchor 4%)
  {
    const int per_group = std::max(1, std::min(BH, ceil_div(g_opt_group_waves * sm_count(),
                                                            static_cast<long long>(p.n_qblocks) * splits)));
    p.head_groups = ceil_div(BH, per_group);
  }
  p.ring_cap = len > 0 ? cap : 1;
  p.ring_head = len > 0 ? head : 0;
  p.ring_len = len;
  p.sink_len = sink_len;
  p.rope_dims = sink_len > 0 ? rope.dims : 0;
  p.rope_shift = rope.shift;
  p.num_splits = splits;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.o = static_cast<__nv_bfloat16*>(o);
  p.lse = lse;
  p.status = status;
  p.budget_ns = budget_ns();
  p.debug_skip_q = static_cast<int>(g_opt_skip_q);
  CUtensorMap top = tq;  // the split partials (TMA stores); unused with one split
  if (p.num_splits > 1) {
    const size_t need = cache_ws_bytes(p.num_splits, BH, rows_q, D);
    if (ws_bytes < need)
      return fail(MW_ERR_WORKSPACE, "workspace %zu bytes, need %zu", ws_bytes, need);
    char* base = static_cast<char*>(ws);
    p.o_part = reinterpret_cast<float*>(base);
    p.lse_part = reinterpret_cast<float*>(
        base + align256(static_cast<size_t>(p.num_splits) * BH * rows_q * D * sizeof(float)));
    MW_TRY(make_map(&top, p.o_part, rows_q, p.num_splits * BH, D, "o_part", mw::kTileRows, true));
  }
  MW_TRY(launch_status(mw::launch_fwd(D, mma_d(d), tq, tk, tv, tkr, tvr, tks, tvs, top, p, rope.omega,
                                      stream),
                       "forward kernel launch"));
  if (p.num_splits > 1)
    MW_TRY(launch_status(mw::launch_combine(D, d, p.o_part, p.lse_part, p.o, lse, p.num_splits, BH,
                                            rows_q, commit, stream),
                         "combine kernel launch"));
  else if (commit.rows > 0)
    MW_TRY(launch_status(mw::launch_commit(commit, stream), "commit kernel launch"));
  return ok();
}

}  // namespace

extern "C" {

const char* mw_status_string(mw_status s) {
  switch (s) {
    case MW_OK: return "MW_OK";
    case MW_ERR_INVALID_ARG: return "MW_ERR_INVALID_ARG";
    case MW_ERR_UNSUPPORTED: return "MW_ERR_UNSUPPORTED";
    case MW_ERR_CUDA: return "MW_ERR_CUDA";
    case MW_ERR_TIMEOUT: return "MW_ERR_TIMEOUT";
    case MW_ERR_WORKSPACE: return "MW_ERR_WORKSPACE";
  }
  return "MW_ERR_UNKNOWN";
}

const char* mw_last_error(void) { return g_last_error.c_str(); }

mw_status mw_set_option(const char* name, long long value) {
  if (name == nullptr) return fail(MW_ERR_INVALID_ARG, "option name is NULL");
  if (value < 0) return fail(MW_ERR_INVALID_ARG, "option %s: negative value", name);
  if (std::strcmp(name, "cache_splits") == 0) {
    if (value > mw::kMaxSplits) return fail(MW_ERR_INVALID_ARG, "cache_splits > %d", mw::kMaxSplits);
    g_opt_cache_splits = value;
  } else if (std::strcmp(name, "wait_budget_ms") == 0) {
    if (value < 1) return fail(MW_ERR_INVALID_ARG, "wait_budget_ms must be >= 1");
    g_opt_budget_ms = value;
  } else if (std::strcmp(name, "debug_skip_q_load") == 0) {
    g_opt_skip_q = value;
  } else if (std::strcmp(name, "fwd_group_waves") == 0) {
    g_opt_group_waves = value > 0 ? value : 3;
  } else if (std::strcmp(name, "bwd_group_heads") == 0) {
    g_opt_bwd_group_heads = value;
  } else if (std::strcmp(name, "pdl") == 0) {
    mw::g_pdl_enabled = value != 0;
  } else {
    return fail(MW_ERR_INVALID_ARG, "unknown option '%s'", name);
  }
  return ok();
}

mw_status mw_bca_fwd(const void* q, const void* k, const void* v, void* o, float* lse, int B,
                     int H, int n_chunks, int T_chunk, int d, float scale, void* stream) {
  MW_TRY(check_dims(B, H, d));
  if (n_chunks < 1 || T_chunk < 1)
    return fail(MW_ERR_INVALID_ARG, "n_chunks=%d and T_chunk=%d must be >= 1", n_chunks, T_chunk);
  const long long N = static_cast<long long>(n_chunks) * T_chunk;
  MW_TRY(check_rows(N, "n_chunks*T_chunk"));
  MW_TRY(check_tokens(static_cast<long long>(B) * H, N));
  if (!(scale > 0.f)) return fail(MW_ERR_INVALID_ARG, "scale must be > 0");
  MW_TRY(check_ptr(q, "q"));
  MW_TRY(check_ptr(k, "k"));
  MW_TRY(check_ptr(v, "v"));
  MW_TRY(check_ptr(o, "o"));
  if (lse && (reinterpret_cast<uintptr_t>(lse) & 3u))
    return fail(MW_ERR_INVALID_ARG, "lse is not 4-byte aligned");
  return fwd_common(q, k, v, nullptr, nullptr, 1, 0, 0, nullptr, nullptr, 0, RopeArgs{}, o, lse,
                    nullptr, 0, B * H, static_cast<int>(N), T_chunk, d, scale, 1, mw::CommitJob{},
                    static_cast<cudaStream_t>(stream));
}

int mw_bca_bwd_head_groups(int B, int H, int n_chunks, int T_chunk, int d, int sm_count_arg) {
  if (check_dims(B, H, d) != MW_OK) return -1;
  if (n_chunks < 1 || T_chunk < 1) {
    fail(MW_ERR_INVALID_ARG, "n_chunks=%d and T_chunk=%d must be >= 1", n_chunks, T_chunk);
    return -1;
  }
  const long long N = static_cast<long long>(n_chunks) * T_chunk;
  if (check_rows(N, "n_chunks*T_chunk") != MW_OK) return -1;
  const int N_pad = ceil_div(N, mw::kTileRows) * mw::kTileRows;
  const int D = kernel_d(d);
  return bwd_head_groups(B * H, N_pad, T_chunk, mw::bwd_q_rows(D), d, D,
                         sm_count_arg > 0 ? sm_count_arg : sm_count());
}

size_t mw_bca_bwd_workspace_size(int B, int H, int n_chunks, int T_chunk, int d) {
  if (B < 1 || H < 1 || n_chunks < 1 || T_chunk < 1 || !d_supported(d)) return 0;
  const long long N = static_cast<long long>(n_chunks) * T_chunk;
  if (N > (1 << 24)) return 0;
  const int N_pad = ceil_div(N, mw::kTileRows) * mw::kTileRows;
  return bwd_ws_layout(B * H, N_pad, kernel_d(d)).total;
}

mw_status mw_bca_bwd_stage(int stage, const void* q, const void* k, const void* v, const void* o,
                           const float* lse, const void* dout, void* dq, void* dk, void* dv,
                           void* workspace, size_t ws_bytes, int B, int H, int n_chunks,
                           int T_chunk, int d, float scale, void* stream) {
  if (stage < 0 || stage > 3) return fail(MW_ERR_INVALID_ARG, "stage=%d not in [0, 3]", stage);
  const bool pre = stage == 0 || stage == 1;
  const bool main = stage == 0 || stage == 2;
  const bool post = stage == 0 || stage == 3;
  MW_TRY(check_dims(B, H, d));
  if (n_chunks < 1 || T_chunk < 1)
    return fail(MW_ERR_INVALID_ARG, "n_chunks=%d and T_chunk=%d must be >= 1", n_chunks, T_chunk);
  const long long N = static_cast<long long>(n_chunks) * T_chunk;
  MW_TRY(check_rows(N, "n_chunks*T_chunk"));
  MW_TRY(check_tokens(static_cast<long long>(B) * H, N));
  if (!(scale > 0.f)) return fail(MW_ERR_INVALID_ARG, "scale must be > 0");
  if (main) {
    MW_TRY(check_ptr(q, "q"));
    MW_TRY(check_ptr(k, "k"));
    MW_TRY(check_ptr(v, "v"));
    MW_TRY(check_ptr(dk, "dk"));
    MW_TRY(check_ptr(dv, "dv"));
  }
  if (pre) {
    MW_TRY(check_ptr(o, "o"));
    MW_TRY(check_ptr(lse, "lse"));
  }
  if (pre || main) MW_TRY(check_ptr(dout, "dout"));
  if (post) MW_TRY(check_ptr(dq, "dq"));
  const int BH = B * H;
  const int N_pad = ceil_div(N, mw::kTileRows) * mw::kTileRows;
  const BwdWs w = bwd_ws_layout(BH, N_pad, kernel_d(d));
  if (workspace == nullptr || ws_bytes < w.total)
    return fail(MW_ERR_WORKSPACE, "workspace %zu bytes, need %zu", ws_bytes, w.total);
  if (reinterpret_cast<uintptr_t>(workspace) & 255u)
    return fail(MW_ERR_INVALID_ARG, "workspace is not 256-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  MW_TRY(scope.status());
  char* base = static_cast<char*>(workspace);
  float* dq_acc = reinterpret_cast<float*>(base + w.dq_acc);
  float* lse2 = reinterpret_cast<float*>(base + w.lse2);
  float* delta = reinterpret_cast<float*>(base + w.delta);
  float* bias = kernel_d(d) == 64 ? reinterpret_cast<float*>(base + w.bias) : nullptr;
  if (pre)
    MW_TRY(launch_status(mw::launch_bwd_pre(kernel_d(d), d, static_cast<const __nv_bfloat16*>(o),
                                            static_cast<const __nv_bfloat16*>(dout), lse, lse2,
                                            delta, dq_acc, bias, 1.f / scale, BH,
                                            static_cast<int>(N), N_pad, s),
                         "backward pre kernel launch"));
  if (main) {
    unsigned* status = nullptr;
    MW_TRY(status_ptr(&status));
    CUtensorMap tq, tk, tv, tdo, tdq;
    const int D = kernel_d(d);
    const int qrows = mw::bwd_q_rows(D);  // query rows per backward step
    MW_TRY(make_map(&tq, q, static_cast<int>(N), BH, d, "q", qrows));
    MW_TRY(make_map(&tk, k, static_cast<int>(N), BH, d, "k"));
    MW_TRY(make_map(&tv, v, static_cast<int>(N), BH, d, "v"));
    MW_TRY(make_map(&tdo, dout, static_cast<int>(N), BH, d, "dout", qrows));
    MW_TRY(make_map(&tdq, dq_acc, N_pad, BH, D, "dq_acc", 32, true));
    CUtensorMap tbias = tdq;  // d = 128: unused
    if (bias != nullptr) MW_TRY(encode_bias_map(&tbias, bias, N_pad, BH, qrows));
    mw::BwdParams p{};
    p.BH = BH;
    p.head_groups = bwd_head_groups(BH, N_pad, T_chunk, qrows, d, D, sm_count());
    p.N = static_cast<int>(N);
    p.N_pad = N_pad;
    p.d_io = d;
    p.T = T_chunk;
    p.scale_log2 = scale * 1.4426950408889634f;
    p.scale = scale;
    p.lse2 = lse2;
    p.delta = delta;
    p.dq_acc = dq_acc;
    p.dk = static_cast<__nv_bfloat16*>(dk);
    p.dv = static_cast<__nv_bfloat16*>(dv);
    p.status = status;
    p.budget_ns = budget_ns();
    p.debug_skip_q = static_cast<int>(g_opt_skip_q);
    MW_TRY(launch_status(mw::launch_bwd_main(D, mma_d(d), tq, tk, tv, tdo, tdq, tbias, p, s),
                         "backward kernel launch"));
  }
  if (post)
    MW_TRY(launch_status(mw::launch_bwd_post(kernel_d(d), d, dq_acc, static_cast<__nv_bfloat16*>(dq), scale, BH,
                                             static_cast<int>(N), N_pad, s),
                         "backward post kernel launch"));
  return ok();
}

mw_status mw_bca_bwd(const void* q, const void* k, const void* v, const void* o, const float* lse,
                     const void* dout, void* dq, void* dk, void* dv, void* workspace,
                     size_t ws_bytes, int B, int H, int n_chunks, int T_chunk, int d, float scale,
                     void* stream) {
  return mw_bca_bwd_stage(0, q, k, v, o, lse, dout, dq, dk, dv, workspace, ws_bytes, B, H,
                          n_chunks, T_chunk, d, scale, stream);
}

size_t mw_bca_cache_workspace_size(int B, int H, int n_q_chunks, int T_chunk, int d,
                                   int cache_len) {
  if (B < 1 || H < 1 || n_q_chunks < 1 || T_chunk < 1 || cache_len < 0 || !d_supported(d))
    return 0;
  const long long rows = static_cast<long long>(n_q_chunks) * T_chunk;
  if (rows > (1 << 24)) return 0;
  const int splits = plan_splits(B * H, static_cast<int>(rows), cache_len);
  return cache_ws_bytes(splits, B * H, static_cast<int>(rows), kernel_d(d));
}

mw_status mw_bca_cache_fwd(const void* q, const void* k_new, const void* v_new,
                           const void* k_cache, const void* v_cache, int cache_cap,
                           int cache_head, int cache_len, void* o, float* lse, void* workspace,
                           size_t ws_bytes, int B, int H, int n_q_chunks, int T_chunk, int d,
                           float scale, void* stream) {
  return mw_bca_cache_fwd_sink(q, k_new, v_new, nullptr, nullptr, 0, k_cache, v_cache, cache_cap,
                               cache_head, cache_len, o, lse, workspace, ws_bytes, B, H,
                               n_q_chunks, T_chunk, d, scale, stream);
}

mw_status mw_bca_cache_fwd_sink(const void* q, const void* k_new, const void* v_new,
                                const void* k_sink, const void* v_sink, int sink_len,
                                const void* k_cache, const void* v_cache, int cache_cap,
                                int cache_head, int cache_len, void* o, float* lse,
                                void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                                int T_chunk, int d, float scale, void* stream) {
  return mw_bca_cache_fwd_rope(q, k_new, v_new, k_sink, v_sink, sink_len, k_cache, v_cache,
                               cache_cap, cache_head, cache_len, 0, 0.f, 0, o, lse, workspace,
                               ws_bytes, B, H, n_q_chunks, T_chunk, d, scale, stream);
}

// The cache forward in all its forms; `commit` (rows > 0) is a ring commit
// that runs once the forward has read the ring.
static mw_status cache_fwd_impl(const void* q, const void* k_new, const void* v_new,
                                const void* k_sink, const void* v_sink, int sink_len,
                                const void* k_cache, const void* v_cache, int cache_cap,
                                int cache_head, int cache_len, int rope_dims, float rope_base,
                                int shift_frames, void* o, float* lse,
                                void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                                int T_chunk, int d, float scale, const mw::CommitJob& commit,
                                void* stream) {
  MW_TRY(check_dims(B, H, d));
  if (n_q_chunks < 1 || T_chunk < 1)
    return fail(MW_ERR_INVALID_ARG, "n_q_chunks=%d and T_chunk=%d must be >= 1", n_q_chunks, T_chunk);
  const long long rows = static_cast<long long>(n_q_chunks) * T_chunk;
  MW_TRY(check_rows(rows, "n_q_chunks*T_chunk"));
  MW_TRY(check_tokens(static_cast<long long>(B) * H, rows));
  if (cache_cap < 1 || cache_cap > (1 << 24))
    return fail(MW_ERR_INVALID_ARG, "cache_cap=%d out of range [1, 2^24]", cache_cap);
  if (cache_head < 0 || cache_head >= cache_cap)
    return fail(MW_ERR_INVALID_ARG, "cache_head=%d not in [0, cache_cap=%d)", cache_head, cache_cap);
  if (cache_len < 0 || cache_len > cache_cap)
    return fail(MW_ERR_INVALID_ARG, "cache_len=%d not in [0, cache_cap=%d]", cache_len, cache_cap);
  if (sink_len < 0 || sink_len > (1 << 24))
    return fail(MW_ERR_INVALID_ARG, "sink_len=%d out of range [0, 2^24]", sink_len);
  if (!(scale > 0.f)) return fail(MW_ERR_INVALID_ARG, "scale must be > 0");
  RopeArgs rope;
  if (rope_dims != 0) {
    if (rope_dims < 0 || rope_dims > d || (rope_dims & 1))
      return fail(MW_ERR_INVALID_ARG, "rope_dims=%d must be even and in [0, d=%d]", rope_dims, d);
    if (!(rope_base > 1.f) || !(rope_base < 1e30f))
      return fail(MW_ERR_INVALID_ARG, "rope_base must be > 1 and finite");
    if (shift_frames < 0 || shift_frames > (1 << 24))
      return fail(MW_ERR_INVALID_ARG, "shift_frames=%d not in [0, 2^24]", shift_frames);
    // only the sink's angles change, so without a sink or a shift this is the
    // plain forward
    if (sink_len > 0 && shift_frames > 0) {
      rope.dims = rope_dims;
      rope.omega = rope_freq(rope_dims, rope_base);
      rope.shift = shift_frames;
    }
  }
  MW_TRY(check_ptr(q, "q"));
  MW_TRY(check_ptr(k_new, "k_new"));
  MW_TRY(check_ptr(v_new, "v_new"));
  MW_TRY(check_ptr(o, "o"));
  if (cache_len > 0) {
    MW_TRY(check_ptr(k_cache, "k_cache"));
    MW_TRY(check_ptr(v_cache, "v_cache"));
  }
  if (sink_len > 0) {
    MW_TRY(check_ptr(k_sink, "k_sink"));
    MW_TRY(check_ptr(v_sink, "v_sink"));
  }
  if (lse && (reinterpret_cast<uintptr_t>(lse) & 3u))
    return fail(MW_ERR_INVALID_ARG, "lse is not 4-byte aligned");
  const int BH = B * H;
  // the split plan counts every cached key (sink and ring alike)
  const int splits = plan_splits(BH, static_cast<int>(rows), sink_len + cache_len);
  const size_t need = cache_ws_bytes(splits, BH, static_cast<int>(rows), kernel_d(d));
  if (need > 0) {
    if (workspace == nullptr || ws_bytes < need)
      return fail(MW_ERR_WORKSPACE, "workspace %zu bytes, need %zu", ws_bytes, need);
    if (reinterpret_cast<uintptr_t>(workspace) & 255u)
      return fail(MW_ERR_INVALID_ARG, "workspace is not 256-byte aligned");
  }
  return fwd_common(q, k_new, v_new, k_cache, v_cache, cache_cap, cache_head, cache_len, k_sink,
                    v_sink, sink_len, rope, o, lse, need > 0 ? workspace : nullptr, ws_bytes, BH,
                    static_cast<int>(rows), T_chunk, d, scale, splits, commit,
                    static_cast<cudaStream_t>(stream));
}

mw_status mw_bca_cache_fwd_rope(const void* q, const void* k_new, const void* v_new,
                                const void* k_sink, const void* v_sink, int sink_len,
                                const void* k_cache, const void* v_cache, int cache_cap,
                                int cache_head, int cache_len, int rope_dims, float rope_base,
                                int shift_frames, void* o, float* lse,
                                void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                                int T_chunk, int d, float scale, void* stream) {
  return cache_fwd_impl(q, k_new, v_new, k_sink, v_sink, sink_len, k_cache, v_cache, cache_cap,
                        cache_head, cache_len, rope_dims, rope_base, shift_frames,
                        o, lse, workspace, ws_bytes, B, H, n_q_chunks, T_chunk, d, scale,
                        mw::CommitJob{}, stream);
}

mw_status mw_bca_cache_step(const void* q, const void* k_new, const void* v_new, void* k_cache,
                            void* v_cache, int cache_cap, int cache_head, int cache_len,
                            int commit_slot, int commit_rows, void* o, float* lse,
                            void* workspace, size_t ws_bytes, int B, int H, int n_q_chunks,
                            int T_chunk, int d, float scale, void* stream) {
  mw::CommitJob job;
  if (commit_rows != 0) {
    const long long rows = static_cast<long long>(n_q_chunks) * T_chunk;
    if (commit_rows < 0 || commit_rows > cache_cap || commit_rows > rows)
      return fail(MW_ERR_INVALID_ARG, "commit_rows=%d not in [0, min(cache_cap, n_q_chunks*T_chunk)]",
                  commit_rows);
    if (commit_slot < 0 || commit_slot >= cache_cap)
      return fail(MW_ERR_INVALID_ARG, "commit_slot=%d not in [0, cache_cap=%d)", commit_slot,
                  cache_cap);
    MW_TRY(check_ptr(k_cache, "k_cache"));
    MW_TRY(check_ptr(v_cache, "v_cache"));
    job.kc = static_cast<__nv_bfloat16*>(k_cache);
    job.vc = static_cast<__nv_bfloat16*>(v_cache);
    job.ks = static_cast<const __nv_bfloat16*>(k_new);
    job.vs = static_cast<const __nv_bfloat16*>(v_new);
    job.cap = cache_cap;
    job.slot = commit_slot;
    job.rows = commit_rows;
    job.src_rows = static_cast<int>(rows);
    job.d = d;
    job.BH = B * H;
  }
  return cache_fwd_impl(q, k_new, v_new, nullptr, nullptr, 0, k_cache, v_cache, cache_cap,
                        cache_head, cache_len, 0, 0.f, 0, o, lse, workspace, ws_bytes, B, H,
                        n_q_chunks, T_chunk, d, scale, job, stream);
}

mw_status mw_bca_cache_commit(void* k_cache, void* v_cache, int cache_cap, int slot_start,
                              const void* k_src, const void* v_src, int rows, int B, int H, int d,
                              void* stream) {
  MW_TRY(check_dims(B, H, d));
  if (cache_cap < 1 || cache_cap > (1 << 24))
    return fail(MW_ERR_INVALID_ARG, "cache_cap=%d out of range [1, 2^24]", cache_cap);
  if (slot_start < 0 || slot_start >= cache_cap)
    return fail(MW_ERR_INVALID_ARG, "slot_start=%d not in [0, cache_cap=%d)", slot_start, cache_cap);
  if (rows < 1 || rows > cache_cap)
    return fail(MW_ERR_INVALID_ARG, "rows=%d not in [1, cache_cap=%d]", rows, cache_cap);
  MW_TRY(check_ptr(k_cache, "k_cache"));
  MW_TRY(check_ptr(v_cache, "v_cache"));
  MW_TRY(check_ptr(k_src, "k_src"));
  MW_TRY(check_ptr(v_src, "v_src"));
  DeviceScope scope(static_cast<cudaStream_t>(stream));
  MW_TRY(scope.status());
  mw::CommitJob job;
  job.kc = static_cast<__nv_bfloat16*>(k_cache);
  job.vc = static_cast<__nv_bfloat16*>(v_cache);
  job.ks = static_cast<const __nv_bfloat16*>(k_src);
  job.vs = static_cast<const __nv_bfloat16*>(v_src);
  job.cap = cache_cap;
  job.slot = slot_start;
  job.rows = rows;
  job.src_rows = rows;
  job.d = d;
  job.BH = B * H;
  return launch_status(mw::launch_commit(job, static_cast<cudaStream_t>(stream)),
                       "commit kernel launch");
}

mw_status mw_qkv_rope_split(const void* qkv, void* q, void* k, void* v, int B, int N, int H,
                            int d, int rope_dims, float rope_base, int tokens_per_frame,
                            int first_frame, void* stream) {
  MW_TRY(check_dims(B, H, d));
  MW_TRY(check_rows(N, "N"));
  MW_TRY(check_tokens(static_cast<long long>(B) * H, N));
  mw::RopeFreq omega{};
  if (rope_dims != 0) {
    if (rope_dims < 0 || rope_dims > d || (rope_dims & 1))
      return fail(MW_ERR_INVALID_ARG, "rope_dims=%d must be even and in [0, d=%d]", rope_dims, d);
    if (!(rope_base > 1.f) || !(rope_base < 1e30f))
      return fail(MW_ERR_INVALID_ARG, "rope_base must be > 1 and finite");
    if (tokens_per_frame < 1)
      return fail(MW_ERR_INVALID_ARG, "tokens_per_frame=%d must be >= 1", tokens_per_frame);
    if (first_frame < 0 ||
        static_cast<long long>(first_frame) + (N - 1) / tokens_per_frame > (1 << 24))
      return fail(MW_ERR_INVALID_ARG,
                  "first_frame=%d: frame positions must stay in [0, 2^24]", first_frame);
    omega = rope_freq(rope_dims, rope_base);
  }
  MW_TRY(check_ptr(qkv, "qkv"));
  MW_TRY(check_ptr(q, "q"));
  MW_TRY(check_ptr(k, "k"));
  MW_TRY(check_ptr(v, "v"));
  DeviceScope scope(static_cast<cudaStream_t>(stream));
  MW_TRY(scope.status());
  return launch_status(
      mw::launch_qkv_rope(static_cast<const __nv_bfloat16*>(qkv), static_cast<__nv_bfloat16*>(q),
                          static_cast<__nv_bfloat16*>(k), static_cast<__nv_bfloat16*>(v), B, N, H,
                          d, rope_dims, omega, rope_dims != 0 ? tokens_per_frame : 1,
                          rope_dims != 0 ? first_frame : 0, static_cast<cudaStream_t>(stream)),
      "qkv split kernel launch");
}

mw_status mw_device_status(void* stream, int clear) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  MW_TRY(scope.status());
  unsigned* ptr = nullptr;
  MW_TRY(status_ptr(&ptr));
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(MW_ERR_CUDA, "cudaStreamSynchronize: %s", cudaGetErrorString(e));
  unsigned word = 0;
  e = cudaMemcpy(&word, ptr, sizeof(word), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(MW_ERR_CUDA, "reading the status word: %s", cudaGetErrorString(e));
  if (clear) {
    e = cudaMemset(ptr, 0, sizeof(unsigned));
    if (e != cudaSuccess) return fail(MW_ERR_CUDA, "clearing the status word: %s", cudaGetErrorString(e));
  }
  if (word & mw::kDevTimeout) return fail(MW_ERR_TIMEOUT, "a kernel wait expired (status 0x%x)", word);
  if (word) return fail(MW_ERR_CUDA, "device status 0x%x (misaligned shared memory)", word);
  return ok();
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of the ring-cache forward.
//
// Callers that cannot allocate device memory (plugin hosts that only hand in
// their own buffers; real-time loops that must not call cudaMalloc/cudaFree,
// which can synchronise the device) get the split-KV partials from this fixed
// array instead of a caller workspace.  It is a file-scope device variable:
// every device that loads the library holds it until the process exits.  In
// host code its name is only a host-side stand-in, so its device address is
// looked up once per device with cudaGetSymbolAddress (with that device
// current) and that address is what the kernels receive.
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[MW_NOALLOC_SCRATCH_BYTES];

void* g_noalloc_ptr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device (set up on the
// first call per device).
mw_status noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(MW_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(MW_ERR_CUDA, "device index %d too large", dev);
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_noalloc_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess)
      return fail(MW_ERR_CUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(e));
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return MW_OK;
}

}  // namespace

extern "C" mw_status mw_bca_cache_fwd_noalloc(const void* q, const void* k_new, const void* v_new,
                                              const void* k_cache, const void* v_cache,
                                              int cache_cap, int cache_head, int cache_len,
                                              void* o, float* lse, int B, int H, int n_q_chunks,
                                              int T_chunk, int d, float scale, void* stream) {
  // sizes first (host only), so that an oversized request is refused before
  // anything touches the device
  MW_TRY(check_dims(B, H, d));
  if (n_q_chunks < 1 || T_chunk < 1)
    return fail(MW_ERR_INVALID_ARG, "n_q_chunks=%d and T_chunk=%d must be >= 1", n_q_chunks, T_chunk);
  const long long rows = static_cast<long long>(n_q_chunks) * T_chunk;
  MW_TRY(check_rows(rows, "n_q_chunks*T_chunk"));
  MW_TRY(check_tokens(static_cast<long long>(B) * H, rows));
  if (cache_len < 0 || cache_len > cache_cap)
    return fail(MW_ERR_INVALID_ARG, "cache_len=%d not in [0, cache_cap=%d]", cache_len, cache_cap);
  const int splits = plan_splits(B * H, static_cast<int>(rows), cache_len);
  const size_t need = cache_ws_bytes(splits, B * H, static_cast<int>(rows), kernel_d(d));
  if (need > MW_NOALLOC_SCRATCH_BYTES)
    return fail(MW_ERR_WORKSPACE,
                "these sizes need %zu bytes of split-KV scratch; the static scratch holds %u "
                "bytes (use mw_bca_cache_fwd with a caller workspace)",
                need, static_cast<unsigned>(MW_NOALLOC_SCRATCH_BYTES));
  void* scratch = nullptr;
  if (need > 0) {
    DeviceScope scope(static_cast<cudaStream_t>(stream));
    MW_TRY(scope.status());
    MW_TRY(noalloc_scratch(&scratch));
  }
  return mw_bca_cache_fwd(q, k_new, v_new, k_cache, v_cache, cache_cap, cache_head, cache_len, o,
                          lse, scratch, need > 0 ? MW_NOALLOC_SCRATCH_BYTES : 0, B, H, n_q_chunks,
                          T_chunk, d, scale, stream);
}
