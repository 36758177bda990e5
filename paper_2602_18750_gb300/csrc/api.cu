// api.cu -- the C ABI of libhill (include/hill.h): argument validation,
// workspace layout and the launch sequence of each call.
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "../../include/hill.h"
#include "hill_internal.h"

namespace hill {

// Device error word of this library (reported by hill_sync_status).
__device__ unsigned int g_error_word = 0;

namespace {

constexpr size_t kAlign = 256;
constexpr int kMaxDevices = 64;

size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

struct DeviceInfo {
  int sms = 0;
  unsigned* err = nullptr;
};

std::mutex g_mu;
DeviceInfo g_dev[kMaxDevices];
std::atomic<uint64_t> g_launches{0};

cudaError_t counted(cudaError_t e, int kernels) {
  if (e == cudaSuccess) g_launches.fetch_add((uint64_t)kernels, std::memory_order_relaxed);
  return e;
}

// Per-device constants: SM count and the device address of the error word.
cudaError_t device_info(DeviceInfo* out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceInfo& d = g_dev[dev];
  if (d.sms == 0) {
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_error_word);
    if (e != cudaSuccess) return e;
    d.err = static_cast<unsigned*>(p);
    d.sms = sms;
  }
  *out = d;
  return cudaSuccess;
}

// cuTensorMapEncodeTiled from the driver, resolved through the runtime (no
// link-time dependency on libcuda).
PFN_cuTensorMapEncodeTiled_v12000 encode_tiled() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Tiled tensor map of the key cache for hill_score_kernel: dimension 0 is the
// head dimension (contiguous, box 64 = 128 bytes, 128-byte swizzle); the
// token, KV-head and sequence dimensions follow in increasing stride order
// (so token-major caches work too), with a box of 32 tokens.
hill_status make_kmap(const hill_desc* d, const void* k, ScoreArgs* a) {
  auto fn = encode_tiled();
  if (!fn) return HILL_ERR_CUDA;
  struct Dim {
    int64_t n, stride;
    int which;  // 0 token, 1 head, 2 sequence
  } v[3] = {{d->capacity, d->k_sn, 0}, {d->num_kv_heads, d->k_sh, 1}, {d->batch, d->k_sb, 2}};
  std::stable_sort(v, v + 3, [](const Dim& x, const Dim& y) { return x.stride < y.stride; });
  cuuint64_t gdim[4] = {(cuuint64_t)kHeadDim, 1, 1, 1};
  cuuint64_t gstr[3];
  cuuint32_t box[4] = {64, 1, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  for (int i = 0; i < 3; ++i) {
    gdim[i + 1] = (cuuint64_t)std::max<int64_t>(v[i].n, 1);
    // a dimension of extent 1 may carry any stride; keep it valid and ordered
    int64_t st = v[i].stride;
    if (v[i].n <= 1) st = std::max<int64_t>(st, i ? (int64_t)gstr[i - 1] / 2 : kHeadDim);
    gstr[i] = (cuuint64_t)(st * 2);
    if (v[i].which == 0) {
      box[i + 1] = 32;
      a->kdim_tok = i + 1;
    } else if (v[i].which == 1) {
      a->kdim_head = i + 1;
    } else {
      a->kdim_seq = i + 1;
    }
  }
  for (int i = 0; i < 3; ++i)
    if (gstr[i] == 0 || (gstr[i] & 15)) return HILL_ERR_UNSUPPORTED;
  const CUtensorMapDataType dt =
      d->dtype == HILL_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  CUresult r = fn(&a->kmap, dt, 4, const_cast<void*>(k), gdim, gstr, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? HILL_OK : HILL_ERR_UNSUPPORTED;
}

// Tiled tensor map of the dense E4M3 key shadow [B][Hkv][cap][128] (one
// byte per code): box = 128 codes (one 128-byte swizzled row) x 32 tokens.
hill_status make_kmap8(const hill_desc* d, const void* k8, ScoreArgs* a) {
  auto fn = encode_tiled();
  if (!fn) return HILL_ERR_CUDA;
  const cuuint64_t cap = (cuuint64_t)std::max(d->capacity, 1), hkv = (cuuint64_t)d->num_kv_heads;
  cuuint64_t gdim[4] = {(cuuint64_t)kHeadDim, cap, hkv, (cuuint64_t)std::max(d->batch, 1)};
  cuuint64_t gstr[3] = {(cuuint64_t)kHeadDim, cap * kHeadDim, hkv * cap * kHeadDim};
  cuuint32_t box[4] = {(cuuint32_t)kHeadDim, 32, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  a->kdim_tok = 1;
  a->kdim_head = 2;
  a->kdim_seq = 3;
  CUresult r = fn(&a->kmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 4, const_cast<void*>(k8), gdim, gstr, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? HILL_OK : HILL_ERR_UNSUPPORTED;
}

// The same shadow for the tensor-core scoring: four maps whose boxes hold
// 32, 64, 96 and 128 token rows (a chunk of one to four 32-token tiles).
hill_status make_kmap8_tc(const hill_desc* d, const void* k8, ScoreTcArgs* a) {
  auto fn = encode_tiled();
  if (!fn) return HILL_ERR_CUDA;
  const cuuint64_t cap = (cuuint64_t)std::max(d->capacity, 1), hkv = (cuuint64_t)d->num_kv_heads;
  cuuint64_t gdim[4] = {(cuuint64_t)kHeadDim, cap, hkv, (cuuint64_t)std::max(d->batch, 1)};
  cuuint64_t gstr[3] = {(cuuint64_t)kHeadDim, cap * kHeadDim, hkv * cap * kHeadDim};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  for (int m = 0; m < 4; ++m) {
    cuuint32_t box[4] = {(cuuint32_t)kHeadDim, (cuuint32_t)(32 * (m + 1)), 1, 1};
    CUresult r = fn(&a->kmap[m], CU_TENSOR_MAP_DATA_TYPE_UINT8, 4, const_cast<void*>(k8), gdim, gstr, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return HILL_ERR_UNSUPPORTED;
  }
  return HILL_OK;
}

// Tiled map of the query codes [rows][128] written by hill_quantize_q_kernel:
// box = 128 codes x 16 rows (one KV head's query rows), 128-byte swizzle.
hill_status make_qmap(const void* q8, int64_t rows, ScoreTcArgs* a) {
  auto fn = encode_tiled();
  if (!fn) return HILL_ERR_CUDA;
  cuuint64_t gdim[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)std::max<int64_t>(rows, 1)};
  cuuint64_t gstr[1] = {(cuuint64_t)kHeadDim};
  cuuint32_t box[2] = {(cuuint32_t)kHeadDim, (cuuint32_t)score_tc_max_group()};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(&a->qmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(q8), gdim, gstr, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? HILL_OK : HILL_ERR_UNSUPPORTED;
}

int cap32_of(const hill_desc* d) { return (d->capacity + 31) & ~31; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool stride_ok(int64_t s) { return s >= 0 && (s % 8) == 0; }

hill_status check_desc(const hill_desc* d) {
  if (!d) return HILL_ERR_INVALID_ARG;
  if (d->batch < 0 || d->num_q_heads <= 0 || d->num_kv_heads <= 0 || d->capacity < 0 || d->head_dim <= 0)
    return HILL_ERR_INVALID_ARG;
  if (d->num_q_heads % d->num_kv_heads) return HILL_ERR_INVALID_ARG;
  if (d->dtype != HILL_F16 && d->dtype != HILL_BF16) return HILL_ERR_INVALID_ARG;
  if (!stride_ok(d->q_sb) || !stride_ok(d->q_sh) || !stride_ok(d->k_sb) || !stride_ok(d->k_sh) ||
      !stride_ok(d->k_sn) || !stride_ok(d->v_sb) || !stride_ok(d->v_sh) || !stride_ok(d->v_sn))
    return HILL_ERR_INVALID_ARG;
  if (d->head_dim != kHeadDim) return HILL_ERR_UNSUPPORTED;
  // any group size G = H / Hkv and any number of KV heads: groups of more
  // than 8 query heads and more than score_max_kv_heads() KV heads run in
  // passes (head_passes)
  if (d->batch > score_max_batch() || d->batch > attn_max_batch()) return HILL_ERR_UNSUPPORTED;
  // the selection keeps a sequence's keys on chip across at most 8 CTAs
  if (select_smem_bytes(d->capacity, select_cluster_size(d->capacity)) > 220 * 1024)
    return HILL_ERR_UNSUPPORTED;
  return HILL_OK;
}

struct Layout {
  size_t scores, logits, partials, stats, hist0, attn_part, q8, sq, total;
  bool has_hist0;
  int score_grid, attn_grid, splits;
  int score_spc;   // ATTN partial slots per scoring CTA
};

// The scoring kernel's grid: one CTA per SM, or in the split step
// (split_grid) 17/20 of them, so that the normalisation and selection of the
// previous layer find whole SMs beside the K stream.  Measured on the 32K and
// 128K workloads: the 16-bit stream, bound by HBM, is as fast on 4/5 or 17/20
// of the SMs and slower on 9/10; the E4M3 stream, bound by the latency of its
// per-tile chain, gains with every SM (4/5: 80 / 48 us per layer, 17/20: 76 /
// 45, 9/10: 74 / 45).  One fraction for both, since end() must find the
// partial slots that begin() wrote without knowing the key format.
int score_grid_for(const hill_desc* d, int sms, bool split_grid = false) {
  const int T = score_tile_tokens();
  const long long items = (long long)d->batch * ((d->capacity + T - 1) / T);
  long long g = split_grid ? sms * 17 / 20 : sms;
  if (items < g) g = items;
  return g < 1 ? 1 : (int)g;
}

// Workspace regions of a call.  score_only: hill_score and its variants,
// which write the caller's scores and run no selection or attention, need
// only the ATTN normalisation's logits, partials and statistics.  e4m3_query:
// room for the query codes and scales of the tensor-core E4M3 scoring (every
// layout but the allocation-free entry point's, which scores 16-bit keys).
Layout layout_for(const hill_desc* d, int mode, int max_k, int sms, bool score_only = false,
                  bool split_grid = false, bool e4m3_query = true) {
  Layout L{};
  const size_t B = d->batch, H = d->num_q_heads, cap = d->capacity;
  L.score_grid = score_grid_for(d, sms, split_grid);
  // few KV heads with large groups (MQA-like): the scoring kernel deals the
  // tiles to several warps per head, each with its own partial slot (more
  // than score_max_kv_heads() KV heads run in passes of at least half that)
  L.score_spc = d->num_kv_heads > score_max_kv_heads()
                    ? 1
                    : score_deal_warps(d->num_kv_heads, d->num_q_heads / d->num_kv_heads);
  L.attn_grid = sms;
  L.splits = score_only ? 0 : attn_max_segments(max_k < 0 ? 0 : max_k);
  size_t off = 0;
  // the step's scores when the caller passes none
  L.scores = off;
  if (!score_only) off += align_up(B * cap * sizeof(float));
  // logits, rows padded to 32 tokens (one 128-byte line per warp and head)
  L.logits = off;
  if (mode == HILL_SCORE_ATTN) off += align_up(B * H * (size_t)cap32_of(d) * sizeof(float));
  L.partials = off;
  if (mode == HILL_SCORE_ATTN) off += align_up(B * (size_t)L.score_grid * L.score_spc * H * sizeof(float2));
  // combined (max, 1/sum) per (b, h), when the normalisation runs in two kernels
  L.stats = off;
  if (mode == HILL_SCORE_ATTN) off += align_up(B * H * sizeof(float2));
  // leading-digit histogram of the selection key, built by the ATTN
  // normalisation when a selection follows (max_k > 0)
  L.hist0 = off;
  L.has_hist0 = mode == HILL_SCORE_ATTN && max_k > 0 && !score_only;
  if (L.has_hist0) off += align_up(B * (size_t)select_hist_bins() * sizeof(uint32_t));
  L.attn_part = off;
  off += align_up(B * H * (size_t)L.splits * (2 + kHeadDim) * sizeof(float));
  // E4M3 query codes [B][Hkv][16][128] and scales [B][H]
  L.q8 = off;
  if (e4m3_query) off += align_up(B * (size_t)d->num_kv_heads * score_tc_max_group() * kHeadDim);
  L.sq = off;
  if (e4m3_query) off += align_up(B * H * sizeof(float));
  L.total = off + kAlign;  // room to align the caller's base pointer
  return L;
}

unsigned char* ws_base(void* ws) {
  uintptr_t p = reinterpret_cast<uintptr_t>(ws);
  return reinterpret_cast<unsigned char*>((p + kAlign - 1) & ~(uintptr_t)(kAlign - 1));
}

hill_status from_cuda(cudaError_t e) { return e == cudaSuccess ? HILL_OK : HILL_ERR_CUDA; }

// The power of two at or above n: the kernels' group template for a pass of
// n query heads per KV head.
int pow2_at_least(int n) {
  int p = 1;
  while (p < n) p <<= 1;
  return p;
}

// The launches a scoring or attention call makes over the heads: passes of
// at most score_max_kv_heads() KV heads (balanced), times passes of at most
// `per_pass` query heads of each group (the last one takes the rest).
// f(goff, nkv, hoff, Gn, first) is called once per pass.
template <typename F>
hill_status head_passes(const hill_desc* d, bool kv_split, F&& f, int per_pass = 8) {
  const int Hkv = d->num_kv_heads, G = d->num_q_heads / d->num_kv_heads;
  const int cap_kv = score_max_kv_heads();
  const int kp = kv_split ? (Hkv + cap_kv - 1) / cap_kv : 1;
  bool first = true;
  for (int p = 0; p < kp; ++p) {
    const int g0 = (int)((int64_t)p * Hkv / kp), g1 = (int)((int64_t)(p + 1) * Hkv / kp);
    for (int h0 = 0; h0 < G; h0 += per_pass) {
      const hill_status s = f(g0, g1 - g0, h0, std::min(per_pass, G - h0), first);
      if (s != HILL_OK) return s;
      first = false;
    }
  }
  return HILL_OK;
}

// Which part of the scoring stage run_score launches: all of it, the K
// stream only (the scoring kernel), or the ATTN normalisation only.
constexpr int kScoreAll = 0, kScoreStream = 1, kScoreNormalise = 2;

hill_status run_score(const hill_desc* d, const void* q, const void* k, const int32_t* lens, int mode,
                      float* scores, float* accum, unsigned char* base, const Layout& L,
                      const DeviceInfo& di, cudaStream_t st, uint32_t* hist0 = nullptr, int recent = 0,
                      const float* kscale = nullptr, bool kvh = false, int part = kScoreAll) {
  if (d->batch == 0 || d->capacity == 0) return HILL_OK;
  const int G = d->num_q_heads / d->num_kv_heads;
  ScoreArgs a{};
  a.q = q;
  a.k = k;
  a.lens = lens;
  a.B = d->batch;
  a.H = d->num_q_heads;
  a.Hkv = d->num_kv_heads;
  a.cap = d->capacity;
  a.q_sb = d->q_sb;
  a.q_sh = d->q_sh;
  a.k_sb = d->k_sb;
  a.k_sh = d->k_sh;
  a.k_sn = d->k_sn;
  a.nslot = L.score_grid * L.score_spc;
  a.err = di.err;
  // kscale != NULL: k is the E4M3 shadow of the keys (asymmetric-precision scoring)
  const bool f8 = kscale != nullptr;
  if (part != kScoreNormalise) {   // the normalisation alone reads no keys
    const hill_status ms = f8 ? make_kmap8(d, k, &a) : make_kmap(d, k, &a);
    if (ms != HILL_OK) return ms;
  }
  a.kscale = kscale;
  a.cap32 = cap32_of(d);
  const bool raw = mode == HILL_SCORE_RAW;
  a.kvh = kvh ? 1 : 0;
  if (raw) {
    a.scores = scores;
    a.accum = accum;
  } else {
    a.logits = reinterpret_cast<float*>(base + L.logits);
    a.lstride = cap32_of(d);
    a.partials = reinterpret_cast<float2*>(base + L.partials);
    a.hist0 = hist0;
    a.hist0_words = (int64_t)d->batch * select_hist_bins();
  }
  // more than score_max_kv_heads() KV heads are scored in passes over their
  // own keys (RAW passes after the first add their sums); groups of more than
  // 8 query heads are scored in passes over the same keys, except by the
  // dealing kernel, which scores up to 32 query heads (four sub-groups of 8)
  // from every key tile; the kernel's group template is the power of two at
  // or above the pass's heads (8 for the dealing kernel)
  const bool deal = L.score_spc > 1;
  a.Gs = G;
  // E4M3 scoring on the tensor cores' native 8-bit path (score_tc.cu) for
  // per-sequence importance with 2 to 16 query heads per KV head (at most
  // score_tc_max_heads() in all, one pass over the KV heads) and at least
  // 64 MB of codes per call; measured against the warp-level kernel, in
  // evaluation + selection per layer: one query head per KV head (4K and 32K
  // MHA) 35.5 / 75.9 us there against 43.5 / 83.3 here; two heads (32K) 63.7
  // against 50.4; four (32K, 128K) 39.9 / 45.5 against 36.8 / 35.9; four at
  // 4K (34 MB of codes) 20.3 against 23.2.  Per-KV-head importance and the
  // dealing layouts keep the warp-level kernel too.
  const bool tc = f8 && !kvh && !deal && G >= 2 && G <= score_tc_max_group() &&
                  d->num_kv_heads <= score_max_kv_heads() && d->num_q_heads <= score_tc_max_heads() &&
                  (int64_t)d->batch * d->capacity * d->num_kv_heads * kHeadDim >= ((int64_t)64 << 20);
  if (part != kScoreNormalise && tc) {
    QuantQArgs qq{};
    qq.q = q;
    qq.q_sb = d->q_sb;
    qq.q_sh = d->q_sh;
    qq.B = d->batch;
    qq.H = d->num_q_heads;
    qq.Hkv = d->num_kv_heads;
    qq.G = G;
    qq.q8 = reinterpret_cast<uint8_t*>(base + L.q8);
    qq.sq = reinterpret_cast<float*>(base + L.sq);
    ScoreTcArgs t{};
    hill_status ms = make_kmap8_tc(d, k, &t);
    if (ms == HILL_OK) ms = make_qmap(qq.q8, (int64_t)d->batch * d->num_kv_heads * score_tc_max_group(), &t);
    if (ms != HILL_OK) return ms;
    t.kscale = kscale;
    t.cap32 = cap32_of(d);
    t.sq = qq.sq;
    t.lens = lens;
    t.B = d->batch;
    t.H = d->num_q_heads;
    t.Hkv = d->num_kv_heads;
    t.cap = d->capacity;
    t.G = G;
    t.goff = 0;
    t.nkv = d->num_kv_heads;
    t.scores = a.scores;
    t.accum = a.accum;
    t.logits = a.logits;
    t.lstride = a.lstride;
    t.partials = a.partials;
    t.nslot = a.nslot;
    t.hist0 = a.hist0;
    t.hist0_words = a.hist0_words;
    t.err = a.err;
    hill_status ts = from_cuda(counted(launch_quantize_q(qq, d->dtype, st), 1));
    if (ts == HILL_OK) ts = from_cuda(counted(launch_score_tc(t, raw, L.score_grid, st), 1));
    if (ts != HILL_OK || raw || part == kScoreStream) return ts;
  }
  hill_status s = part == kScoreNormalise || tc ? HILL_OK : head_passes(d, true, [&](int goff, int nkv, int hoff,
                                                                                      int Gn, bool first) {
    a.goff = goff;
    a.nkv = nkv;
    a.hoff = hoff;
    a.Gn = Gn;
    // RAW passes add to what an earlier pass stored in the same rows: every
    // pass shares the per-sequence rows (b, j), but a per-KV-head row (b, g, j)
    // is shared only by the query-head passes of KV head g (hoff > 0), so a
    // later KV-head pass stores into rows no pass has written yet
    a.raw_add = kvh ? (hoff > 0 ? 1 : 0) : (first ? 0 : 1);
    // the dealing kernel exists for the group template 8 (it is chosen for
    // groups of 5 or more heads)
    return from_cuda(
        counted(launch_score(a, d->dtype, deal ? 8 : pow2_at_least(Gn), raw, f8, deal, L.score_grid, st), 1));
  }, deal ? 4 * 8 : 8);
  if (s != HILL_OK || raw || part == kScoreStream) return s;
  FinalizeArgs f{};
  f.logits = a.logits;
  f.lstride = a.lstride;
  f.partials = a.partials;
  f.lens = lens;
  f.B = d->batch;
  f.H = d->num_q_heads;
  f.cap = d->capacity;
  f.nslot = L.score_grid * L.score_spc;
  f.spc = L.score_spc;
  f.scores = scores;
  f.accum = accum;
  f.hist0 = hist0;
  f.recent = recent;
  f.kvh = kvh ? 1 : 0;
  f.Hkv = d->num_kv_heads;
  f.stats = reinterpret_cast<float2*>(base + L.stats);
  int kernels = 0;
  // the split step's normalisation takes the two-kernel form, whose finalize
  // kernel fits beside a scoring CTA on one SM
  const cudaError_t e = launch_attn_finalize(f, di.sms, st, &kernels, part == kScoreNormalise);
  return from_cuda(counted(e, kernels));
}

hill_status run_select(const hill_desc* d, const float* key, const int32_t* lens, const int32_t* k,
                       int max_k, int32_t* idx, int32_t* count, const DeviceInfo& di, cudaStream_t st,
                       const uint32_t* hist0 = nullptr, int recent = 0, uint16_t* hits = nullptr,
                       bool kvh = false) {
  if (d->batch == 0) return HILL_OK;
  SelectArgs a{};
  a.key = key;
  a.lens = lens;
  a.k = k;
  a.B = d->batch;
  a.cap = d->capacity;
  a.max_k = max_k;
  a.idx = idx;
  a.count = count;
  a.hist0 = hist0;
  a.recent = recent;
  a.hits = hits;
  a.rows_per_seq = kvh ? d->num_kv_heads : 1;
  a.err = di.err;
  return from_cuda(counted(launch_select(a, st), 1));
}

hill_status run_attn(const hill_desc* d, const void* q, const void* k, const void* v, const int32_t* idx,
                     const int32_t* count, int max_k, float* out, unsigned char* base, const Layout& L,
                     const DeviceInfo& di, cudaStream_t st,
                     bool kvh = false) {
  if (d->batch == 0) return HILL_OK;
  // the gather forms row offsets as 32-bit stride x 32-bit index products
  if (d->k_sn > INT32_MAX || d->v_sn > INT32_MAX) return HILL_ERR_UNSUPPORTED;
  AttnArgs a{};
  a.q = q;
  a.k = k;
  a.v = v;
  a.idx = idx;
  a.count = count;
  a.B = d->batch;
  a.H = d->num_q_heads;
  a.Hkv = d->num_kv_heads;
  a.cap = d->capacity;
  a.max_k = max_k;
  a.q_sb = d->q_sb;
  a.q_sh = d->q_sh;
  a.k_sb = d->k_sb;
  a.k_sh = d->k_sh;
  a.k_sn = d->k_sn;
  a.v_sb = d->v_sb;
  a.v_sh = d->v_sh;
  a.v_sn = d->v_sn;
  a.out = out;
  a.part = reinterpret_cast<float*>(base + L.attn_part);
  a.splits = L.splits;
  a.kvh = kvh ? 1 : 0;
  a.err = di.err;
  // G > 16 query heads per KV head: passes of at most 16 heads over the same
  // selected rows, then one merge of the split partials over all heads
  const int G = d->num_q_heads / d->num_kv_heads;
  a.Gs = G;
  return head_passes(d, false, [&](int, int, int hoff, int Gn, bool) {
    a.hoff = hoff;
    a.Gn = Gn;
    const bool last = hoff + Gn == G;
    return from_cuda(
        counted(launch_sparse_attn(a, d->dtype, pow2_at_least(Gn), L.attn_grid, last, st), last ? 2 : 1));
  }, 16);
}

}  // namespace
}  // namespace hill

using namespace hill;

extern "C" {

int32_t hill_abi_version(void) { return 100; }

uint64_t hill_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

const char* hill_status_string(hill_status s) {
  switch (s) {
    case HILL_OK: return "HILL_OK";
    case HILL_ERR_INVALID_ARG: return "HILL_ERR_INVALID_ARG";
    case HILL_ERR_UNSUPPORTED: return "HILL_ERR_UNSUPPORTED";
    case HILL_ERR_WORKSPACE: return "HILL_ERR_WORKSPACE";
    case HILL_ERR_CUDA: return "HILL_ERR_CUDA";
    case HILL_ERR_TIMEOUT: return "HILL_ERR_TIMEOUT";
    case HILL_ERR_DEVICE: return "HILL_ERR_DEVICE";
  }
  return "HILL_ERR_UNKNOWN";
}

size_t hill_workspace_bytes(const hill_desc* desc, hill_score_mode mode, int32_t max_k) {
  if (check_desc(desc) != HILL_OK) return 0;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return 0;
  if (max_k < 0) return 0;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return 0;
  return layout_for(desc, mode, max_k, di.sms).total;
}

hill_status hill_score(const hill_desc* desc, const void* q, const void* k_cache, const int32_t* lens,
                       hill_score_mode mode, float* scores, float* accum, void* ws, size_t ws_bytes,
                       void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (!q || !k_cache || !lens || !scores) return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_cache)) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, 0, di.sms, true);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  return run_score(desc, q, k_cache, lens, mode, scores, accum, ws_base(ws), L, di,
                   static_cast<cudaStream_t>(stream));
}

hill_status hill_topk_select(const hill_desc* desc, const float* scores, const int32_t* lens, const int32_t* k,
                             int32_t max_k, int32_t* idx, int32_t* count, void* ws, size_t ws_bytes,
                             void* stream) {
  (void)ws;
  (void)ws_bytes;
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (max_k < 0 || !scores || !lens || !k || !count || (max_k > 0 && !idx)) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  return run_select(desc, scores, lens, k, max_k, idx, count, di, static_cast<cudaStream_t>(stream));
}

hill_status hill_gather_sparse_attn(const hill_desc* desc, const void* q, const void* k_cache,
                                    const void* v_cache, const int32_t* idx, const int32_t* count,
                                    int32_t max_k, float* out, void* ws, size_t ws_bytes, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (max_k < 0 || !q || !k_cache || !v_cache || !count || !out || (max_k > 0 && !idx))
    return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache)) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, HILL_SCORE_RAW, max_k, di.sms);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  return run_attn(desc, q, k_cache, v_cache, idx, count, max_k, out, ws_base(ws), L, di,
                  static_cast<cudaStream_t>(stream));
}

static hill_status evict_step(const hill_desc* desc, const void* q, const void* k_cache, const void* v_cache,
                              const int32_t* lens, const int32_t* k, int32_t recent, int32_t max_k,
                              hill_score_mode mode, float* accum, float* scores, int32_t* idx, int32_t* count,
                              uint16_t* hits, float* out, void* ws, size_t ws_bytes, void* stream,
                              const uint8_t* k8 = nullptr, const float* kscale = nullptr) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (max_k < 0 || recent < 0 || !q || !lens || !k || !count || (max_k > 0 && !idx)) return HILL_ERR_INVALID_ARG;
  if (k8 ? (!kscale || !aligned16(k8) || !aligned16(kscale)) : !k_cache) return HILL_ERR_INVALID_ARG;
  if (out && (!k_cache || !v_cache)) return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || (k_cache && !aligned16(k_cache)) || (out && !aligned16(v_cache)))
    return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, max_k, di.sms);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  unsigned char* base = ws_base(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* s_out = scores ? scores : (accum ? nullptr : reinterpret_cast<float*>(base + L.scores));
  // ATTN: the normalisation also counts the leading key digit for the selection
  uint32_t* hist0 = L.has_hist0 ? reinterpret_cast<uint32_t*>(base + L.hist0) : nullptr;
  s = run_score(desc, q, k8 ? static_cast<const void*>(k8) : k_cache, lens, mode, s_out, accum, base, L, di, st,
                hist0, recent, kscale);
  if (s != HILL_OK) return s;
  const float* key = accum ? accum : s_out;
  s = run_select(desc, key, lens, k, max_k, idx, count, di, st, hist0, recent, hits);
  if (s != HILL_OK || !out) return s;
  return run_attn(desc, q, k_cache, v_cache, idx, count, max_k, out, base, L, di, st);
}

hill_status hill_evict_step(const hill_desc* desc, const void* q, const void* k_cache, const void* v_cache,
                            const int32_t* lens, const int32_t* k, int32_t max_k, hill_score_mode mode,
                            float* accum, float* scores, int32_t* idx, int32_t* count, float* out, void* ws,
                            size_t ws_bytes, void* stream) {
  return evict_step(desc, q, k_cache, v_cache, lens, k, 0, max_k, mode, accum, scores, idx, count, nullptr, out,
                    ws, ws_bytes, stream);
}

hill_status hill_evict_step_bkp(const hill_desc* desc, const void* q, const void* k_cache, const void* v_cache,
                                const int32_t* lens, const int32_t* k, int32_t recent, int32_t max_k,
                                hill_score_mode mode, float* accum, float* scores, int32_t* idx, int32_t* count,
                                uint16_t* hits, float* out, void* ws, size_t ws_bytes, void* stream) {
  return evict_step(desc, q, k_cache, v_cache, lens, k, recent, max_k, mode, accum, scores, idx, count, hits, out,
                    ws, ws_bytes, stream);
}

hill_status hill_topk_select_bkp(const hill_desc* desc, const float* scores, const int32_t* lens,
                                 const int32_t* k, int32_t recent, int32_t max_k, int32_t* idx, int32_t* count,
                                 uint16_t* hits, void* ws, size_t ws_bytes, void* stream) {
  (void)ws;
  (void)ws_bytes;
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (max_k < 0 || recent < 0 || !scores || !lens || !k || !count || (max_k > 0 && !idx))
    return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  return run_select(desc, scores, lens, k, max_k, idx, count, di, static_cast<cudaStream_t>(stream), nullptr,
                    recent, hits);
}

}  // extern "C"

namespace {
// The K stream of the split step, from the 16-bit cache (kscale NULL) or from
// its E4M3 shadow (k = the codes, kscale = the row scales).
hill_status evict_step_begin(const hill_desc* desc, const void* q, const void* k, const float* kscale,
                             const int32_t* lens, int32_t max_k, hill_score_mode mode, float* accum, float* scores,
                             void* ws, size_t ws_bytes, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (max_k < 0 || !q || !k || !lens) return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || (kscale && !aligned16(kscale))) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, max_k, di.sms, false, true);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  unsigned char* base = ws_base(ws);
  float* s_out = scores ? scores : (accum ? nullptr : reinterpret_cast<float*>(base + L.scores));
  uint32_t* hist0 = L.has_hist0 ? reinterpret_cast<uint32_t*>(base + L.hist0) : nullptr;
  return run_score(desc, q, k, lens, mode, s_out, accum, base, L, di, static_cast<cudaStream_t>(stream), hist0, 0,
                   kscale, false, kScoreStream);
}
}  // namespace

extern "C" {

hill_status hill_evict_step_begin(const hill_desc* desc, const void* q, const void* k_cache, const int32_t* lens,
                                  int32_t max_k, hill_score_mode mode, float* accum, float* scores, void* ws,
                                  size_t ws_bytes, void* stream) {
  return evict_step_begin(desc, q, k_cache, nullptr, lens, max_k, mode, accum, scores, ws, ws_bytes, stream);
}

hill_status hill_evict_step_begin_f8(const hill_desc* desc, const void* q, const uint8_t* k8, const float* kscale,
                                     const int32_t* lens, int32_t max_k, hill_score_mode mode, float* accum,
                                     float* scores, void* ws, size_t ws_bytes, void* stream) {
  if (!k8 || !kscale) return HILL_ERR_INVALID_ARG;
  return evict_step_begin(desc, q, k8, kscale, lens, max_k, mode, accum, scores, ws, ws_bytes, stream);
}

hill_status hill_evict_step_end(const hill_desc* desc, const int32_t* lens, const int32_t* k, int32_t recent,
                                int32_t max_k, hill_score_mode mode, float* accum, float* scores, int32_t* idx,
                                int32_t* count, uint16_t* hits, void* ws, size_t ws_bytes, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (max_k < 0 || recent < 0 || !lens || !k || !count || (max_k > 0 && !idx)) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, max_k, di.sms, false, true);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  unsigned char* base = ws_base(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* s_out = scores ? scores : (accum ? nullptr : reinterpret_cast<float*>(base + L.scores));
  uint32_t* hist0 = L.has_hist0 ? reinterpret_cast<uint32_t*>(base + L.hist0) : nullptr;
  if (mode == HILL_SCORE_ATTN) {
    s = run_score(desc, nullptr, nullptr, lens, mode, s_out, accum, base, L, di, st, hist0, recent, nullptr, false,
                  kScoreNormalise);
    if (s != HILL_OK) return s;
  }
  return run_select(desc, accum ? accum : s_out, lens, k, max_k, idx, count, di, st, hist0, recent, hits);
}

hill_status hill_evict_step_kvh(const hill_desc* desc, const void* q, const void* k_cache, const void* v_cache,
                                const int32_t* lens, const int32_t* k, int32_t max_k, hill_score_mode mode,
                                float* accum, float* scores, int32_t* idx, int32_t* count, float* out, void* ws,
                                size_t ws_bytes, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (max_k < 0 || !q || !k_cache || !lens || !k || !count || (max_k > 0 && !idx) || (!scores && !accum))
    return HILL_ERR_INVALID_ARG;
  if (out && !v_cache) return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_cache) || (out && !aligned16(v_cache))) return HILL_ERR_INVALID_ARG;
  // the attention keeps one table entry per (b, g) on chip
  if ((int64_t)desc->batch * desc->num_kv_heads > attn_max_batch()) return HILL_ERR_UNSUPPORTED;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, max_k, di.sms);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  unsigned char* base = ws_base(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  s = run_score(desc, q, k_cache, lens, mode, scores, accum, base, L, di, st, nullptr, 0, nullptr, true);
  if (s != HILL_OK) return s;
  s = run_select(desc, accum ? accum : scores, lens, k, max_k, idx, count, di, st, nullptr, 0, nullptr, true);
  if (s != HILL_OK || !out) return s;
  return run_attn(desc, q, k_cache, v_cache, idx, count, max_k, out, base, L, di, st, true);
}

hill_status hill_quantize_k(const hill_desc* desc, const void* k_cache, const int32_t* row_begin,
                            const int32_t* row_end, int32_t max_rows, uint8_t* k8, float* kscale, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (!k_cache || !row_begin || !row_end || !k8 || !kscale || max_rows < 0) return HILL_ERR_INVALID_ARG;
  if (!aligned16(k_cache) || !aligned16(k8) || !aligned16(kscale)) return HILL_ERR_INVALID_ARG;
  if (desc->batch == 0 || desc->capacity == 0 || max_rows == 0) return HILL_OK;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  QuantArgs a{};
  a.k = k_cache;
  a.row_begin = row_begin;
  a.row_end = row_end;
  a.B = desc->batch;
  a.Hkv = desc->num_kv_heads;
  a.cap = desc->capacity;
  a.cap32 = cap32_of(desc);
  a.k_sb = desc->k_sb;
  a.k_sh = desc->k_sh;
  a.k_sn = desc->k_sn;
  a.k8 = k8;
  a.kscale = kscale;
  return from_cuda(counted(launch_quantize_k(a, desc->dtype, std::min(max_rows, desc->capacity),
                                             static_cast<cudaStream_t>(stream)), 1));
}

hill_status hill_score_f8(const hill_desc* desc, const void* q, const uint8_t* k8, const float* kscale,
                          const int32_t* lens, hill_score_mode mode, float* scores, float* accum, void* ws,
                          size_t ws_bytes, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (!q || !k8 || !kscale || !lens || !scores) return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k8) || !aligned16(kscale)) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, 0, di.sms, true);
  if (!ws || ws_bytes < L.total) return HILL_ERR_WORKSPACE;
  return run_score(desc, q, k8, lens, mode, scores, accum, ws_base(ws), L, di, static_cast<cudaStream_t>(stream),
                   nullptr, 0, kscale);
}

hill_status hill_evict_step_f8(const hill_desc* desc, const void* q, const uint8_t* k8, const float* kscale,
                               const void* k_cache, const void* v_cache, const int32_t* lens, const int32_t* k,
                               int32_t max_k, hill_score_mode mode, float* accum, float* scores, int32_t* idx,
                               int32_t* count, float* out, void* ws, size_t ws_bytes, void* stream) {
  if (!k8 || !kscale) return HILL_ERR_INVALID_ARG;
  return evict_step(desc, q, k_cache, v_cache, lens, k, 0, max_k, mode, accum, scores, idx, count, nullptr, out,
                    ws, ws_bytes, stream, k8, kscale);
}

hill_status hill_selftest_wait(uint32_t limit_us, void* stream) {
  if (limit_us == 0 || limit_us > 1000000u) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  return from_cuda(counted(launch_selftest_wait(1000ull * limit_us, di.err, static_cast<cudaStream_t>(stream)), 1));
}

hill_status hill_sync_status(void* stream) {
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return HILL_ERR_CUDA;
  unsigned w = 0;
  if (cudaMemcpy(&w, di.err, sizeof(w), cudaMemcpyDeviceToHost) != cudaSuccess) return HILL_ERR_CUDA;
  if (w) {
    const unsigned zero = 0;
    if (cudaMemcpy(di.err, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess) return HILL_ERR_CUDA;
  }
  if (w & kErrTimeout) return HILL_ERR_TIMEOUT;
  if (w & kErrDevArg) return HILL_ERR_DEVICE;
  return HILL_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// hill_score_noalloc: hill_score with its scratch in a fixed device array, for
// callers that cannot allocate device memory (see include/hill.h).
namespace hill {
namespace {

// The scratch of hill_score_noalloc.  Every GPU that loads this library
// holds these bytes until the process exits; all calls share them.
static __device__ __align__(256) unsigned char g_score_scratch[HILL_SCORE_NOALLOC_MAX_SCRATCH];

void* g_scratch_dev[kMaxDevices];

// Device address of g_score_scratch on the current device, looked up once per
// device (host code cannot use the symbol itself as a device address).
cudaError_t score_scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_score_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_dev[dev] = p;
  }
  *out = g_scratch_dev[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace hill

extern "C" hill_status hill_score_noalloc(const hill_desc* desc, const void* q, const void* k_cache,
                                          const int32_t* lens, hill_score_mode mode, float* scores,
                                          float* accum, void* stream) {
  hill_status s = check_desc(desc);
  if (s != HILL_OK) return s;
  if (mode != HILL_SCORE_ATTN && mode != HILL_SCORE_RAW) return HILL_ERR_INVALID_ARG;
  if (!q || !k_cache || !lens || !scores) return HILL_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_cache)) return HILL_ERR_INVALID_ARG;
  DeviceInfo di;
  if (device_info(&di) != cudaSuccess) return HILL_ERR_CUDA;
  const Layout L = layout_for(desc, mode, 0, di.sms, true, false, false);
  // the array is already 256-byte aligned: the alignment slack is not needed
  if (L.total - kAlign > (size_t)HILL_SCORE_NOALLOC_MAX_SCRATCH) return HILL_ERR_WORKSPACE;
  void* scratch = nullptr;
  if (score_scratch_address(&scratch) != cudaSuccess) return HILL_ERR_CUDA;
  return run_score(desc, q, k_cache, lens, mode, scores, accum, static_cast<unsigned char*>(scratch), L, di,
                   static_cast<cudaStream_t>(stream));
}
