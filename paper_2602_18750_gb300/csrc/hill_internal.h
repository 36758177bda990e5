// hill_internal.h -- argument blocks and launchers shared between the API
// translation unit (api.cu) and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hill_common.cuh"

namespace hill {

struct ScoreArgs {
  CUtensorMap kmap;   // K cache: 4-D tiled map, 128-byte swizzle, box = 64 dims x kT tokens
                      // (E4M3 shadow: box = 128 codes x kT tokens)
  const float* kscale;   // E4M3 shadow: [B][Hkv][cap32] row scales
  int cap32;
  int kdim_tok, kdim_head, kdim_seq;   // which tensor-map dimension holds token, KV head, sequence
  const void* q;
  const void* k;
  const int32_t* lens;
  int B, H, Hkv, cap;
  int64_t q_sb, q_sh, k_sb, k_sh, k_sn;
  float* scores;      // RAW: per-token sums, may be NULL when accum is given
  float* accum;       // RAW: running importance (+=), may be NULL
  float* logits;      // ATTN: [B][H][lstride] (lstride = cap rounded up to 32: a warp's 32 tokens of a head fill one 128-byte line)
  int64_t lstride;
  float2* partials;   // ATTN: [B][nslot][H] (max, sum 2^(z2 - max)), base-2 logits z2 = z * log2 e
  int nslot;          // = grid size of the launch x score_deal_warps(nkv, G) (one slot per warp share)
  int kvh;            // RAW with per-KV-head selection: scores/accum [B][Hkv][cap], summed over each group only
  // Query heads per KV head in the data (Gs), the first one this launch
  // handles (hoff) and how many (Gn, at most the kernel's template group G,
  // the rows past Gn being zero): a launch covers heads g * Gs + hoff +
  // [0, Gn) of the KV heads g in [goff, goff + nkv).  Groups of more than 8
  // heads are scored in passes of at most 8 (the dealing kernel: 32), and more
  // than 32 KV heads in passes of at most 32; RAW passes after the first add
  // to scores (raw_add) instead of storing.
  int Gs, hoff, Gn, goff, nkv, raw_add;
  uint32_t* hist0;    // optional: zero-filled here (hist0_words words) for the normalisation to count into
  int64_t hist0_words;
  unsigned* err;
};

struct FinalizeArgs {
  const float* logits;   // [B][H][lstride]; every line read is discarded from L2 afterwards (dead data)
  int64_t lstride;
  const float2* partials;
  const int32_t* lens;
  int B, H, cap, nslot;
  int spc;            // partial slots per scoring CTA (nslot = CTAs x spc)
  float* scores;      // may be NULL when accum is given
  float* accum;       // may be NULL
  uint32_t* hist0;    // optional [B][2048]: counts of the leading 11-bit digit of the selection key
  int recent;         // tokens j >= len - min(recent, len) are left out of hist0 (pinned, not ranked)
  int kvh;            // 1: scores/accum are [B][Hkv][cap], the sum over each KV head's G query heads
  int Hkv;
  float2* stats;      // [B][H] (max, 1/sum) per head, or NULL: every finalize CTA combines the partials
  int tpt;            // blocks of 256 tokens per finalize CTA (set by the launcher)
};

// The E4M3 scoring on the tensor cores' native 8-bit path (score_tc.cu):
// the K stream of ScoreArgs for E4M3 shadows, per-sequence ATTN or RAW, one
// pass over at most score_max_kv_heads() KV heads with at most 16 query heads
// each.
struct ScoreTcArgs {
  CUtensorMap kmap[4];   // codes [B][Hkv][cap][128]: 4-D maps (128, cap, Hkv, B), boxes of 128 codes x 32, 64, 96, 128 rows, 128-byte swizzle
  CUtensorMap qmap;   // query codes [B*Hkv*16][128]: 2-D map, box 128 x 16 rows, 128-byte swizzle
  const float* kscale;   // [B][Hkv][cap32] row scales
  int cap32;
  const float* sq;    // [B][H] query scales
  const int32_t* lens;
  int B, H, Hkv, cap, G, goff, nkv;
  float* scores;      // RAW: per-token sums (may be NULL when accum is given)
  float* accum;       // RAW: running importance (+=), may be NULL
  float* logits;      // ATTN: [B][H][lstride]
  int64_t lstride;
  float2* partials;   // ATTN: [B][nslot][H] (max, sum 2^(z2 - max)), one slot per CTA meeting the sequence
  int nslot;
  uint32_t* hist0;    // optional: zero-filled here for the normalisation to count into
  int64_t hist0_words;
  unsigned* err;
};

// Query rows cast to E4M3 for the tensor-core scoring: q8[(b*Hkv + g)*16 + r]
// holds query head g*G + r (rows r >= G zero), sq[b*H + h] its scale.
struct QuantQArgs {
  const void* q;
  int64_t q_sb, q_sh;
  int B, H, Hkv, G;
  uint8_t* q8;
  float* sq;
};

struct QuantArgs {
  const void* k;              // 16-bit K cache, strides k_sb, k_sh, k_sn
  const int32_t* row_begin;   // [B] rows [row_begin[b], row_end[b]) are quantised
  const int32_t* row_end;
  int B, Hkv, cap, cap32;     // cap32 = cap rounded up to 32 (row length of kscale)
  int64_t k_sb, k_sh, k_sn;
  uint8_t* k8;                // [B][Hkv][cap][128] E4M3 codes
  float* kscale;              // [B][Hkv][cap32]
};

struct SelectArgs {
  const float* key;   // [B][cap]
  const int32_t* lens;
  const int32_t* k;
  int B, cap, max_k;
  int chunk;          // filled by the launcher
  const uint32_t* hist0;   // optional [B][2048]: counts of the leading 11-bit key digit (tokens j < len - recent)
  int rows_per_seq;   // key rows per sequence: 1, or Hkv with per-KV-head selection (row r reads lens/k of r / rows_per_seq)
  int recent;         // BKP: the most recent min(recent, len) tokens are kept outright (0: none)
  uint16_t* hits;     // BKP: optional [B][cap] hit-rate table, +1 (saturating) per kept token
  int32_t* idx;
  int32_t* count;
  unsigned* err;
};

struct AttnArgs {
  const void* q;
  const void* k;
  const void* v;
  const int32_t* idx;
  const int32_t* count;
  int B, H, Hkv, cap, max_k;
  int64_t q_sb, q_sh, k_sb, k_sh, k_sn, v_sb, v_sh, v_sn;
  float* out;         // [B][H][d]
  float* part;        // [B*H][splits][2 + d] partials of split (b, g) pairs
  int splits;         // partial slots per (b, h)
  int kvh;            // 0: idx [B][max_k], count [B] shared by the KV heads; 1: idx [B][Hkv][max_k], count [B][Hkv]
  int Gs, hoff, Gn;   // as in ScoreArgs: heads g * Gs + hoff + [0, Gn) of KV head g
  unsigned* err;
};

// Raise a kernel's dynamic shared-memory limit to `bytes` on the current
// device if it is not there yet; `cache` (64 entries, one per device) records
// what was set, so that steady-state launches -- including ones under stream
// capture -- make no attribute calls.
inline cudaError_t ensure_smem_attr(const void* func, int bytes, int* cache) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (bytes > cache[dev]) {
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    cache[dev] = bytes;
  }
  return cudaSuccess;
}

// Launch `kern` as a programmatic dependent of the preceding kernel in the
// stream (its prologue may overlap that kernel's tail; the kernel itself
// calls pdl_wait() before touching data the predecessor produced), with an
// optional cluster shape.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       int cluster_x, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  int n = 1;
  if (cluster_x > 0) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    n = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, args...);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// score.cu
size_t score_smem_bytes(int G, bool f8);
int score_tile_tokens();
int score_warps();
int score_max_batch();
int score_max_kv_heads();
// Warps of the scoring kernel that share one KV head (the partial slots per
// CTA) when a call's launches cover nkv KV heads with groups of G query heads:
// kNW / nkv for nkv <= kNW / 2 and G >= 5, whose launches then all take the
// dealing kernel (deal = true, group template 8); else 1.
int score_deal_warps(int nkv, int G);
cudaError_t launch_score(const ScoreArgs& a, int dtype, int G, bool raw, bool f8, bool deal, int grid,
                         cudaStream_t st);
// Launches the normalisation (one or two kernels: *kernels is set to the
// count).  two_kernel: always combine the partials in their own kernel first,
// so that the finalize kernel takes its small form (at most 64 registers),
// which fits beside a scoring CTA on one SM.
cudaError_t launch_attn_finalize(const FinalizeArgs& a, int sms, cudaStream_t st, int* kernels,
                                 bool two_kernel = false);

// score_tc.cu
int score_tc_max_group();
int score_tc_max_heads();
cudaError_t launch_quantize_q(const QuantQArgs& a, int dtype, cudaStream_t st);
cudaError_t launch_score_tc(const ScoreTcArgs& a, bool raw, int grid, cudaStream_t st);

// selftest.cu
cudaError_t launch_selftest_wait(unsigned long long limit_ns, unsigned* err, cudaStream_t st);

// quant.cu
cudaError_t launch_quantize_k(const QuantArgs& a, int dtype, int max_rows, cudaStream_t st);

// select.cu
int select_cluster_size(int cap);
size_t select_smem_bytes(int cap, int C);
int select_hist_bins();
cudaError_t launch_select(const SelectArgs& a, cudaStream_t st);


// attn.cu
int attn_batch_tokens();
int attn_max_batch();
int attn_max_segments(int max_k);
// The attention kernel for one pass of G heads per KV head, and (combine)
// the merge of split partials over all heads.
cudaError_t launch_sparse_attn(const AttnArgs& a, int dtype, int G, int grid, bool combine, cudaStream_t st);

}  // namespace hill
