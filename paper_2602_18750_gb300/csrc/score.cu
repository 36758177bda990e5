// score.cu -- the K-cache streaming kernel (Eq. 1 over the whole cache) and
// the ATTN-mode normalisation (Sec. 4.1 column sum of softmax weights).
//
// hill_score_kernel: persistent CTAs, one producer warp and kNC consumer
// warps.  A work item is a tile of kT consecutive tokens of one sequence; for
// each KV head g of the item the producer issues one bulk TMA copy of the
// tile's kT key rows (kT x 256 B, or kT row copies if the rows are strided)
// plus the G query rows of that head group into a shared-memory stage, and
// consumer warp (g mod kNC) computes the G dot products of every row.  Each
// lane owns 16 bytes of a row (a half-warp covers one 256-byte row), keeps
// fp32 partial sums for 16 rows and finishes them with a 15-shuffle
// transposed reduction, after which lane l holds token 2*(l%16) + l/16.
//
//   RAW : the per-token sum over heads is reduced across the consumer warps
//         in shared memory at the end of each item (fixed order) and written
//         to scores (and added to accum).  Since the RAW importance is linear
//         in q, the G query heads of a group are summed first (one dot/row).
//   ATTN: every logit z = q.K/sqrt(d) is written to a [B][H][cap] buffer and
//         each warp keeps, per (sequence, head), a running (max, sum exp) over
//         the tiles it processed; these per-CTA partials are combined in
//         hill_attn_finalize_kernel, which then forms
//         s[b,j] = sum_h exp(z[b,h,j] - m_bh) / L_bh.
#include "hill_internal.h"

namespace hill {

namespace {

constexpr int kT = 32;                      // tokens per tile (= rows per stage)
constexpr int kNC = 8;                      // consumer warps
constexpr int kSW = 2;                      // stages per consumer warp
constexpr int kStages = kNC * kSW;
constexpr int kThreads = (kNC + 1) * 32;
constexpr int kMaxBatchSmem = 2048;         // sequences held in the tile prefix table
constexpr int kTstartInts = kMaxBatchSmem + 4;  // B + 1 entries, padded to keep 16-byte alignment
constexpr int kRunSlots = 64;               // running (m, l) slots per warp (Hkv/kNC * G)

template <int G>
struct ScoreSmem {
  static constexpr int kStageBytes = kT * kRowBytes + G * kRowBytes;
};

__device__ __forceinline__ int find_seq(const int* tstart, int B, int item) {
  int lo = 0, hi = B;  // tstart[lo] <= item < tstart[hi]
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (tstart[mid] <= item) lo = mid; else hi = mid;
  }
  return lo;
}

template <int DT, int G, bool RAW>
__global__ void __launch_bounds__(kThreads, 1) hill_score_kernel(ScoreArgs a) {
  extern __shared__ __align__(1024) unsigned char smem[];
  constexpr int kStageBytes = ScoreSmem<G>::kStageBytes;
  constexpr int kNH = RAW ? 1 : (G < 4 ? G : 4);   // heads per pass over a stage
  constexpr int kPasses = RAW ? 1 : G / kNH;

  unsigned char* stage_base = smem;
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* empty_bar = full_bar + kStages;
  int* tstart = reinterpret_cast<int*>(empty_bar + kStages);            // [B+1]
  float* red = reinterpret_cast<float*>(tstart + kTstartInts);          // [2][kNC][kT]
  float2* run = reinterpret_cast<float2*>(red + 2 * kNC * kT);          // [kNC][kRunSlots]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int B = a.B, H = a.H, Hkv = a.Hkv, cap = a.cap;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_addr(&full_bar[s]), 1);
      mbar_init(smem_addr(&empty_bar[s]), 1);
    }
    fence_barrier_init();
    int acc = 0;
    tstart[0] = 0;
    for (int b = 0; b < B; ++b) {
      int len = a.lens[b];
      if (len < 0 || len > cap) {
        raise_error(a.err, kErrDevArg);
        len = len < 0 ? 0 : cap;
      }
      acc += (len + kT - 1) / kT;
      tstart[b + 1] = acc;
    }
  }
  __syncthreads();
  const int n_items = tstart[B];

  if (warp == kNC) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = l2_evict_first_policy();
      const auto* kbase = static_cast<const uint16_t*>(a.k);
      const auto* qbase = static_cast<const uint16_t*>(a.q);
      uint32_t cnt[kNC];
#pragma unroll
      for (int w = 0; w < kNC; ++w) cnt[w] = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        const int b = find_seq(tstart, B, item);
        const int j0 = (item - tstart[b]) * kT;
        int len = a.lens[b];
        len = len < 0 ? 0 : (len > cap ? cap : len);
        const int nv = min(kT, len - j0);
        for (int g = 0; g < Hkv; ++g) {
          const int w = g % kNC;
          const int slot = w * kSW + (cnt[w] % kSW);
          const uint32_t par = (cnt[w] / kSW) & 1u;
          if (!mbar_wait(smem_addr(&empty_bar[slot]), par ^ 1u, a.err)) { ok = false; break; }
          const uint32_t fb = smem_addr(&full_bar[slot]);
          const uint32_t dst = smem_addr(stage_base + slot * kStageBytes);
          mbar_arrive_expect_tx(fb, (uint32_t)(nv + G) * kRowBytes);
          const uint16_t* ksrc = kbase + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh + (int64_t)j0 * a.k_sn;
          if (a.k_sn == kHeadDim) {
            bulk_g2s(dst, ksrc, (uint32_t)nv * kRowBytes, fb, pol);
          } else {
            for (int r = 0; r < nv; ++r)
              bulk_g2s(dst + r * kRowBytes, ksrc + (int64_t)r * a.k_sn, kRowBytes, fb, pol);
          }
          const uint16_t* qsrc = qbase + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh;
          const uint32_t qdst = dst + kT * kRowBytes;
          if (a.q_sh == kHeadDim) {
            bulk_g2s(qdst, qsrc, G * kRowBytes, fb);
          } else {
#pragma unroll
            for (int r = 0; r < G; ++r) bulk_g2s(qdst + r * kRowBytes, qsrc + (int64_t)r * a.q_sh, kRowBytes, fb);
          }
          cnt[w]++;
        }
      }
      // Before leaving, make sure no copy issued by this CTA is still in
      // flight (they all are consumed in a normal run; this matters only
      // after a timeout).
      for (int w = 0; w < kNC; ++w) {
        for (int s = 0; s < kSW; ++s) {
          uint32_t c = cnt[w];
          if (c == 0) continue;
          // the last copy into slot (w, s) was number (c - 1 - ((c - 1 - s) % kSW))
          if (c <= (uint32_t)s) continue;
          uint32_t last = (c - 1) - ((c - 1 + kSW - s) % kSW);
          mbar_wait(smem_addr(&full_bar[w * kSW + s]), (last / kSW) & 1u, a.err);
        }
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int l16 = lane & 15;
  const int half = lane >> 4;
  const int tok = 2 * l16 + half;          // token (within the tile) this lane ends with
  const float scale = kInvSqrtD;
  const int ng = (Hkv - warp + kNC - 1) / kNC;   // KV heads of this warp per item
  float2* myrun = run + warp * kRunSlots;
  int cur_b = -1, cur_slot = 0;
  uint32_t cnt = 0;
  int item_no = 0;
  bool ok = true;

  auto flush = [&](int b, int slot) {
    // running (max, sum exp) of this warp's heads for sequence b -> global partials
    for (int e = lane; e < ng * G; e += 32) {
      const int r = e / G, hh = e % G;
      const int h = (warp + r * kNC) * G + hh;
      a.partials[((int64_t)b * a.nslot + slot) * H + h] = myrun[e];
    }
  };

  __shared__ int abort_flag;
  if (threadIdx.x == 0) abort_flag = 0;
  named_sync(1, kNC * 32);

  for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x, ++item_no) {
    const int b = find_seq(tstart, B, item);
    const int tile = item - tstart[b];
    const int j0 = tile * kT;
    int len = a.lens[b];
    len = len < 0 ? 0 : (len > cap ? cap : len);
    const int nv = min(kT, len - j0);
    const bool valid = tok < nv;
    float rsum = 0.f;

    if (!RAW && b != cur_b) {
      if (cur_b >= 0) flush(cur_b, cur_slot);
      __syncwarp();
      for (int e = lane; e < ng * G; e += 32) myrun[e] = make_float2(-INFINITY, 0.f);
      __syncwarp();
      cur_b = b;
      cur_slot = tile;   // = item - tstart[b]: this CTA's first item in b
    }

    for (int r = 0; r < ng; ++r) {
      const int g = warp + r * kNC;
      const int slot = warp * kSW + (cnt % kSW);
      const uint32_t par = (cnt / kSW) & 1u;
      ++cnt;
      if (!mbar_wait(smem_addr(&full_bar[slot]), par, a.err)) {
        ok = false;
        abort_flag = 1;
        break;
      }
      const uint32_t sb = smem_addr(stage_base + slot * kStageBytes);
      const uint32_t qb = sb + kT * kRowBytes;

#pragma unroll
      for (int pass = 0; pass < kPasses; ++pass) {
        float qf[kNH][8];
        if (RAW) {
#pragma unroll
          for (int e = 0; e < 8; ++e) qf[0][e] = 0.f;
#pragma unroll
          for (int hh = 0; hh < G; ++hh) {
            float t[8];
            to_float8<DT>(lds128(qb + hh * kRowBytes + l16 * 16), t);
#pragma unroll
            for (int e = 0; e < 8; ++e) qf[0][e] += t[e];
          }
        } else {
#pragma unroll
          for (int hh = 0; hh < kNH; ++hh)
            to_float8<DT>(lds128(qb + (pass * kNH + hh) * kRowBytes + l16 * 16), qf[hh]);
        }
        float acc[kNH][16];
#pragma unroll
        for (int it = 0; it < 16; ++it) {
          const uint4 v = lds128(sb + (2 * it + half) * kRowBytes + l16 * 16);
          float kf[8];
          to_float8<DT>(v, kf);
#pragma unroll
          for (int hh = 0; hh < kNH; ++hh) {
            float s = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) s = fmaf(qf[hh][e], kf[e], s);
            acc[hh][it] = s;
          }
        }
        if (pass == kPasses - 1) {
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_addr(&empty_bar[slot]));
        }
#pragma unroll
        for (int hh = 0; hh < kNH; ++hh) {
          const float z = half_transpose_reduce(acc[hh], lane) * scale;
          if (RAW) {
            rsum += z;
          } else {
            const int hl = pass * kNH + hh;            // head within the group
            const int h = g * G + hl;
            if (valid) a.logits[((int64_t)b * H + h) * cap + j0 + tok] = z;
            const float mt = warp_max(valid ? z : -INFINITY);
            const float lt = warp_sum(valid ? expf(z - mt) : 0.f);
            const int e = r * G + hl;
            float2 cur = myrun[e];
            const float mn = fmaxf(cur.x, mt);
            const float ln = cur.y * expf(cur.x - mn) + lt * expf(mt - mn);
            __syncwarp();
            if (lane == 0) myrun[e] = make_float2(mn, ln);
            __syncwarp();
          }
        }
      }
    }
    if (RAW) {
      // sum over the consumer warps in a fixed order, double-buffered by item;
      // a warp whose wait timed out still reaches the barrier, and all warps
      // then leave together
      float* rb = red + (item_no & 1) * kNC * kT;
      rb[warp * kT + tok] = rsum;
      named_sync(1, kNC * 32);
      if (abort_flag) break;
      if (warp == (item_no % kNC) && valid) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < kNC; ++w) s += rb[w * kT + tok];
        const int64_t o = (int64_t)b * cap + j0 + tok;
        if (a.scores) a.scores[o] = s;
        if (a.accum) a.accum[o] += s;
      }
    }
  }
  if (!RAW && cur_b >= 0) flush(cur_b, cur_slot);
}

// Combine the per-CTA (max, sum exp) partials of every head of sequence b,
// then s[b,j] = sum_h exp(z[b,h,j] - m_h) / L_h for this CTA's token chunk.
constexpr int kFinChunk = 512;
constexpr int kFinThreads = 256;

__global__ void __launch_bounds__(kFinThreads) hill_attn_finalize_kernel(FinalizeArgs a) {
  extern __shared__ float fsm[];
  float* mh = fsm;            // [H]
  float* il = fsm + a.H;      // [H]
  const int b = blockIdx.y;
  int len = a.lens[b];
  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  const int jb = blockIdx.x * kFinChunk;
  if (jb >= len) return;
  const int tiles = (len + kT - 1) / kT;
  const int ns = min(tiles, a.nslot);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int h = warp; h < a.H; h += kFinThreads / 32) {
    float m = -INFINITY;
    for (int s = lane; s < ns; s += 32) m = fmaxf(m, a.partials[((int64_t)b * a.nslot + s) * a.H + h].x);
    m = warp_max(m);
    float l = 0.f;
    for (int s = lane; s < ns; s += 32) {
      const float2 p = a.partials[((int64_t)b * a.nslot + s) * a.H + h];
      l += p.y * expf(p.x - m);
    }
    l = warp_sum(l);
    if (lane == 0) {
      mh[h] = m;
      il[h] = 1.f / l;
    }
  }
  __syncthreads();
  const int je = min(jb + kFinChunk, len);
  for (int j = jb + threadIdx.x; j < je; j += kFinThreads) {
    float s = 0.f;
    const float* zp = a.logits + (int64_t)b * a.H * a.cap + j;
    for (int h = 0; h < a.H; ++h) s += expf(zp[(int64_t)h * a.cap] - mh[h]) * il[h];
    const int64_t o = (int64_t)b * a.cap + j;
    if (a.scores) a.scores[o] = s;
    if (a.accum) a.accum[o] += s;
  }
}

template <int DT, int G, bool RAW>
cudaError_t launch_score_t(const ScoreArgs& a, int grid, cudaStream_t st) {
  const size_t smem = score_smem_bytes(G);
  auto kern = hill_score_kernel<DT, G, RAW>;
  static int cache[64] = {0};
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), (int)smem, cache);
  if (e != cudaSuccess) return e;
  kern<<<grid, kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

template <int DT, bool RAW>
cudaError_t launch_score_g(const ScoreArgs& a, int G, int grid, cudaStream_t st) {
  switch (G) {
    case 1: return launch_score_t<DT, 1, RAW>(a, grid, st);
    case 2: return launch_score_t<DT, 2, RAW>(a, grid, st);
    case 4: return launch_score_t<DT, 4, RAW>(a, grid, st);
    case 8: return launch_score_t<DT, 8, RAW>(a, grid, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

size_t score_smem_bytes(int G) {
  const size_t stage = (size_t)kT * kRowBytes + (size_t)G * kRowBytes;
  return kStages * stage + 2 * kStages * sizeof(uint64_t) + kTstartInts * sizeof(int) +
         2 * kNC * kT * sizeof(float) + kNC * kRunSlots * sizeof(float2);
}

int score_tile_tokens() { return kT; }
int score_max_batch() { return kMaxBatchSmem; }
int score_max_kv_heads(int G) { return (kRunSlots / G) * kNC; }

cudaError_t launch_score(const ScoreArgs& a, int dtype, int G, bool raw, int grid, cudaStream_t st) {
  if (dtype == 0) return raw ? launch_score_g<0, true>(a, G, grid, st) : launch_score_g<0, false>(a, G, grid, st);
  return raw ? launch_score_g<1, true>(a, G, grid, st) : launch_score_g<1, false>(a, G, grid, st);
}

cudaError_t launch_attn_finalize(const FinalizeArgs& a, cudaStream_t st) {
  dim3 grid((a.cap + kFinChunk - 1) / kFinChunk, a.B);
  hill_attn_finalize_kernel<<<grid, kFinThreads, 2 * a.H * sizeof(float), st>>>(a);
  return cudaGetLastError();
}

}  // namespace hill
