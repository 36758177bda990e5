// score.cu -- the K-cache streaming kernel (Eq. 1 over the whole cache) and
// the ATTN-mode normalisation (Sec. 4.1 column sum of softmax weights).
//
// hill_score_kernel: persistent CTAs of kNW warps.  A work item is a tile of
// kT consecutive tokens of one sequence; the KV heads g of an item are dealt
// to the warps (g mod kNW).  Every warp streams its own (item, g) sequence
// through a private ring of kSW shared-memory stages: lane 0 issues one bulk
// TMA copy of the tile's kT key rows (kT x 256 B, or kT row copies when the
// rows are strided) plus the G query rows of the head group, completing on
// the stage's mbarrier; the warp copies a landed stage into registers, hands
// the slot straight back to the copy engine for the stage kSW ahead, and
// computes.  Each lane owns 16 bytes of a row (a half-warp covers one 256-B
// row), keeps fp32 partial sums for 16 rows and finishes them with a
// 15-shuffle transposed reduction, after which lane l holds token
// 2*(l%16) + l/16 of the tile.
//
//   RAW : the per-token sum over heads is reduced across the warps in shared
//         memory at the end of each item (fixed order) and written to scores
//         (and added to accum).  The RAW importance is linear in q, so the G
//         query heads of a group are summed first (one dot product per row).
//   ATTN: every logit z = q.K/sqrt(d) is written to a [B][H][cap] buffer and
//         each lane keeps an online (max, sum exp) of its tokens per head;
//         when the CTA leaves a sequence the warp merges them and writes one
//         partial per (sequence, head, CTA).  hill_attn_finalize_kernel
//         combines the partials and forms s[b,j] = sum_h exp(z - m_bh) / L_bh.
#include "hill_internal.h"

namespace hill {

namespace {

constexpr int kT = 32;                      // tokens per tile (= rows per stage)
constexpr int kNW = 8;                      // warps per CTA
constexpr int kThreads = kNW * 32;
constexpr int kMaxBatchSmem = 512;          // sequences held in the per-CTA tables
constexpr int kTableInts = kMaxBatchSmem + 4;  // B + 1 entries, padded (16-byte alignment)
constexpr int kMaxRun = 8;                  // (KV heads per warp) x G online-softmax states per lane

template <int G>
struct ScoreCfg {
  static constexpr int kStageBytes = kT * kRowBytes + G * kRowBytes;
  static constexpr int kSW = G <= 4 ? 3 : 2;             // stages per warp
  static constexpr int kStages = kNW * kSW;
};

__device__ __forceinline__ int find_seq(const int* tstart, int B, int item) {
  int lo = 0, hi = B;  // tstart[lo] <= item < tstart[hi]
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (tstart[mid] <= item) lo = mid; else hi = mid;
  }
  return lo;
}

// Online (max, sum exp) of one lane's tokens.
__device__ __forceinline__ void online_push(float& m, float& l, float z) {
  if (z > m) {
    l = l * expf(m - z) + 1.f;
    m = z;
  } else {
    l += expf(z - m);
  }
}

__device__ __forceinline__ void online_merge_warp(float& m, float& l) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float l2 = __shfl_xor_sync(0xffffffffu, l, o);
    const float mx = fmaxf(m, m2);
    l = (mx == -INFINITY) ? 0.f : l * expf(m - mx) + l2 * expf(m2 - mx);
    m = mx;
  }
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Position of a warp in its own stage sequence: item (global tile index) and
// r (its r-th KV head of that item, g = warp + r * kNW).
struct Cursor {
  int item, r;
};

template <int DT, int G, bool RAW>
__global__ void __launch_bounds__(kThreads, 1) hill_score_kernel(ScoreArgs a) {
  using Cfg = ScoreCfg<G>;
  constexpr int kStageBytes = Cfg::kStageBytes;
  constexpr int kSW = Cfg::kSW;
  constexpr int kStages = Cfg::kStages;
  constexpr int kNH = RAW ? 1 : (G < 4 ? G : 4);   // heads per pass over a stage
  constexpr int kPasses = RAW ? 1 : G / kNH;
  constexpr int kMaxNg = RAW ? 1 : kMaxRun / G;    // KV heads per warp per item (ATTN)

  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* stage_base = smem;
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  int* tstart = reinterpret_cast<int*>(full_bar + kStages);             // [B+1] tile prefix
  int* slen = tstart + kTableInts;                                      // [B] clamped lengths
  float* red = reinterpret_cast<float*>(slen + kTableInts);             // [2][kNW][kT]
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int B = a.B, H = a.H, Hkv = a.Hkv, cap = a.cap;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_addr(&full_bar[s]), 1);
    fence_barrier_init();
    abort_flag = 0;
  }
  for (int b = threadIdx.x; b < B; b += kThreads) {
    int len = a.lens[b];
    if (len < 0 || len > cap) {
      raise_error(a.err, kErrDevArg);
      len = len < 0 ? 0 : cap;
    }
    slen[b] = len;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    tstart[0] = 0;
    for (int b = 0; b < B; ++b) {
      acc += (slen[b] + kT - 1) / kT;
      tstart[b + 1] = acc;
    }
  }
  __syncthreads();
  const int n_items = tstart[B];
  const int ng = (Hkv - warp + kNW - 1) / kNW;   // KV heads of this warp per item

  const uint64_t pol = l2_evict_first_policy();
  const auto* kbase = static_cast<const uint16_t*>(a.k);
  const auto* qbase = static_cast<const uint16_t*>(a.q);
  const uint32_t stage0 = smem_addr(stage_base) + warp * kSW * kStageBytes;
  const uint32_t bar0 = smem_addr(&full_bar[warp * kSW]);

  auto advance = [&](Cursor& c) {
    if (++c.r >= ng) {
      c.r = 0;
      c.item += gridDim.x;
    }
  };
  // lane 0: load stage `no` of this warp's sequence (position c) into its slot
  auto issue = [&](const Cursor& c, uint32_t no) {
    const int b = find_seq(tstart, B, c.item);
    const int j0 = (c.item - tstart[b]) * kT;
    const int nv = min(kT, slen[b] - j0);
    const int g = warp + c.r * kNW;
    const uint32_t s = no % kSW;
    const uint32_t fb = bar0 + s * 8;
    const uint32_t dst = stage0 + s * kStageBytes;
    mbar_arrive_expect_tx(fb, (uint32_t)(nv + G) * kRowBytes);
    const uint16_t* ksrc = kbase + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh + (int64_t)j0 * a.k_sn;
    if (a.k_sn == kHeadDim) {
      bulk_g2s(dst, ksrc, (uint32_t)nv * kRowBytes, fb, pol);
    } else {
      for (int r = 0; r < nv; ++r) bulk_g2s(dst + r * kRowBytes, ksrc + (int64_t)r * a.k_sn, kRowBytes, fb, pol);
    }
    const uint16_t* qsrc = qbase + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh;
    const uint32_t qdst = dst + kT * kRowBytes;
    if (a.q_sh == kHeadDim) {
      bulk_g2s(qdst, qsrc, G * kRowBytes, fb);
    } else {
#pragma unroll
      for (int r = 0; r < G; ++r) bulk_g2s(qdst + r * kRowBytes, qsrc + (int64_t)r * a.q_sh, kRowBytes, fb);
    }
  };

  // prologue: the first kSW stages of this warp
  Cursor pc{(int)blockIdx.x, 0};
  uint32_t issued = 0;
  if (ng > 0) {
    for (; issued < (uint32_t)kSW && pc.item < n_items; ++issued) {
      if (lane == 0) issue(pc, issued);
      advance(pc);
    }
  }

  const int l16 = lane & 15;
  const int half = lane >> 4;
  const int tok = 2 * l16 + half;          // token (within the tile) this lane ends with
  uint32_t used = 0;                       // stages consumed
  int item_no = 0;
  bool ok = true;

  float run_m[RAW ? 1 : kMaxRun], run_l[RAW ? 1 : kMaxRun];
  int cur_b = -1, cur_slot = 0;
  auto reset_run = [&]() {
#pragma unroll
    for (int e = 0; e < (RAW ? 1 : kMaxRun); ++e) {
      run_m[e] = -INFINITY;
      run_l[e] = 0.f;
    }
  };
  auto flush = [&]() {
    if (RAW) return;
#pragma unroll
    for (int r = 0; r < kMaxNg; ++r) {
      if (r >= ng) break;
#pragma unroll
      for (int hl = 0; hl < G; ++hl) {
        float m = run_m[r * G + hl], l = run_l[r * G + hl];
        online_merge_warp(m, l);
        const int h = (warp + r * kNW) * G + hl;
        if (lane == 0) a.partials[((int64_t)cur_b * a.nslot + cur_slot) * H + h] = make_float2(m, l);
      }
    }
  };
  reset_run();

  for (int item = blockIdx.x; item < n_items; item += gridDim.x, ++item_no) {
    const int b = find_seq(tstart, B, item);
    const int tile = item - tstart[b];
    const int j0 = tile * kT;
    const int nv = min(kT, slen[b] - j0);
    const bool valid = tok < nv;
    float rsum = 0.f;

    if (!RAW && b != cur_b) {
      if (cur_b >= 0) flush();
      reset_run();
      cur_b = b;
      cur_slot = tile;   // = item - tstart[b]: this CTA's first item in b
    }

#pragma unroll 1
    for (int r = 0; r < ng && ok; ++r) {
      const int g = warp + r * kNW;
      const uint32_t s = used % kSW;
      if (!mbar_wait(bar0 + s * 8, (used / kSW) & 1u, a.err)) {
        ok = false;
        abort_flag = 1;
        break;
      }
      const uint32_t sb = stage0 + s * kStageBytes;
      const uint32_t qb = sb + kT * kRowBytes;
      // copy the stage into registers, then refill the slot with the stage
      // kSW ahead while this one is computed
      uint4 kv[16];
#pragma unroll
      for (int it = 0; it < 16; ++it) kv[it] = lds128(sb + (2 * it + half) * kRowBytes + l16 * 16);
      uint4 qv[G];
#pragma unroll
      for (int hh = 0; hh < G; ++hh) qv[hh] = lds128(qb + hh * kRowBytes + l16 * 16);
      ++used;
      __syncwarp();
      if (pc.item < n_items) {
        if (lane == 0) {
          fence_proxy_async_smem();
          issue(pc, issued);
        }
        ++issued;
        advance(pc);
      }

#pragma unroll
      for (int pass = 0; pass < kPasses; ++pass) {
        float qf[kNH][8];
        if (RAW) {
#pragma unroll
          for (int e = 0; e < 8; ++e) qf[0][e] = 0.f;
#pragma unroll
          for (int hh = 0; hh < G; ++hh) {
            float t[8];
            to_float8<DT>(qv[hh], t);
#pragma unroll
            for (int e = 0; e < 8; ++e) qf[0][e] += t[e];
          }
        } else {
#pragma unroll
          for (int hh = 0; hh < kNH; ++hh) to_float8<DT>(qv[pass * kNH + hh], qf[hh]);
        }
        float acc[kNH][16];
#pragma unroll
        for (int it = 0; it < 16; ++it) {
          float kf[8];
          to_float8<DT>(kv[it], kf);
#pragma unroll
          for (int hh = 0; hh < kNH; ++hh) {
            float sum = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) sum = fmaf(qf[hh][e], kf[e], sum);
            acc[hh][it] = sum;
          }
        }
#pragma unroll
        for (int hh = 0; hh < kNH; ++hh) {
          const float z = half_transpose_reduce(acc[hh], lane) * kInvSqrtD;
          if (RAW) {
            rsum += z;
          } else {
            const int hl = pass * kNH + hh;            // head within the group
            const int h = g * G + hl;
            if (valid) {
              a.logits[((int64_t)b * H + h) * cap + j0 + tok] = z;
              // r is warp-uniform; select the register slot with a static index
#pragma unroll
              for (int rr = 0; rr < kMaxNg; ++rr)
                if (rr == r) online_push(run_m[rr * G + hl], run_l[rr * G + hl], z);
            }
          }
        }
      }
    }
    if (RAW) {
      // sum over the warps in a fixed order, double-buffered by item; a warp
      // whose wait timed out still reaches the barrier, and all warps then
      // leave together
      float* rb = red + (item_no & 1) * kNW * kT;
      rb[warp * kT + tok] = rsum;
      named_sync(1, kThreads);
      if (abort_flag) break;
      if (warp == (item_no % kNW) && valid) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < kNW; ++w) sum += rb[w * kT + tok];
        const int64_t o = (int64_t)b * cap + j0 + tok;
        if (a.scores) a.scores[o] = sum;
        if (a.accum) a.accum[o] += sum;
      }
    } else if (!ok) {
      break;
    }
  }
  if (!RAW && cur_b >= 0 && ok) flush();
  // after a timeout: give every copy this warp issued and did not consume one
  // more bounded wait before the CTA's shared memory is released
  if (!ok && lane == 0) {
    for (uint32_t u = used; u < issued; ++u) mbar_wait(bar0 + (u % kSW) * 8, (u / kSW) & 1u, a.err);
  }
}

// Combine the per-CTA (max, sum exp) partials of every head of sequence b,
// then s[b,j] = sum_h exp(z[b,h,j] - m_h) / L_h, one token per thread.  Both
// phases issue all their loads before using them: the partials of a head are
// spread over 8 threads, and each thread loads the logits of 16 heads of its
// token at once (they were just written and are mostly L2 resident).
constexpr int kFinThreads = 256;
constexpr int kFinChunk = kFinThreads;
constexpr int kFinPartThreads = 8;                 // threads combining one head
constexpr int kFinPartMax = 32;                    // partials per thread held in registers

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
  const float2* pb = a.partials + (int64_t)b * a.nslot * a.H;
  const int sub = threadIdx.x % kFinPartThreads;
  for (int h = threadIdx.x / kFinPartThreads; h < a.H; h += kFinThreads / kFinPartThreads) {
    float2 p[kFinPartMax];
#pragma unroll
    for (int u = 0; u < kFinPartMax; ++u) {
      const int s = sub + u * kFinPartThreads;
      p[u] = s < ns ? pb[(int64_t)s * a.H + h] : make_float2(-INFINITY, 0.f);
    }
    float m = -INFINITY;
#pragma unroll
    for (int u = 0; u < kFinPartMax; ++u) m = fmaxf(m, p[u].x);
    // slots beyond kFinPartMax * kFinPartThreads (grids of more than 256
    // CTAs) are folded in sequentially
    for (int s = sub + kFinPartMax * kFinPartThreads; s < ns; s += kFinPartThreads)
      m = fmaxf(m, pb[(int64_t)s * a.H + h].x);
#pragma unroll
    for (int o = kFinPartThreads / 2; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float l = 0.f;
#pragma unroll
    for (int u = 0; u < kFinPartMax; ++u) l += p[u].y > 0.f ? p[u].y * expf(p[u].x - m) : 0.f;
    for (int s = sub + kFinPartMax * kFinPartThreads; s < ns; s += kFinPartThreads) {
      const float2 q = pb[(int64_t)s * a.H + h];
      l += q.y * expf(q.x - m);
    }
#pragma unroll
    for (int o = kFinPartThreads / 2; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    if (sub == 0) {
      mh[h] = m;
      il[h] = 1.f / l;
    }
  }
  __syncthreads();
  const int j = jb + threadIdx.x;
  if (j >= len) return;
  const float* zp = a.logits + (int64_t)b * a.H * a.cap + j;
  float s = 0.f;
  int h = 0;
  for (; h + 16 <= a.H; h += 16) {
    float z[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) z[u] = zp[(int64_t)(h + u) * a.cap];
#pragma unroll
    for (int u = 0; u < 16; ++u) s += expf(z[u] - mh[h + u]) * il[h + u];
  }
  for (; h < a.H; ++h) s += expf(zp[(int64_t)h * a.cap] - mh[h]) * il[h];
  const int64_t o = (int64_t)b * a.cap + j;
  if (a.scores) a.scores[o] = s;
  if (a.accum) a.accum[o] += s;
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

template <int G>
size_t smem_for() {
  using Cfg = ScoreCfg<G>;
  return (size_t)Cfg::kStages * Cfg::kStageBytes + Cfg::kStages * sizeof(uint64_t) +
         2 * kTableInts * sizeof(int) + 2 * kNW * kT * sizeof(float);
}

}  // namespace

size_t score_smem_bytes(int G) {
  switch (G) {
    case 1: return smem_for<1>();
    case 2: return smem_for<2>();
    case 4: return smem_for<4>();
    default: return smem_for<8>();
  }
}

int score_tile_tokens() { return kT; }
int score_max_batch() { return kMaxBatchSmem; }
int score_max_kv_heads(int G) { return (kMaxRun / G) * kNW; }

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
