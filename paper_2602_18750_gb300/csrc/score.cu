// score.cu -- the K-cache streaming kernel (Eq. 1 over the whole cache) and
// the ATTN-mode normalisation (Sec. 4.1 column sum of softmax weights).
//
// hill_score_kernel: persistent CTAs of kNW warps.  A work item is a tile of
// kT = 32 consecutive tokens of one sequence; the KV heads g of an item are
// dealt to the warps (g mod kNW).  Every warp streams its own (item, g)
// sequence through a private ring of kSW shared-memory stages: lane 0 issues
// two tiled TMA loads (dims 0-63 and 64-127 of the tile's 32 key rows, 128-
// byte swizzle) plus a bulk copy of the G query rows of the head group, all
// completing on the stage's mbarrier.  The warp moves a landed tile into
// registers with ldmatrix (conflict-free thanks to the swizzle), hands the
// slot back to the copy engine for the stage kSW ahead, and computes the
// [32 tokens x 128] . [128 x G heads] product with 16 mma.sync m16n8k16
// (fp32 accumulation; the G query heads fill the N = 8 columns, so one
// instruction stream serves MHA and GQA alike).
//
//   RAW : the per-token sum over heads is reduced across the warps in shared
//         memory at the end of each item (fixed order) and written to scores
//         (and added to accum).
//   ATTN: every logit z = q.K/sqrt(d) is written to a [B][H][cap] buffer; per
//         stage the warp reduces each head's tile (max, sum exp) and merges it
//         into a running state in shared memory; when the CTA leaves a
//         sequence the warp writes one partial per (sequence, head, CTA).
//         hill_attn_finalize_kernel combines the partials and forms
//         s[b,j] = sum_h exp(z[b,h,j] - m_bh) / L_bh.
#include "hill_internal.h"

namespace hill {

namespace {

constexpr int kT = 32;                      // tokens per tile (= rows per stage)
constexpr int kNW = 8;                      // warps per CTA
constexpr int kThreads = kNW * 32;
constexpr int kMaxBatchSmem = 512;          // sequences held in the per-CTA tables
constexpr int kTableInts = kMaxBatchSmem + 4;  // B + 1 entries, padded (16-byte alignment)
constexpr int kMaxNg = 4;                   // KV heads per warp per item (Hkv <= kNW * kMaxNg)
constexpr int kBoxBytes = kT * 128;         // one 64-dim half of a tile: 32 swizzled 128-byte rows
constexpr int kKBytes = 2 * kBoxBytes;

template <int G>
struct ScoreCfg {
  static constexpr int kSlotBytes = ((kKBytes + G * kRowBytes + 1023) / 1024) * 1024;
  static constexpr int kSW = G <= 4 ? 3 : 2;             // stages per warp
  static constexpr int kStages = kNW * kSW;
  // shared-memory layout (offsets from a 1024-byte aligned base)
  static constexpr int kOffBar = kStages * kSlotBytes;
  static constexpr int kOffTab = kOffBar + kStages * 8;
  static constexpr int kOffRed = kOffTab + 2 * kTableInts * 4;
  static constexpr int kOffStat = kOffRed + 2 * kNW * kT * 4;
  static constexpr int kOffFlag = kOffStat + kNW * kMaxNg * 8 * 8;
  static constexpr int kBytes = kOffFlag + 16 + 1024;        // + alignment slack
};

__device__ __forceinline__ int find_seq(const int* tstart, int B, int item) {
  int lo = 0, hi = B;  // tstart[lo] <= item < tstart[hi]
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (tstart[mid] <= item) lo = mid; else hi = mid;
  }
  return lo;
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Merge two (max, sum exp) pairs.
__device__ __forceinline__ float2 merge_ml(float2 x, float2 y) {
  const float m = fmaxf(x.x, y.x);
  if (m == -INFINITY) return make_float2(-INFINITY, 0.f);
  return make_float2(m, x.y * expf(x.x - m) + y.y * expf(y.x - m));
}

// Position of a warp in its own stage sequence: item (global tile index) and
// r (its r-th KV head of that item, g = warp + r * kNW).
struct Cursor {
  int item, r;
};

template <int DT, int G, bool RAW>
__global__ void __launch_bounds__(kThreads, 1) hill_score_kernel(const __grid_constant__ ScoreArgs a) {
  using Cfg = ScoreCfg<G>;
  constexpr int kSlotBytes = Cfg::kSlotBytes;
  constexpr int kSW = Cfg::kSW;
  constexpr int kStages = Cfg::kStages;

  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw_addr = smem_addr(smem_raw);
  const uint32_t base_addr = (raw_addr + 1023u) & ~1023u;
  unsigned char* base = smem_raw + (base_addr - raw_addr);
  int* tstart = reinterpret_cast<int*>(base + Cfg::kOffTab);          // [B+1] tile prefix
  int* slen = tstart + kTableInts;                                     // [B] clamped lengths
  float* red = reinterpret_cast<float*>(base + Cfg::kOffRed);          // [2][kNW][kT]
  float2* stat = reinterpret_cast<float2*>(base + Cfg::kOffStat);      // [kNW][kMaxNg][8]
  volatile int* abort_flag = reinterpret_cast<int*>(base + Cfg::kOffFlag);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int B = a.B, H = a.H, Hkv = a.Hkv, cap = a.cap;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(base_addr + Cfg::kOffBar + s * 8, 1);
    fence_barrier_init();
    *abort_flag = 0;
    prefetch_tmap(&a.kmap);
  }
  pdl_wait();
  pdl_launch_dependents();
  for (int b = threadIdx.x; b < B; b += kThreads) {
    int len = a.lens[b];
    if (len < 0 || len > cap) {
      raise_error(a.err, kErrDevArg);
      len = len < 0 ? 0 : cap;
    }
    slen[b] = len;
  }
  __syncthreads();
  // an item holds every KV head of one tile
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
  const int ng = (Hkv - warp + kNW - 1) / kNW;   // KV heads of this warp per tile

  const uint64_t pol = l2_evict_first_policy();
  const auto* qbase = static_cast<const uint16_t*>(a.q);
  const uint32_t stage0 = base_addr + warp * kSW * kSlotBytes;
  const uint32_t bar0 = base_addr + Cfg::kOffBar + warp * kSW * 8;

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
    const int g = warp + c.r * kNW;
    const uint32_t s = no % kSW;
    const uint32_t fb = bar0 + s * 8;
    const uint32_t dst = stage0 + s * kSlotBytes;
    mbar_arrive_expect_tx(fb, (uint32_t)(kKBytes + G * kRowBytes));
    int crd[4] = {0, 0, 0, 0};
    crd[a.kdim_tok] = j0;
    crd[a.kdim_head] = g;
    crd[a.kdim_seq] = b;
    tma_load_4d(dst, &a.kmap, 0, crd[1], crd[2], crd[3], fb, pol);
    tma_load_4d(dst + kBoxBytes, &a.kmap, 64, crd[1], crd[2], crd[3], fb, pol);
    const uint16_t* qsrc = qbase + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh;
    const uint32_t qdst = dst + kKBytes;
    if (a.q_sh == kHeadDim) {
      bulk_g2s(qdst, qsrc, G * kRowBytes, fb);
    } else {
#pragma unroll
      for (int r = 0; r < G; ++r) bulk_g2s(qdst + r * kRowBytes, qsrc + (int64_t)r * a.q_sh, kRowBytes, fb);
    }
  };

  // per-warp running (max, sum exp) of each (stage slot r, head) of the current sequence
  float2* wstat = stat + warp * kMaxNg * 8;
  auto reset_stat = [&]() {
    __syncwarp();
    wstat[lane] = make_float2(-INFINITY, 0.f);   // kMaxNg * 8 == 32 entries
    __syncwarp();
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

  // fragment coordinates (mma.sync m16n8k16): C row = token lane/4 (+8),
  // C columns = heads 2*(lane%4) and 2*(lane%4)+1 of the group
  const int grp = lane >> 2, tig = lane & 3;
  const int hA = 2 * tig, hB = 2 * tig + 1;
  // ldmatrix row address pieces: matrix m = lane/8 covers rows (m&1)*8.., k half m>>1
  const int lm_row = (lane & 7) + ((lane >> 3) & 1) * 8;
  const int lm_khalf = lane >> 4;
  uint32_t used = 0;                       // stages consumed
  int item_no = 0;
  bool ok = true;
  int cur_b = -1, cur_slot = 0;
  if (!RAW) reset_stat();

  auto flush = [&]() {
    if constexpr (!RAW) {
      __syncwarp();
      if (lane < ng * G) {
        const int r = lane / G, hl = lane % G;
        const int h = (warp + r * kNW) * G + hl;
        a.partials[((int64_t)cur_b * a.nslot + cur_slot) * H + h] = wstat[r * 8 + hl];
      }
      __syncwarp();
    }
  };

  for (int item = blockIdx.x; item < n_items; item += gridDim.x, ++item_no) {
    const int b = find_seq(tstart, B, item);
    const int tile = item - tstart[b];
    const int j0 = tile * kT;
    const int nv = min(kT, slen[b] - j0);
    float rs[4] = {0.f, 0.f, 0.f, 0.f};   // RAW: token sums of rows grp, grp+8, 16+grp, 24+grp

    if (!RAW && b != cur_b) {
      if (cur_b >= 0) flush();
      reset_stat();
      cur_b = b;
      cur_slot = tile;   // = item - tstart[b]: this CTA's first item in b (< gridDim.x)
    }

#pragma unroll 1
    for (int r = 0; r < ng && ok; ++r) {
      const int g = warp + r * kNW;
      const int sr = r;   // running-state slot of this KV head
      const uint32_t s = used % kSW;
      if (!mbar_wait(bar0 + s * 8, (used / kSW) & 1u, a.err)) {
        ok = false;
        *abort_flag = 1;
        break;
      }
      const uint32_t sb = stage0 + s * kSlotBytes;
      const uint32_t qb = sb + kKBytes;
      // K tile -> A fragments (2 blocks of 16 tokens x 8 blocks of 16 dims)
      uint32_t af[2][8][4];
#pragma unroll
      for (int mb = 0; mb < 2; ++mb) {
        const int t = mb * 16 + lm_row;
#pragma unroll
        for (int kb = 0; kb < 8; ++kb) {
          const int chunk = kb * 2 + lm_khalf;          // 16-byte chunk of the 256-byte row
          const uint32_t addr = sb + (chunk >> 3) * kBoxBytes + t * 128 + (((chunk & 7) ^ (t & 7)) << 4);
          ldmatrix_x4(addr, af[mb][kb]);
        }
      }
      // q rows -> B fragments (rows n >= G of the 8 columns are zero)
      uint32_t bf[8][2];
#pragma unroll
      for (int kb = 0; kb < 8; ++kb) {
        if (grp < G) {
          const uint32_t qa = qb + grp * kRowBytes + (kb * 16 + tig * 2) * 2;
          bf[kb][0] = lds32(qa);
          bf[kb][1] = lds32(qa + 16);
        } else {
          bf[kb][0] = 0u;
          bf[kb][1] = 0u;
        }
      }
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

      float acc[2][4];
#pragma unroll
      for (int mb = 0; mb < 2; ++mb)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[mb][e] = 0.f;
#pragma unroll
      for (int kb = 0; kb < 8; ++kb)
#pragma unroll
        for (int mb = 0; mb < 2; ++mb) mma_16816<DT>(acc[mb], af[mb][kb], bf[kb][0], bf[kb][1]);

      // acc[mb][0|1] = token mb*16 + grp, heads hA|hB; acc[mb][2|3] = token mb*16 + grp + 8
      if (RAW) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int mb = u >> 1, e = (u & 1) * 2;
          float v = (hA < G ? acc[mb][e] : 0.f) + (hB < G ? acc[mb][e + 1] : 0.f);
          v += __shfl_xor_sync(0xffffffffu, v, 1);
          v += __shfl_xor_sync(0xffffffffu, v, 2);
          rs[u] += v * kInvSqrtD;
        }
      } else {
        float zA[4], zB[4];
        bool tv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int mb = u >> 1, e = (u & 1) * 2;
          zA[u] = acc[mb][e] * kInvSqrtD;
          zB[u] = acc[mb][e + 1] * kInvSqrtD;
          tv[u] = (mb * 16 + grp + (u & 1) * 8) < nv;
        }
        float* lg = a.logits + ((int64_t)b * H + g * G) * cap + j0;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int t = (u >> 1) * 16 + grp + (u & 1) * 8;
          if (tv[u]) {
            if (hA < G) lg[(int64_t)hA * cap + t] = zA[u];
            if (hB < G) lg[(int64_t)hB * cap + t] = zB[u];
          }
        }
        // tile (max, sum exp) of heads hA and hB over the 8 lanes of this column pair
        float mA = -INFINITY, mB = -INFINITY;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (tv[u]) {
            mA = fmaxf(mA, zA[u]);
            mB = fmaxf(mB, zB[u]);
          }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          mA = fmaxf(mA, __shfl_xor_sync(0xffffffffu, mA, o));
          mB = fmaxf(mB, __shfl_xor_sync(0xffffffffu, mB, o));
        }
        float lA = 0.f, lB = 0.f;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (tv[u]) {
            lA += expf(zA[u] - mA);
            lB += expf(zB[u] - mB);
          }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          lA += __shfl_xor_sync(0xffffffffu, lA, o);
          lB += __shfl_xor_sync(0xffffffffu, lB, o);
        }
        if (lane < 4) {
          if (hA < G) wstat[sr * 8 + hA] = merge_ml(wstat[sr * 8 + hA], make_float2(mA, lA));
          if (hB < G) wstat[sr * 8 + hB] = merge_ml(wstat[sr * 8 + hB], make_float2(mB, lB));
        }
        __syncwarp();
      }
    }
    if (RAW) {
      // sum over the warps in a fixed order, double-buffered by item; a warp
      // whose wait timed out still reaches the barrier, and all warps then
      // leave together
      float* rb = red + (item_no & 1) * kNW * kT;
      if (tig == 0) {
#pragma unroll
        for (int u = 0; u < 4; ++u) rb[warp * kT + (u >> 1) * 16 + grp + (u & 1) * 8] = rs[u];
      }
      named_sync(1, kThreads);
      if (*abort_flag) break;
      if (warp == (item_no % kNW) && lane < nv) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < kNW; ++w) sum += rb[w * kT + lane];
        const int64_t o = (int64_t)b * cap + j0 + lane;
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
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.y;
  int len = a.lens[b];
  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  const int jb = blockIdx.x * kFinChunk;
  if (jb >= len) return;
  const int items = (len + kT - 1) / kT;
  const int ns = min(items, a.nslot);
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
  return launch_pdl(kern, dim3(grid), dim3(kThreads), smem, st, 0, a);
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
  return (size_t)ScoreCfg<G>::kBytes;
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
int score_warps() { return kNW; }
int score_max_batch() { return kMaxBatchSmem; }
int score_max_kv_heads(int G) {
  (void)G;
  return kMaxNg * kNW;
}

cudaError_t launch_score(const ScoreArgs& a, int dtype, int G, bool raw, int grid, cudaStream_t st) {
  if (dtype == 0) return raw ? launch_score_g<0, true>(a, G, grid, st) : launch_score_g<0, false>(a, G, grid, st);
  return raw ? launch_score_g<1, true>(a, G, grid, st) : launch_score_g<1, false>(a, G, grid, st);
}

cudaError_t launch_attn_finalize(const FinalizeArgs& a, cudaStream_t st) {
  dim3 grid((a.cap + kFinChunk - 1) / kFinChunk, a.B);
  return launch_pdl(hill_attn_finalize_kernel, grid, dim3(kFinThreads), 2 * a.H * sizeof(float), st, 0, a);
}

}  // namespace hill
