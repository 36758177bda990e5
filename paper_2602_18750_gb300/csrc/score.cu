// score.cu -- the K-cache streaming kernel (Eq. 1 over the whole cache) and
// the ATTN-mode normalisation (Sec. 4.1 column sum of softmax weights).
//
// hill_score_kernel: persistent CTAs of kNW warps.  A work item is a tile of
// kT = 32 consecutive tokens of one sequence; CTA x takes the contiguous
// range of items [x * per, (x + 1) * per), so it meets one or two sequences
// and loads their queries and flushes their partials once (measured faster
// than dealing items round robin, by 4 % at 32K and more for short
// sequences, where round robin changes sequence at every item).  The KV
// heads g of an item are dealt to the warps (g mod kNW).  Every warp streams
// its own (item, g)
// sequence through a private ring of kSW shared-memory stages: lane 0 issues
// two tiled TMA loads (dims 0-63 and 64-127 of the tile's 32 key rows, 128-
// byte swizzle) completing on the stage's mbarrier.  The warp moves a landed tile into
// registers with ldmatrix (conflict-free thanks to the swizzle), hands the
// slot back to the copy engine for the stage kSW ahead, and computes the
// [32 tokens x 128] . [128 x G heads] product with 16 mma.sync m16n8k16
// (fp32 accumulation; the G query heads fill the N = 8 columns, so one
// instruction stream serves MHA and GQA alike).
//
//   RAW : the per-token sum over heads is reduced across the warps in shared
//         memory at the end of each item (fixed order) and written to scores
//         (and added to accum).
//   ATTN: every logit, pre-scaled by log2 e, is written to a [B][H][cap]
//         buffer; each lane keeps a running (max, sum 2^(z2 - max)) of its
//         own tokens per head in registers, and the lanes of a head are
//         combined once, when the CTA leaves a sequence, into one partial per
//         (sequence, head, CTA).  hill_attn_finalize_kernel combines the
//         partials and forms s[b,j] = sum_h exp(z[b,h,j] - m_bh) / L_bh; when
//         that kernel would need more than two CTAs per SM (long sequences),
//         hill_attn_stats_kernel first combines the partials once per
//         (sequence, head).
//
// The query rows of a warp's heads are held as mma B fragments in registers
// for the whole sequence.  Before its dependency wait the kernel builds its
// tile table from the lengths and, with 16-bit keys, starts its first stages
// (inputs of the call only; every global write comes after the wait).
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

template <int G, bool F8>
struct ScoreCfg {
  // one K tile (a multiple of 1024): 8 KB of 16-bit keys, or 4 KB of E4M3 codes
  static constexpr int kSlotBytes = F8 ? kT * 128 : kKBytes;
  static constexpr int kSW = F8 ? 6 : 3;                   // stages per warp (same bytes in flight)
  static constexpr int kStages = kNW * kSW;
  // shared-memory layout (offsets from a 1024-byte aligned base)
  static constexpr int kOffScale = kStages * kSlotBytes;   // F8: the kT token scales of each stage
  static constexpr int kOffBar = kOffScale + (F8 ? kStages * kT * 4 : 0);
  static constexpr int kOffTab = kOffBar + kStages * 8;
  static constexpr int kOffRed = kOffTab + 2 * kTableInts * 4;
  static constexpr int kOffFlag = kOffRed + 2 * kNW * kT * 4;
  static constexpr int kOffIssued = kOffFlag + kNW * 4;       // warps that issued their last stage
  static constexpr int kBytes = kOffIssued + 16 + 1024;   // + alignment slack
};

constexpr int kL2Ahead = 4;   // stages per warp brought into L2 before the dependency wait
// Registers per thread of the scoring kernel: at most 192, so that one CTA
// of 256 threads at 64 registers (the two-kernel normalisation's finalize)
// still fits beside it in the SM's 65536 registers and the layer-pipelined
// evaluation can run it during the next layer's K stream.
constexpr int kScoreMaxRegs = 192;

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

// Position of a warp in its own stage sequence: item (global tile index), r
// (its r-th KV head of that item, g = goff + warp + r * kNW) and b (the item's
// sequence, advanced incrementally).
struct Cursor {
  int item, r, b;
};

template <int DT, int G, bool RAW, bool F8, bool DEAL>
__global__ void __maxnreg__(kScoreMaxRegs) hill_score_kernel(const __grid_constant__ ScoreArgs a) {
  using Cfg = ScoreCfg<G, F8>;
  constexpr int kSlotBytes = Cfg::kSlotBytes;
  constexpr int kSW = Cfg::kSW;
  constexpr int kStages = Cfg::kStages;
  // accumulator columns that can hold a head of the group: 2*tig (+1 when G > 1)
  constexpr int kCols = G >= 2 ? 2 : 1;
  // heads of the group this launch handles (G itself unless G is 4 or 8 and
  // the group is 3, or 5 to 7 heads: the query rows past Gn are zero)
  const int Gn = G <= 2 ? G : a.Gn;

  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw_addr = smem_addr(smem_raw);
  const uint32_t base_addr = (raw_addr + 1023u) & ~1023u;
  unsigned char* base = smem_raw + (base_addr - raw_addr);
  int* tstart = reinterpret_cast<int*>(base + Cfg::kOffTab);          // [B+1] tile prefix
  int* slen = tstart + kTableInts;                                     // [B] clamped lengths
  float* red = reinterpret_cast<float*>(base + Cfg::kOffRed);          // [2][kNW][kT]
  volatile int* abort_flag = reinterpret_cast<int*>(base + Cfg::kOffFlag);   // [kNW]: one per warp group

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int B = a.B, H = a.H, Hkv = a.Hkv, cap = a.cap;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(base_addr + Cfg::kOffBar + s * 8, 1);
    fence_barrier_init();
    for (int w = 0; w < kNW; ++w) abort_flag[w] = 0;
    *reinterpret_cast<int*>(base + Cfg::kOffIssued) = 0;
    prefetch_tmap(&a.kmap);
  }
  // Before the dependency wait this kernel reads only the inputs of the call
  // (lengths, and with 16-bit keys the K cache itself), which the caller has
  // completed before the call (include/hill.h): it builds the tile table and
  // starts the first stages of every warp, so their DRAM latency overlaps the
  // end of the previous kernel.  Every write to global memory (the histogram
  // zeroing, logits, partials, scores) comes after the wait.  The E4M3 shadow
  // is written by hill_quantize_k, possibly the kernel just before, so with
  // F8 the first loads wait too.
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
  const int per = (n_items + gridDim.x - 1) / gridDim.x;     // items per CTA
  const int it_lo = min(n_items, (int)blockIdx.x * per), it_hi = min(n_items, it_lo + per);
  // The warps' shares.  Without DEAL (W = 1) the KV heads are dealt to the
  // warps -- warp w takes g0 + r * kNW, r < ng (0 .. kMaxNg) -- and every warp
  // visits every item of the CTA.  With DEAL (launches of at most kNW / 2 KV
  // heads), W = kNW / nkv warps share each head and deal the items instead:
  // warp sub * nkv + i takes head goff + i of items it_lo + sub, + W, ...,
  // so that every warp streams (W * nkv < kNW leaves the rest idle).
  const int W = DEAL ? kNW / a.nkv : 1;
  const int sub = DEAL ? warp / a.nkv : 0;
  const int g0 = a.goff + (DEAL ? warp % a.nkv : warp);
  const int ng = DEAL ? (warp < W * a.nkv ? 1 : 0) : (a.nkv - warp + kNW - 1) / kNW;
  const int it0 = (DEAL && ng == 0) ? it_hi : it_lo + sub;   // this warp's first item
  // With DEAL a warp holds one KV head, and the query heads of its group in
  // up to kMaxNg sub-groups of 8 (a launch covers up to 32 heads per KV head):
  // each K tile is read once and scored for every sub-group, so groups larger
  // than 8 stream their keys once.  Fragment/statistics slot q of a warp is
  // its q-th KV head (no DEAL) or its q-th sub-group (DEAL).
  const int nsub = DEAL ? (a.Gn + 7) / 8 : 1;
  auto head0_of = [&](int q) {   // first query head of slot q
    return (DEAL ? g0 : g0 + q * kNW) * a.Gs + a.hoff + (DEAL ? 8 * q : 0);
  };
  auto gn_of = [&](int q) { return DEAL ? min(8, a.Gn - 8 * q) : Gn; };   // heads of slot q

  const uint64_t pol = l2_evict_first_policy();
  // the logits stay in L2 until the normalisation reads (and discards) them
  const uint64_t pol_keep = l2_evict_last_policy();
  const uint32_t stage0 = base_addr + warp * kSW * kSlotBytes;
  const uint32_t bar0 = base_addr + Cfg::kOffBar + warp * kSW * 8;
  const uint32_t scale0 = base_addr + Cfg::kOffScale + warp * kSW * kT * 4;   // F8 only
  const int b_first = it0 < it_hi ? find_seq(tstart, B, it0) : 0;

  auto advance = [&](Cursor& c) {
    if (++c.r >= ng) {
      c.r = 0;
      c.item += W;
      while (c.b < B - 1 && tstart[c.b + 1] <= c.item) ++c.b;
    }
  };
  // lane 0: load the K tile of position c into slot s
  auto issue = [&](const Cursor& c, uint32_t s) {
    const int j0 = (c.item - tstart[c.b]) * kT;
    const int g = g0 + c.r * kNW;
    const uint32_t fb = bar0 + s * 8;
    const uint32_t dst = stage0 + s * kSlotBytes;
    // tensor-map coordinates: dimension 0 is d, the others are ordered by stride
    const int c1 = a.kdim_tok == 1 ? j0 : (a.kdim_head == 1 ? g : c.b);
    const int c2 = a.kdim_tok == 2 ? j0 : (a.kdim_head == 2 ? g : c.b);
    const int c3 = a.kdim_tok == 3 ? j0 : (a.kdim_head == 3 ? g : c.b);
    if constexpr (F8) {
      // 32 rows of 128 codes (one swizzled box) and the rows' 32 scales
      mbar_arrive_expect_tx(fb, (uint32_t)(kSlotBytes + kT * 4));
      tma_load_4d(dst, &a.kmap, 0, c1, c2, c3, fb, pol);
      bulk_g2s(scale0 + s * kT * 4, a.kscale + ((int64_t)c.b * Hkv + g) * a.cap32 + j0, kT * 4, fb, pol);
    } else {
      mbar_arrive_expect_tx(fb, (uint32_t)kKBytes);
      tma_load_4d(dst, &a.kmap, 0, c1, c2, c3, fb, pol);
      tma_load_4d(dst + kBoxBytes, &a.kmap, 64, c1, c2, c3, fb, pol);
    }
  };

  // prologue: the first kSW stages of this warp
  Cursor pc{it0, 0, b_first};
  uint32_t issued = 0, is_slot = 0;
  // with 16-bit keys, once every warp of the CTA has issued its last stage the
  // next kernel may launch (its CTAs take the SMs this grid's CTAs leave as
  // they drain); the E4M3 path, whose loads wait for the shadow's row of this
  // step, measured slower so and keeps the release at exit
  bool marked = F8;
  auto mark_if_done = [&]() {
    if (!marked && (ng == 0 || pc.item >= it_hi)) {
      marked = true;
      if (lane == 0 && atomicAdd(reinterpret_cast<int*>(base + Cfg::kOffIssued), 1) == kNW - 1)
        pdl_launch_dependents();
    }
  };
  auto prologue = [&]() {
    if (ng > 0) {
      for (; issued < (uint32_t)kSW && pc.item < it_hi; ++issued) {
        if (lane == 0) issue(pc, is_slot);
        is_slot = is_slot + 1 == (uint32_t)kSW ? 0u : is_slot + 1;
        advance(pc);
      }
    }
  };
  if constexpr (!F8) {
    prologue();
    // and the next kL2Ahead stages into L2, so that the HBM stream keeps going
    // while the previous kernel finishes
    if (lane == 0 && ng > 0) {
      Cursor lc = pc;
      for (int u = 0; u < kL2Ahead && lc.item < it_hi; ++u) {
        const int j0 = (lc.item - tstart[lc.b]) * kT;
        const int g = g0 + lc.r * kNW;
        const int c1 = a.kdim_tok == 1 ? j0 : (a.kdim_head == 1 ? g : lc.b);
        const int c2 = a.kdim_tok == 2 ? j0 : (a.kdim_head == 2 ? g : lc.b);
        const int c3 = a.kdim_tok == 3 ? j0 : (a.kdim_head == 3 ? g : lc.b);
        tma_prefetch_l2_4d(&a.kmap, 0, c1, c2, c3);
        tma_prefetch_l2_4d(&a.kmap, 64, c1, c2, c3);
        advance(lc);
      }
    }
  }
  pdl_wait();
  // No trigger here: a dependent launches once every CTA has issued its last
  // stage (mark_if_done) or exited.  A trigger at the start would let the next
  // layer's scoring grid (the next launch in this stream) take the SMs this
  // grid leaves free for the normalisation and selection running beside it
  // on another stream; one at the last issued stage lets it start on the SMs
  // this grid's CTAs release as they drain.
  if (a.hist0) {   // this CTA's share of the leading-digit histogram, zeroed for the normalisation
    const int64_t hper = (a.hist0_words + gridDim.x - 1) / gridDim.x;
    const int64_t w0 = min((int64_t)blockIdx.x * hper, a.hist0_words);
    const int64_t w1 = min(w0 + hper, a.hist0_words);
    for (int64_t w = w0 + threadIdx.x; w < w1; w += kThreads) a.hist0[w] = 0u;
  }
  if (it_lo >= it_hi) return;
  if constexpr (F8) prologue();
  mark_if_done();

  // fragment coordinates (mma.sync m16n8k16): C row = token lane/4 (+8),
  // C columns = heads 2*(lane%4) and 2*(lane%4)+1 of the group
  const int grp = lane >> 2, tig = lane & 3;
  // ldmatrix row address pieces: matrix m = lane/8 covers rows (m&1)*8.., k half m>>1
  const int lm_row = (lane & 7) + ((lane >> 3) & 1) * 8;
  const int lm_khalf = lane >> 4;
  uint32_t used = 0, cs = 0, cph = 0;      // stages consumed; slot and phase of the next one
  int item_no = 0;
  bool ok = true;
  int cur_b = -1, cur_slot = 0;

  // q of this warp's heads for the current sequence, as mma B fragments:
  // column grp is query head g*Gs + hoff + grp (zero for grp >= Gn), k = 16*kb + 2*tig (+8)
  // F8: the same rows cast to E4M3 with one scale per head, as m16n8k32 B
  // fragments (k = 32*kb + 4*tig .. +3, and +16), and the scales of this
  // lane's accumulator columns (heads 2*tig and 2*tig + 1)
  uint32_t bq[kMaxNg][F8 ? 4 : 8][2];
  float sqA[kMaxNg], sqB[kMaxNg];
  auto load_q = [&](int b) {
#pragma unroll
    for (int r = 0; r < kMaxNg; ++r) {
      const bool has = (DEAL ? (ng > 0 && r < nsub) : r < ng) && grp < gn_of(r);
      const int64_t row = has ? (int64_t)b * a.q_sb + (int64_t)(head0_of(r) + grp) * a.q_sh : 0;
      if constexpr (F8) {
        const auto* qh = static_cast<const uint16_t*>(a.q) + row;
        float v[4][8];
        float amax = 0.f;
#pragma unroll
        for (int kb = 0; kb < 4; ++kb) {
          uint2 lo{0u, 0u}, hi{0u, 0u};
          if (has) {
            lo = __ldg(reinterpret_cast<const uint2*>(qh + kb * 32 + 4 * tig));
            hi = __ldg(reinterpret_cast<const uint2*>(qh + kb * 32 + 16 + 4 * tig));
          }
          to_float8<DT>(uint4{lo.x, lo.y, hi.x, hi.y}, v[kb]);
#pragma unroll
          for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(v[kb][i]));
        }
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 2));   // the head's 4 lanes hold all 128 dims
        const float rq = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
#pragma unroll
        for (int kb = 0; kb < 4; ++kb) {
          bq[r][kb][0] = e4m3x2(__fmul_rn(v[kb][0], rq), __fmul_rn(v[kb][1], rq)) |
                         (e4m3x2(__fmul_rn(v[kb][2], rq), __fmul_rn(v[kb][3], rq)) << 16);
          bq[r][kb][1] = e4m3x2(__fmul_rn(v[kb][4], rq), __fmul_rn(v[kb][5], rq)) |
                         (e4m3x2(__fmul_rn(v[kb][6], rq), __fmul_rn(v[kb][7], rq)) << 16);
        }
        const float sq = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
        sqA[r] = __shfl_sync(0xffffffffu, sq, 8 * tig);
        sqB[r] = __shfl_sync(0xffffffffu, sq, 8 * tig + 4);
      } else {
        const auto* q32 = static_cast<const uint32_t*>(a.q);
#pragma unroll
        for (int kb = 0; kb < 8; ++kb) {
          bq[r][kb][0] = has ? __ldg(q32 + row / 2 + kb * 8 + tig) : 0u;
          bq[r][kb][1] = has ? __ldg(q32 + row / 2 + kb * 8 + 4 + tig) : 0u;
        }
        sqA[r] = sqB[r] = 1.f;
      }
    }
  };
  // ATTN: this lane's running (max, sum 2^(z2 - max)) over its own tokens of
  // the current sequence, per KV head r and column c (z2 = logit * log2 e);
  // lanes are combined only when the CTA leaves the sequence
  float st_m[kMaxNg][kCols], st_l[kMaxNg][kCols];
  auto reset_stat = [&]() {
#pragma unroll
    for (int r = 0; r < kMaxNg; ++r)
#pragma unroll
      for (int c = 0; c < kCols; ++c) {
        st_m[r][c] = kNegHuge;
        st_l[r][c] = 0.f;
      }
  };
  auto flush = [&]() {
#pragma unroll
    for (int r = 0; r < kMaxNg; ++r) {
      if (DEAL ? (ng == 0 || r >= nsub) : r >= ng) break;
#pragma unroll
      for (int c = 0; c < kCols; ++c) {
        float m = st_m[r][c], l = st_l[r][c];
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {   // the 8 lanes of one column
          const float mo = __shfl_xor_sync(0xffffffffu, m, o);
          const float lo = __shfl_xor_sync(0xffffffffu, l, o);
          const float mn = fmaxf(m, mo);
          l = l * ex2(m - mn) + lo * ex2(mo - mn);
          m = mn;
        }
        const int hl = 2 * tig + c;
        if (grp == 0 && hl < gn_of(r))
          a.partials[((int64_t)cur_b * a.nslot + cur_slot) * H + head0_of(r) + hl] = make_float2(m, l);
      }
    }
  };
  // ATTN with DEAL: a warp owns one partial slot in every sequence its CTA
  // meets, and writes a neutral one (-inf, 0) where it visited no tile of it
  // (the normalisation skips entries whose sum is 0).  b_next: the first
  // sequence of the CTA this warp has not written yet.
  const int b_cta_last = it_lo < it_hi ? find_seq(tstart, B, it_hi - 1) : -1;
  int b_next = it_lo < it_hi ? find_seq(tstart, B, it_lo) : 0;
  auto neutral_until = [&](int b_end) {   // sequences [b_next, b_end)
    if constexpr (!RAW && DEAL) {
      if (ng == 0) return;
      for (; b_next < b_end; ++b_next) {
        if (tstart[b_next + 1] == tstart[b_next]) continue;   // empty: no slots
        const int slot = ((int)blockIdx.x - tstart[b_next] / per) * W + sub;
#pragma unroll
        for (int q = 0; q < kMaxNg; ++q) {
          if (q >= nsub) break;
#pragma unroll
          for (int c = 0; c < kCols; ++c) {
            const int hl = 2 * tig + c;
            if (grp == 0 && hl < gn_of(q))
              a.partials[((int64_t)b_next * a.nslot + slot) * H + head0_of(q) + hl] = make_float2(-INFINITY, 0.f);
          }
        }
      }
    }
  };

  for (int item = it0, b = b_first; item < it_hi; item += W, ++item_no) {
    while (b < B - 1 && tstart[b + 1] <= item) ++b;
    const int tile = item - tstart[b];
    const int j0 = tile * kT;
    const int nv = min(kT, slen[b] - j0);
    float rs[4] = {0.f, 0.f, 0.f, 0.f};   // RAW: token sums of rows grp, grp+8, 16+grp, 24+grp

    if (b != cur_b) {
      if (!RAW && cur_b >= 0) flush();
      neutral_until(b);
      b_next = b + 1;
      load_q(b);
      if (!RAW) reset_stat();
      cur_b = b;
      // this warp's partial slot in b: the CTA's rank among the CTAs whose
      // ranges meet b, times W, plus the warp's item share
      cur_slot = ((int)blockIdx.x - tstart[b] / per) * W + sub;
    }

    constexpr int kStagesPerItem = DEAL ? 1 : kMaxNg;   // (at most; ng of them)
#pragma unroll
    for (int r = 0; r < kStagesPerItem; ++r) {
      if (r >= ng || !ok) break;
      const int g = DEAL ? g0 : g0 + r * kNW;
      // every lane waits; the warp goes on only if all of them saw the phase
      // complete, so it takes the same path and its shuffles stay converged
      if (!__all_sync(0xffffffffu, mbar_wait(bar0 + cs * 8, cph, a.err))) {
        ok = false;
        abort_flag[sub] = 1;
        break;
      }
      const uint32_t sb = stage0 + cs * kSlotBytes;
      // K tile -> A fragments: 16-bit keys, 2 blocks of 16 tokens x 8 blocks
      // of 16 dims; E4M3 codes, 2 blocks of 16 tokens x 4 blocks of 32 dims
      constexpr int kKB = F8 ? 4 : 8;
      uint32_t af[2][kKB][4];
#pragma unroll
      for (int mb = 0; mb < 2; ++mb) {
        const int t = mb * 16 + lm_row;
#pragma unroll
        for (int kb = 0; kb < kKB; ++kb) {
          const int chunk = kb * 2 + lm_khalf;   // 16-byte chunk of the row
          const uint32_t addr = F8 ? sb + t * 128 + ((chunk ^ (t & 7)) << 4)
                                   : sb + (chunk >> 3) * kBoxBytes + t * 128 + (((chunk & 7) ^ (t & 7)) << 4);
          ldmatrix_x4(addr, af[mb][kb]);
        }
      }
      // F8: the scales of this lane's token rows mb*16 + grp (+8)
      float ksc[4] = {1.f, 1.f, 1.f, 1.f};
      if constexpr (F8) {
        const uint32_t sc = scale0 + cs * kT * 4;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          ksc[u] = __uint_as_float(lds32(sc + ((u >> 1) * 16 + grp + (u & 1) * 8) * 4));
      }
      ++used;
      cph ^= (cs + 1 == (uint32_t)kSW) ? 1u : 0u;
      const uint32_t freed = cs;
      cs = cs + 1 == (uint32_t)kSW ? 0u : cs + 1;
      __syncwarp();
      if (pc.item < it_hi) {   // the slot just read takes the stage kSW ahead
        if (lane == 0) {
          fence_proxy_async_smem();
          issue(pc, freed);
        }
        ++issued;
        advance(pc);
        mark_if_done();
      }

      // the tile is scored for each fragment slot q: this stage's KV head
      // (no DEAL), or every query sub-group of the warp's KV head (DEAL)
      constexpr int kSlotsPerStage = DEAL ? kMaxNg : 1;
#pragma unroll
      for (int qs = 0; qs < kSlotsPerStage; ++qs) {
      if (DEAL && qs >= nsub) break;
      const int q = DEAL ? qs : r;
      const int hq0 = head0_of(q);    // first query head of the slot
      const int gnq = gn_of(q);       // its heads
      float acc[2][4];
#pragma unroll
      for (int mb = 0; mb < 2; ++mb)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[mb][e] = 0.f;
#pragma unroll
      for (int kb = 0; kb < kKB; ++kb)
#pragma unroll
        for (int mb = 0; mb < 2; ++mb) {
          if constexpr (F8) mma_16832_e4m3(acc[mb], af[mb][kb], bq[q][kb][0], bq[q][kb][1]);
          else mma_16816<DT>(acc[mb], af[mb][kb], bq[q][kb][0], bq[q][kb][1]);
        }
      if constexpr (F8) {   // back to the key and query scales
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc[u >> 1][(u & 1) * 2] *= sqA[q] * ksc[u];
          acc[u >> 1][(u & 1) * 2 + 1] *= sqB[q] * ksc[u];
        }
      }

      // acc[mb][c] = token mb*16 + grp, column 2*tig + c; acc[mb][2 + c] = token
      // mb*16 + grp + 8.  Columns >= Gn are zero (their q fragments are zero).
      if constexpr (RAW) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int mb = u >> 1, e = (u & 1) * 2;
          float v = acc[mb][e];
          if constexpr (G >= 2) v += acc[mb][e + 1];
          if constexpr (G >= 4) v += __shfl_xor_sync(0xffffffffu, v, 1);
          if constexpr (G >= 8) v += __shfl_xor_sync(0xffffffffu, v, 2);
          // complete in the tig == 0 lanes
          if (a.kvh) {   // per-KV-head importance: this group's sum is the score of (b, g)
            const int t = mb * 16 + grp + (u & 1) * 8;
            if (tig == 0 && t < nv) {
              const int64_t o = ((int64_t)b * Hkv + g) * cap + j0 + t;
              const float val = v * kInvSqrtD;
              // later sub-groups of the same KV head add to the first one's sum
              if (a.scores) a.scores[o] = (a.raw_add || qs > 0) ? a.scores[o] + val : val;
              if (a.accum) a.accum[o] += val;
            }
          } else {
            rs[u] += v;
          }
        }
      } else {
        float* lg = a.logits + ((int64_t)b * H + hq0) * a.lstride + j0;
#pragma unroll
        for (int c = 0; c < kCols; ++c) {
          const int hl = 2 * tig + c;
          float z[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int mb = u >> 1, e = (u & 1) * 2 + c;
            const int t = mb * 16 + grp + (u & 1) * 8;
            z[u] = t < nv ? acc[mb][e] * kLog2eInvSqrtD : -INFINITY;
            if (t < nv && hl < gnq) st_global_hint(lg + (int64_t)hl * a.lstride + t, z[u], pol_keep);
          }
          const float mn = fmaxf(st_m[q][c], fmaxf(fmaxf(z[0], z[1]), fmaxf(z[2], z[3])));
          st_l[q][c] = st_l[q][c] * ex2(st_m[q][c] - mn) +
                       ((ex2(z[0] - mn) + ex2(z[1] - mn)) + (ex2(z[2] - mn) + ex2(z[3] - mn)));
          st_m[q][c] = mn;
        }
      }
      }   // fragment slots
    }
    if (RAW && !a.kvh) {
      // sum over the warps holding the item's heads -- all kNW (W = 1), or
      // the nkv warps of group sub -- in a fixed order, double-buffered by
      // item; a warp whose wait timed out still reaches its group's barrier
      // after raising the group's flag, and the group then leaves together
      const int wg0 = DEAL ? sub * a.nkv : 0, gw = DEAL ? a.nkv : kNW;
      float* rb = red + (item_no & 1) * kNW * kT;
      if (tig == 0) {
#pragma unroll
        for (int u = 0; u < 4; ++u) rb[warp * kT + (u >> 1) * 16 + grp + (u & 1) * 8] = rs[u];
      }
      named_sync(1 + sub, gw * 32);
      if (abort_flag[sub]) break;
      if (warp == wg0 + item_no % gw && lane < nv) {
        float sum = 0.f;
        for (int w = 0; w < gw; ++w) sum += rb[(wg0 + w) * kT + lane];
        sum *= kInvSqrtD;
        const int64_t o = (int64_t)b * cap + j0 + lane;
        if (a.scores) a.scores[o] = a.raw_add ? a.scores[o] + sum : sum;
        if (a.accum) a.accum[o] += sum;
      }
    } else if (!ok) {
      break;
    }
  }
  if (!RAW && cur_b >= 0 && ok) flush();
  if (ok) neutral_until(b_cta_last + 1);
  // after a timeout: give every copy this warp issued and did not consume one
  // more bounded wait before the CTA's shared memory is released
  if (!ok && lane == 0) {
    for (uint32_t u = used; u < issued; ++u) mbar_wait(bar0 + (u % kSW) * 8, (u / kSW) & 1u, a.err);
  }
}

// Combine the per-CTA (max, sum) partials of every head of sequence b, then
// s[b,j] = sum_h 2^(z2[b,h,j] - m_h) / L_h, one token per thread (logits and
// partials are in the base-2 scale z2 = z * log2 e, so each term is the
// softmax weight e^(z - m) / sum e^(z - m)).  Both phases issue all their
// loads before using them: the partials of a head are spread over 8 threads,
// and each thread loads the logits of 16 heads of its token at once (they
// were just written and are mostly L2 resident).
constexpr int kFinThreads = 256;
constexpr int kFinChunk = kFinThreads;
constexpr int kFinPartThreads = 8;                 // threads combining one head
constexpr int kFinPartMax = 32;                    // partials per thread held in registers
constexpr int kFinPartFew = 4;                     // the same when a sequence has few (<= 32) slots
constexpr int kHistBins = 2048;                    // leading 11 bits of the order-preserving key
constexpr int kFinZReg = 32;                       // logits per token held in registers
constexpr int kFinMaxTpt = 16;                     // token blocks per CTA at most (split step)

// Combine the ns per-CTA partials (max, sum) of every head of sequence b into
// mh[h] (max) and il[h] (1 / sum): kFinPartThreads threads per head, each
// holding PM partials in registers with all their loads in flight; slots
// beyond PM * kFinPartThreads are folded in sequentially.  A warp covers
// kHeadsPerWarp consecutive heads per pass.  The loop runs while the warp's
// first head exists, so every lane of a warp takes the same trips and the
// full-mask shuffles always have all 32 lanes; lanes whose head is past H
// combine nothing and write nothing.
template <int PM>
__device__ __forceinline__ void combine_partials(const FinalizeArgs& a, int b, int ns, float* mh, float* il) {
  const float2* pb = a.partials + (int64_t)b * a.nslot * a.H;
  const int sub = threadIdx.x % kFinPartThreads;
  constexpr int kHeadsPerWarp = 32 / kFinPartThreads;
  for (int h0 = (threadIdx.x >> 5) * kHeadsPerWarp; h0 < a.H; h0 += kFinThreads / kFinPartThreads) {
    const int h = h0 + (threadIdx.x & 31) / kFinPartThreads;
    const bool hv = h < a.H;
    float2 p[PM];
#pragma unroll
    for (int u = 0; u < PM; ++u) {
      const int s = sub + u * kFinPartThreads;
      p[u] = hv && s < ns ? pb[(int64_t)s * a.H + h] : make_float2(-INFINITY, 0.f);
    }
    float m = -INFINITY;
#pragma unroll
    for (int u = 0; u < PM; ++u) m = fmaxf(m, p[u].x);
    for (int s = sub + PM * kFinPartThreads; hv && s < ns; s += kFinPartThreads)
      m = fmaxf(m, pb[(int64_t)s * a.H + h].x);
#pragma unroll
    for (int o = kFinPartThreads / 2; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float l = 0.f;
#pragma unroll
    for (int u = 0; u < PM; ++u) l += p[u].y > 0.f ? p[u].y * ex2(p[u].x - m) : 0.f;
    for (int s = sub + PM * kFinPartThreads; hv && s < ns; s += kFinPartThreads) {
      const float2 q = pb[(int64_t)s * a.H + h];
      l += q.y > 0.f ? q.y * ex2(q.x - m) : 0.f;
    }
#pragma unroll
    for (int o = kFinPartThreads / 2; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    if (sub == 0 && hv) {
      mh[h] = m;
      il[h] = 1.f / l;
    }
  }
}

// STATS: the per-head (max, 1/sum) come from hill_attn_stats_kernel instead of
// every CTA combining the partials itself (long sequences: many CTAs).  KVH:
// per-KV-head importance (a.kvh), a variant of its own so that its group sums
// do not weigh on the registers of the plain kernel.
template <bool STATS, bool KVH>
__global__ void __launch_bounds__(kFinThreads, STATS ? 4 : 2) hill_attn_finalize_kernel(FinalizeArgs a) {
  extern __shared__ float fsm[];
  float* mh = fsm;            // [H]
  float* il = fsm + a.H;      // [H]
  uint32_t* hcount = reinterpret_cast<uint32_t*>(fsm + 2 * a.H);   // [kHistBins] when a.hist0
  // The lengths are inputs of the call: this kernel only ever follows the
  // scoring kernel of the same call, whose own dependency wait covered every
  // earlier write, so they are read before this kernel's wait and overlap
  // the end of the scoring kernel.  Everything the scoring kernel writes
  // (logits, partials) is read after the wait.
  const int b = blockIdx.y;
  int len = a.lens[b];
  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  // this CTA's tokens: a.tpt blocks of kFinChunk from jb
  const int jb = blockIdx.x * kFinChunk * a.tpt;
  if (jb >= len) return;
  // the scoring CTAs that met b wrote slots 0 .. ns-1
  // (every thread counts the tiles of a share of the sequences)
  __shared__ int s_first, s_total;
  if (threadIdx.x == 0) s_first = s_total = 0;
  __syncthreads();
  {
    int f = 0, t = 0;
    for (int bb = threadIdx.x; bb < a.B; bb += kFinThreads) {
      int lb = a.lens[bb];
      lb = lb < 0 ? 0 : (lb > a.cap ? a.cap : lb);
      const int tiles = (lb + kT - 1) / kT;
      f += bb < b ? tiles : 0;
      t += tiles;
    }
    if (f) atomicAdd(&s_first, f);
    if (t) atomicAdd(&s_total, t);
  }
  __syncthreads();
  const int first_item = s_first;
  const int grid = a.nslot / a.spc;   // CTAs of the scoring launch
  const int per = (s_total + grid - 1) / grid;
  const int items = (len + kT - 1) / kT;
  const int ns = ((first_item + items - 1) / per - first_item / per + 1) * a.spc;
  pdl_wait();
  pdl_launch_dependents();
  // this token's logits of the first kFinZReg heads, loaded before the
  // partials are combined so that both round trips overlap
  int j = jb + threadIdx.x;
  bool valid = j < len;
  const float* zp = a.logits + (int64_t)b * a.H * a.lstride + j;
  float zr[kFinZReg];
#pragma unroll
  for (int u = 0; u < kFinZReg; ++u) zr[u] = (valid && u < a.H) ? zp[(int64_t)u * a.lstride] : 0.f;
  if constexpr (STATS) {
    for (int h = threadIdx.x; h < a.H; h += kFinThreads) {
      const float2 st = a.stats[(int64_t)b * a.H + h];
      mh[h] = st.x;
      il[h] = st.y;
    }
  }
  if constexpr (!STATS) {
    // ns is the same for the whole CTA, so every warp takes the same branch
    if (ns <= kFinPartThreads * kFinPartFew) combine_partials<kFinPartFew>(a, b, ns, mh, il);
    else combine_partials<kFinPartMax>(a, b, ns, mh, il);
  }
  if (a.hist0)
    for (int i = threadIdx.x; i < kHistBins; i += kFinThreads) hcount[i] = 0u;
  __syncthreads();
  for (int blk = 0;;) {   // the CTA's token blocks (one unless a.tpt > 1)
  if (KVH && valid) {
    // per-KV-head importance: the sum over each group of G query heads,
    // stored as soon as the group is complete (heads of a group are adjacent)
    const int G = a.H / a.Hkv;
    int g = 0, in_g = 0;   // the group being summed and its heads so far
    auto put = [&](float v) {
      const int64_t o = ((int64_t)b * a.Hkv + g) * a.cap + j;
      if (a.scores) a.scores[o] = v;
      if (a.accum) a.accum[o] += v;
    };
    float sg = 0.f;
#pragma unroll
    for (int u = 0; u < kFinZReg; ++u)
      if (u < a.H) {
        sg += ex2(zr[u] - mh[u]) * il[u];
        if (++in_g == G) {
          put(sg);
          ++g;
          in_g = 0;
          sg = 0.f;
        }
      }
    for (int h = kFinZReg; h < a.H; h += 16) {
      float z[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) z[u] = h + u < a.H ? zp[(int64_t)(h + u) * a.lstride] : 0.f;
#pragma unroll
      for (int u = 0; u < 16; ++u)
        if (h + u < a.H) {
          sg += ex2(z[u] - mh[h + u]) * il[h + u];
          if (++in_g == G) {
            put(sg);
            ++g;
            in_g = 0;
            sg = 0.f;
          }
        }
    }
  } else if (!KVH && valid) {
    float s = 0.f;
#pragma unroll
    for (int u = 0; u < kFinZReg; ++u)
      if (u < a.H) s += ex2(zr[u] - mh[u]) * il[u];
    int h = kFinZReg;
    for (; h + 16 <= a.H; h += 16) {
      float z[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) z[u] = zp[(int64_t)(h + u) * a.lstride];
#pragma unroll
      for (int u = 0; u < 16; ++u) s += ex2(z[u] - mh[h + u]) * il[h + u];
    }
    for (; h < a.H; ++h) s += ex2(zp[(int64_t)h * a.lstride] - mh[h]) * il[h];
    const int64_t o = (int64_t)b * a.cap + j;
    if (a.scores) a.scores[o] = s;
    float key = s;
    if (a.accum) {
      key = a.accum[o] + s;
      a.accum[o] = key;
    }
    if (a.hist0 && j < len - min(a.recent, len)) atomicAdd(&hcount[ordered_key(key) >> 21], 1u);
  }
  // The logits are dead once read: drop this warp's lines from L2 without
  // writing them back (each 128-byte line holds the warp's 32 tokens of one
  // head; every lane has consumed its loads before the warp passes the sync).
  {
    const int j0 = j - (int)(threadIdx.x & 31);
    __syncwarp();
    if (j0 < len)
      for (int h = threadIdx.x & 31; h < a.H; h += 32)
        l2_discard_line(a.logits + ((int64_t)b * a.H + h) * a.lstride + j0);
  }
  // the next block of tokens (its logits loaded before they are used)
  if (++blk >= a.tpt || jb + blk * kFinChunk >= len) break;
  j = jb + blk * kFinChunk + threadIdx.x;
  valid = j < len;
  zp = a.logits + (int64_t)b * a.H * a.lstride + j;
#pragma unroll
  for (int u = 0; u < kFinZReg; ++u) zr[u] = (valid && u < a.H) ? zp[(int64_t)u * a.lstride] : 0.f;
  }
  if (a.hist0) {
    __syncthreads();
    uint32_t* hg = a.hist0 + (int64_t)b * kHistBins;
    for (int i = threadIdx.x; i < kHistBins; i += kFinThreads) {
      const uint32_t v = hcount[i];
      if (v) atomicAdd(hg + i, v);
    }
  }
}

// Combine the per-CTA (max, sum) partials of one (b, h) into its softmax
// statistics (max, 1 / sum) in the base-2 scale: one warp per pair, each lane
// taking every 32nd partial with a running maximum, the lanes then merged by
// shuffles.  Used ahead of hill_attn_finalize_kernel<true, *> when the
// normalisation has many CTAs per sequence.
constexpr int kStatsWarps = 8;
constexpr int kStatsPer = 8;   // partials per lane whose loads are in flight together

__global__ void __launch_bounds__(kStatsWarps * 32) hill_attn_stats_kernel(FinalizeArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pair = blockIdx.x * kStatsWarps + warp;
  if (pair >= a.B * a.H) return;
  const int b = pair / a.H, h = pair - b * a.H;
  // the slots 0 .. ns-1 of b (lengths are inputs of the call: read before the wait)
  int f = 0, t = 0;
  for (int bb = lane; bb < a.B; bb += 32) {
    int lb = a.lens[bb];
    lb = lb < 0 ? 0 : (lb > a.cap ? a.cap : lb);
    const int tiles = (lb + kT - 1) / kT;
    f += bb < b ? tiles : 0;
    t += tiles;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    f += __shfl_xor_sync(0xffffffffu, f, o);
    t += __shfl_xor_sync(0xffffffffu, t, o);
  }
  int len = a.lens[b];
  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  const int items = (len + kT - 1) / kT;
  const int grid = a.nslot / a.spc;   // CTAs of the scoring launch
  const int per = (t + grid - 1) / grid;
  const int ns = items == 0 ? 0 : ((f + items - 1) / per - f / per + 1) * a.spc;
  pdl_wait();
  pdl_launch_dependents();
  const float2* pb = a.partials + (int64_t)b * a.nslot * a.H + h;
  float m = -INFINITY, l = 0.f;
  for (int s0 = lane; s0 < ns; s0 += 32 * kStatsPer) {
    float2 p[kStatsPer];
#pragma unroll
    for (int u = 0; u < kStatsPer; ++u) {
      const int s = s0 + 32 * u;
      p[u] = s < ns ? pb[(int64_t)s * a.H] : make_float2(-INFINITY, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kStatsPer; ++u) {
      if (!(p[u].y > 0.f)) continue;
      const float mn = fmaxf(m, p[u].x);
      l = l * ex2(m - mn) + p[u].y * ex2(p[u].x - mn);
      m = mn;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float mo = __shfl_xor_sync(0xffffffffu, m, o);
    const float lo = __shfl_xor_sync(0xffffffffu, l, o);
    const float mn = fmaxf(m, mo);
    l = (l > 0.f ? l * ex2(m - mn) : 0.f) + (lo > 0.f ? lo * ex2(mo - mn) : 0.f);
    m = mn;
  }
  if (lane == 0) a.stats[pair] = make_float2(m, 1.f / l);
}

template <int DT, int G, bool RAW, bool F8, bool DEAL>
cudaError_t launch_score_t(const ScoreArgs& a, int grid, cudaStream_t st) {
  const size_t smem = (size_t)ScoreCfg<G, F8>::kBytes;
  auto kern = hill_score_kernel<DT, G, RAW, F8, DEAL>;
  static int cache[64] = {0};
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), (int)smem, cache);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(kThreads), smem, st, 0, a);
}

template <int DT, bool RAW, bool F8>
cudaError_t launch_score_g(const ScoreArgs& a, int G, bool deal, int grid, cudaStream_t st) {
  if (deal) return G == 8 ? launch_score_t<DT, 8, RAW, F8, true>(a, grid, st) : cudaErrorInvalidValue;
  switch (G) {
    case 1: return launch_score_t<DT, 1, RAW, F8, false>(a, grid, st);
    case 2: return launch_score_t<DT, 2, RAW, F8, false>(a, grid, st);
    case 4: return launch_score_t<DT, 4, RAW, F8, false>(a, grid, st);
    case 8: return launch_score_t<DT, 8, RAW, F8, false>(a, grid, st);
  }
  return cudaErrorInvalidValue;
}

template <int DT, bool F8>
cudaError_t launch_score_m(const ScoreArgs& a, int G, bool raw, bool deal, int grid, cudaStream_t st) {
  return raw ? launch_score_g<DT, true, F8>(a, G, deal, grid, st)
             : launch_score_g<DT, false, F8>(a, G, deal, grid, st);
}

}  // namespace

size_t score_smem_bytes(int G, bool f8) {
  switch (G) {
    case 1: return f8 ? ScoreCfg<1, true>::kBytes : ScoreCfg<1, false>::kBytes;
    case 2: return f8 ? ScoreCfg<2, true>::kBytes : ScoreCfg<2, false>::kBytes;
    case 4: return f8 ? ScoreCfg<4, true>::kBytes : ScoreCfg<4, false>::kBytes;
    default: return f8 ? ScoreCfg<8, true>::kBytes : ScoreCfg<8, false>::kBytes;
  }
}

int score_tile_tokens() { return kT; }
int score_warps() { return kNW; }
int score_max_batch() { return kMaxBatchSmem; }
int score_max_kv_heads() { return kMaxNg * kNW; }
int score_deal_warps(int nkv, int G) { return nkv <= kNW / 2 && G >= 5 ? kNW / nkv : 1; }

cudaError_t launch_score(const ScoreArgs& a, int dtype, int G, bool raw, bool f8, bool deal, int grid,
                         cudaStream_t st) {
  if (dtype == 0)
    return f8 ? launch_score_m<0, true>(a, G, raw, deal, grid, st) : launch_score_m<0, false>(a, G, raw, deal, grid, st);
  return f8 ? launch_score_m<1, true>(a, G, raw, deal, grid, st) : launch_score_m<1, false>(a, G, raw, deal, grid, st);
}

cudaError_t launch_attn_finalize(const FinalizeArgs& a0, int sms, cudaStream_t st, int* kernels,
                                 bool two_kernel) {
  FinalizeArgs a = a0;
  a.tpt = 1;
  // The split step's normalisation runs beside the next layer's scoring
  // kernel, which leaves room for about one such CTA per SM: each thread
  // takes several tokens so that the grid needs at most about two rounds of
  // CTAs instead of trickling through in many.
  if (two_kernel)
    while (a.tpt < kFinMaxTpt &&
           (long long)a.B * ((a.cap + kFinChunk * a.tpt - 1) / (kFinChunk * a.tpt)) > 2LL * sms)
      a.tpt <<= 1;
  dim3 grid((a.cap + kFinChunk * a.tpt - 1) / (kFinChunk * a.tpt), a.B);
  const size_t smem = 2 * a.H * sizeof(float) + (a.hist0 ? kHistBins * sizeof(uint32_t) : 0);
  // more than two normalisation CTAs per SM: combine the partials once per
  // (b, h) in a kernel of their own instead of once per CTA
  if (a.stats && (two_kernel || (long long)grid.x * grid.y > 2LL * sms)) {
    *kernels = 2;
    const int pairs = a.B * a.H;
    cudaError_t e = launch_pdl(hill_attn_stats_kernel, dim3((pairs + kStatsWarps - 1) / kStatsWarps),
                               dim3(kStatsWarps * 32), 0, st, 0, a);
    if (e != cudaSuccess) return e;
    return a.kvh ? launch_pdl(hill_attn_finalize_kernel<true, true>, grid, dim3(kFinThreads), smem, st, 0, a)
                 : launch_pdl(hill_attn_finalize_kernel<true, false>, grid, dim3(kFinThreads), smem, st, 0, a);
  }
  *kernels = 1;
  return a.kvh ? launch_pdl(hill_attn_finalize_kernel<false, true>, grid, dim3(kFinThreads), smem, st, 0, a)
               : launch_pdl(hill_attn_finalize_kernel<false, false>, grid, dim3(kFinThreads), smem, st, 0, a);
}

}  // namespace hill
