// score_tc.cu -- the K-cache stream of Eq. 1 on the E4M3 key shadow of
// Sec. 4.4 through the tensor cores' native 8-bit path (tcgen05.mma,
// kind::f8f6f4, accumulators in tensor memory).
//
// On this GPU an E4M3 mma.sync runs as 16-bit tensor operations plus operand
// conversions, which leaves the warp-level scoring kernel of score.cu bound
// by instruction latency on the 8-bit stream.  Here single threads issue the
// products and the epilogue reads them back one token per thread.  A CTA runs
// two independent pipelines, each with its own rings, barriers and half of
// the tensor memory, taking alternate chunks of its work range:
//
//   producer    (warps 0, 1) per unit -- a chunk of up to 128 tokens of one
//               sequence and two of its KV heads -- one box of up to 128 rows x
//               128 codes per KV head (128-byte swizzle), the 16 x 128-code
//               box of that KV head's query codes, and the rows' scales, all
//               completing on the stage's barrier (the scales in a ring of
//               their own, released by the epilogue);
//   products    (warps 2, 3) one thread issues, per KV head of the unit, the
//               [128 tokens x 128] . [128 x 16 heads] product as 4 tcgen05.mma
//               of K = 32 into a 16-column accumulator, then commits the stage
//               back to the producer and the unit's accumulators to the
//               epilogue;
//   epilogue    (warps 4-7, 8-11) each warp reads its 32 tensor-memory lanes
//               (tokens) of two units at a time with tcgen05.ld, applies the
//               query and row scales, and either sums the heads per token across
//               the chunk's KV heads (RAW) or writes the base-2 logits and folds
//               each into this token's running (max, sum 2^(z2 - max)) of the
//               head in shared memory (ATTN); when the CTA leaves a sequence all
//               epilogue warps meet and reduce those into one partial per
//               (sequence, head, CTA).
//
// A CTA takes the same contiguous range of 32-token tiles as the warp-level
// kernel of score.cu ([x * per, (x + 1) * per) over all sequences), so the
// normalisation finds the partial slots where it expects them whichever
// kernel ran; it walks the range in chunks of up to four tiles of one
// sequence (one box of 32, 64, 96 or 128 rows).  Every wait is bounded;
// after a timeout each role leaves its loop, in-flight copies and products
// get one more bounded wait, and the tensor memory is released.
#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kTcT = 128;                     // token rows of a product (M)
constexpr int kTcSub = 32;                    // tokens per tile of the work ranges (as the warp-level kernel)
constexpr int kTcChunk = kTcT / kTcSub;       // tiles per product at most
constexpr int kTcN = 16;                      // query-head rows of B (zero past the group)
constexpr int kTcPipes = 2;                   // independent pipelines per CTA (alternate chunks)
constexpr int kTcU = 2;                       // KV heads per unit (one barrier round for their products)
constexpr int kTcStages = 2;                  // per pipeline: ring of codes and query codes
constexpr int kTcScSlots = 4;                 // per pipeline: ring of row scales (released by the epilogue)
constexpr int kTcBatch = 2;                   // units an epilogue takes per trip
constexpr int kTcAcc = 2 * kTcBatch;          // per pipeline: unit accumulators in tensor memory
constexpr int kTcPipeCols = kTcAcc * kTcU * 16;   // tensor-memory columns of one pipeline
constexpr int kTcCols = kTcPipes * kTcPipeCols;   // allocated (a power of two)
constexpr int kTcKBytes = kTcT * 128;         // 16 KB of codes per unit
constexpr int kTcQBytes = kTcN * 128;         // 2 KB of query codes per unit
constexpr int kTcScBytes = kTcU * kTcT * 4;   // the unit's row scales
constexpr int kTcStageBytes = kTcU * (kTcKBytes + kTcQBytes);   // codes x U | query codes x U, a multiple of 1024
constexpr int kTcEpiWarps = 4;                // per pipeline
// warps 0-1 producers, 2-3 product issuers, 4-7 and 8-11 the epilogues of pipelines 0 and 1
constexpr int kTcWarps = 2 * kTcPipes + kTcPipes * kTcEpiWarps;
constexpr int kTcThreads = kTcWarps * 32;
constexpr int kTcMaxBatch = 512;
constexpr int kTcMaxHeads = 32;               // per-thread softmax statistics in shared memory: [pipe][H][128]
constexpr int kTcTableInts = kTcMaxBatch + 4;

// shared-memory layout (offsets from a 1024-byte aligned base); pipeline p's
// rings and barriers at p times their per-pipeline size
constexpr int kOffScale = kTcPipes * kTcStages * kTcStageBytes;
constexpr int kOffBars = kOffScale + kTcPipes * kTcScSlots * kTcScBytes;
// per pipeline: full[S], empty[S], accf[A], acce[A], sce[SC], done
constexpr int kBFull = 0, kBEmpty = kBFull + kTcStages, kBAccF = kBEmpty + kTcStages, kBAccE = kBAccF + kTcAcc,
              kBScE = kBAccE + kTcAcc, kBDone = kBScE + kTcScSlots, kBPerPipe = kBDone + 1;
constexpr int kOffBarEpi = kOffBars + kTcPipes * kBPerPipe * 8;   // two meeting points of all epilogue warps
constexpr int kOffTmem = kOffBarEpi + 16;
constexpr int kOffAbort = kOffTmem + 8;
constexpr int kOffTab = (kOffAbort + 4 + 15) & ~15;        // tile prefix [B + 1], lengths [B]
constexpr int kOffStats = kOffTab + 2 * kTcTableInts * 4;  // ATTN: [pipe][H][128 tokens of a unit] (max, sum)
static_assert(kOffTab % 16 == 0 && kOffStats % 16 == 0, "alignment");

// instruction descriptor of the kind::f8f6f4 product: fp32 accumulation
// (bits 4-5 = 1), A and B E4M3 (format 0), both K-major, N / 8 at bit 17,
// M / 16 at bit 24
constexpr uint32_t kTcIdesc = (1u << 4) | ((uint32_t)(kTcN >> 3) << 17) | ((uint32_t)(kTcT >> 4) << 24);

// Shared-memory matrix descriptor of a K-major operand whose rows are 128
// bytes with the 128-byte swizzle (as the tiled TMA writes them): start
// address / 16, leading offset 16 B (unused for this layout), stride 1024 B
// between groups of 8 rows, descriptor version 1, swizzle mode 2 (128 B).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
  return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

__device__ __forceinline__ void tmem_alloc(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D (tensor memory) = A . B^T (+ D when acc != 0), both operands from shared memory
__device__ __forceinline__ void tc_mma_f8(uint32_t d, uint64_t a, uint64_t b, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(kTcIdesc), "r"(acc)
      : "memory");
}
// arrive once on `bar` when every product this thread issued so far has completed
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
// 16 consecutive columns of this warp's 32 lanes: thread i gets lane i's
// values once tc_wait_ld() has returned
__device__ __forceinline__ void tc_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tc_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(tmap), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}

// Query rows to E4M3: one warp per row (b, g, r), 4 elements per lane; the
// float32 steps are those of the warp-level kernel (amax over the row,
// 448 / amax, round-to-nearest products, saturating conversion).
template <int DT>
__global__ void __launch_bounds__(256) hill_quantize_q_kernel(const QuantQArgs a) {
  pdl_wait();   // the previous call may still read the codes this writes
  const int lane = threadIdx.x & 31;
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int64_t rows = (int64_t)a.B * a.Hkv * kTcN;
  if (row >= rows) return;
  const int r = (int)(row % kTcN);
  const int64_t bg = row / kTcN;
  const int g = (int)(bg % a.Hkv), b = (int)(bg / a.Hkv);
  uint32_t codes = 0u;
  if (r < a.G) {
    const int h = g * a.G + r;
    const auto* qh = static_cast<const uint16_t*>(a.q) + (int64_t)b * a.q_sb + (int64_t)h * a.q_sh;
    const uint2 raw = __ldg(reinterpret_cast<const uint2*>(qh + 4 * lane));
    float v[8];
    to_float8<DT>(uint4{raw.x, raw.y, 0u, 0u}, v);
    float amax = fmaxf(fmaxf(fabsf(v[0]), fabsf(v[1])), fmaxf(fabsf(v[2]), fabsf(v[3])));
    amax = warp_max(amax);
    const float rq = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
    codes = e4m3x2(__fmul_rn(v[0], rq), __fmul_rn(v[1], rq)) | (e4m3x2(__fmul_rn(v[2], rq), __fmul_rn(v[3], rq)) << 16);
    if (lane == 0) a.sq[(int64_t)b * a.H + h] = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
  }
  reinterpret_cast<uint32_t*>(a.q8 + row * 128)[lane] = codes;
}

template <bool RAW>
__global__ void __launch_bounds__(kTcThreads, 1) hill_score_tc_kernel(const __grid_constant__ ScoreTcArgs a) {
  extern __shared__ unsigned char tsm_raw[];
  const uint32_t raw_addr = smem_addr(tsm_raw);
  const uint32_t base_addr = (raw_addr + 1023u) & ~1023u;
  unsigned char* base = tsm_raw + (base_addr - raw_addr);
  int* tstart = reinterpret_cast<int*>(base + kOffTab);
  int* slen = tstart + kTcTableInts;
  float2* stats_all = reinterpret_cast<float2*>(base + kOffStats);
  volatile int* abort_flag = reinterpret_cast<int*>(base + kOffAbort);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int B = a.B, H = a.H;
  // barrier i of pipeline p
  auto bar = [&](int p, int i) { return base_addr + kOffBars + (uint32_t)((p * kBPerPipe + i) * 8); };

  if (threadIdx.x == 0) {
    for (int p = 0; p < kTcPipes; ++p) {
      for (int s = 0; s < kTcStages; ++s) {
        mbar_init(bar(p, kBFull + s), 1);
        mbar_init(bar(p, kBEmpty + s), 1);
      }
      for (int i = 0; i < kTcAcc; ++i) {
        mbar_init(bar(p, kBAccF + i), 1);
        mbar_init(bar(p, kBAccE + i), kTcEpiWarps);
      }
      for (int i = 0; i < kTcScSlots; ++i) mbar_init(bar(p, kBScE + i), kTcEpiWarps);
      mbar_init(bar(p, kBDone), 1);
    }
    mbar_init(base_addr + kOffBarEpi, kTcPipes * kTcEpiWarps);
    mbar_init(base_addr + kOffBarEpi + 8, kTcPipes * kTcEpiWarps);
    *abort_flag = 0;
    fence_barrier_init();
  }
  // the table of 32-token tiles (lengths are inputs of the call)
  for (int b = threadIdx.x; b < B; b += kTcThreads) {
    int len = a.lens[b];
    if (len < 0 || len > a.cap) {
      raise_error(a.err, kErrDevArg);
      len = len < 0 ? 0 : a.cap;
    }
    slen[b] = len;
  }
  if (!RAW)
    for (int i = threadIdx.x; i < kTcPipes * H * kTcT; i += kTcThreads) stats_all[i] = make_float2(-INFINITY, 0.f);
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    tstart[0] = 0;
    for (int b = 0; b < B; ++b) {
      acc += (slen[b] + kTcSub - 1) / kTcSub;
      tstart[b + 1] = acc;
    }
  }
  __syncthreads();
  // the CTA's range of 32-token tiles, by the rule of the warp-level kernel
  // (so that the normalisation finds the same partial slots)
  const int n_items = tstart[B];
  const int per = (n_items + gridDim.x - 1) / gridDim.x;
  const int it_lo = min(n_items, (int)blockIdx.x * per), it_hi = min(n_items, it_lo + per);
  pdl_wait();
  if (!RAW && a.hist0) {   // this CTA's share of the leading-digit histogram, zeroed for the normalisation
    const int64_t hper = (a.hist0_words + gridDim.x - 1) / gridDim.x;
    const int64_t w0 = min((int64_t)blockIdx.x * hper, a.hist0_words);
    const int64_t w1 = min(w0 + hper, a.hist0_words);
    for (int64_t w = w0 + threadIdx.x; w < w1; w += kTcThreads) a.hist0[w] = 0u;
  }
  if (it_lo >= it_hi) return;

  if (warp == 0) {
    tmem_alloc(base_addr + kOffTmem, kTcCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(base + kOffTmem);
  const int nkv = a.nkv;
  // The range is walked in chunks of up to kTcChunk consecutive tiles of one
  // sequence (a chunk ends at the range's or the sequence's end); chunk k of
  // the walk belongs to pipeline k % kTcPipes, and a unit is (chunk, KV
  // head), KV heads innermost.  Every role walks every chunk.
  int b_first = 0;
  while (b_first < B - 1 && tstart[b_first + 1] <= it_lo) ++b_first;
  auto chunk_at = [&](int item, int b) { return min(kTcChunk, min(it_hi, tstart[b + 1]) - item); };
  auto next_chunk = [&](int& item, int& b, int c) {
    item += c;
    while (b < B - 1 && tstart[b + 1] <= item) ++b;
  };

  if (warp < kTcPipes) {
    // ---- producer of pipeline p
    const int p = warp;
    if (lane == 0) {
      for (int m = 0; m < kTcChunk; ++m) prefetch_tmap(&a.kmap[m]);
      prefetch_tmap(&a.qmap);
      const uint64_t pol = l2_evict_first_policy();
      int n = 0, k = 0;
      for (int item = it_lo, b = b_first; item < it_hi && !*abort_flag; ++k) {
        const int c = chunk_at(item, b);
        if (k % kTcPipes == p) {
          const int j0 = (item - tstart[b]) * kTcSub;
          for (int gi = 0; gi < nkv; gi += kTcU, ++n) {
            const int uh = min(kTcU, nkv - gi);   // KV heads of this unit
            const int s = n % kTcStages, sc = n % kTcScSlots;
            const uint32_t ph = (uint32_t)(n / kTcStages) & 1u, sph = (uint32_t)(n / kTcScSlots) & 1u;
            if (*abort_flag || !mbar_wait(bar(p, kBEmpty + s), ph ^ 1u, a.err) ||
                !mbar_wait(bar(p, kBScE + sc), sph ^ 1u, a.err)) {
              *abort_flag = 1;
              break;
            }
            const uint32_t full = bar(p, kBFull + s);
            const uint32_t dst = base_addr + (uint32_t)((p * kTcStages + s) * kTcStageBytes);
            const uint32_t scd = base_addr + kOffScale + (uint32_t)((p * kTcScSlots + sc) * kTcScBytes);
            // the codes, the query codes and the row scales complete on the
            // stage's barrier; the scales land in their own ring
            mbar_arrive_expect_tx(full, (uint32_t)(uh * (c * kTcSub * (128 + 4) + kTcQBytes)));
            for (int u = 0; u < uh; ++u) {
              const int g = a.goff + gi + u;
              tma_load_4d(dst + u * kTcKBytes, &a.kmap[c - 1], 0, j0, g, b, full, pol);
              tma_load_2d(dst + kTcU * kTcKBytes + u * kTcQBytes, &a.qmap, 0, (b * a.Hkv + g) * kTcN, full);
              bulk_g2s(scd + u * kTcT * 4, a.kscale + ((int64_t)b * a.Hkv + g) * a.cap32 + j0,
                       (uint32_t)(c * kTcSub * 4), full, pol);
            }
          }
        }
        next_chunk(item, b, c);
      }
      if (*abort_flag) {   // the copies of the last stages get one more bounded wait
        for (int u = max(0, n - kTcStages); u < n; ++u)
          mbar_wait(bar(p, kBFull + u % kTcStages), (uint32_t)(u / kTcStages) & 1u, a.err);
      }
    }
  } else if (warp < 2 * kTcPipes) {
    // ---- products of pipeline p
    const int p = warp - kTcPipes;
    if (lane == 0) {
      const uint32_t tmem_p = tmem + (uint32_t)(p * kTcPipeCols);
      int n = 0, k = 0;
      for (int item = it_lo, b = b_first; item < it_hi && !*abort_flag; ++k) {
        const int c = chunk_at(item, b);
        if (k % kTcPipes == p) {
          for (int gi = 0; gi < nkv; gi += kTcU, ++n) {
            const int uh = min(kTcU, nkv - gi);
            const int s = n % kTcStages, ac = n % kTcAcc;
            const uint32_t ph = (uint32_t)(n / kTcStages) & 1u, aph = (uint32_t)(n / kTcAcc) & 1u;
            if (*abort_flag || !mbar_wait(bar(p, kBFull + s), ph, a.err) ||
                !mbar_wait(bar(p, kBAccE + ac), aph ^ 1u, a.err)) {
              *abort_flag = 1;
              break;
            }
            tc_fence_after();
            // rows of the stage past the chunk hold stale codes; their products
            // land in accumulator rows the epilogue does not read
            const uint32_t st0 = base_addr + (uint32_t)((p * kTcStages + s) * kTcStageBytes);
            for (int u = 0; u < uh; ++u) {
              const uint32_t ka = st0 + u * kTcKBytes, qa = st0 + kTcU * kTcKBytes + u * kTcQBytes;
#pragma unroll
              for (int kb = 0; kb < 4; ++kb)
                tc_mma_f8(tmem_p + (uint32_t)((ac * kTcU + u) * kTcN), smem_desc_sw128(ka + kb * 32),
                          smem_desc_sw128(qa + kb * 32), kb > 0 ? 1u : 0u);
            }
            tc_commit(bar(p, kBEmpty + s));
            tc_commit(bar(p, kBAccF + ac));
          }
        }
        next_chunk(item, b, c);
      }
      // every product issued has completed before the tensor memory is released
      tc_commit(bar(p, kBDone));
      mbar_wait(bar(p, kBDone), 0u, a.err);
    }
  } else {
    // ---- epilogue of pipeline p: warp quarter qw owns tensor-memory lanes
    // (tokens) 32*qw .. of the pipeline's accumulators
    const int p = (warp - 2 * kTcPipes) / kTcEpiWarps;
    const int ew = warp - 2 * kTcPipes;   // 0 .. 7 over both pipelines
    const int qw = warp & 3;
    const int t = qw * 32 + lane;
    const uint64_t pol_keep = l2_evict_last_policy();
    const uint32_t taddr_w = tmem + (uint32_t)(p * kTcPipeCols) + ((uint32_t)(qw * 32) << 16);
    float2* stats = stats_all + (size_t)p * H * kTcT;
    int cur_b = -1;
    // all epilogue warps meet at one of two mbarriers (a bounded wait, so that
    // a warp that left after a timeout cannot hold the others forever)
    uint32_t epi_ph = 0;
    auto epi_meet = [&](uint32_t mb) -> bool {
      __syncwarp();
      if (lane == 0) mbar_arrive(mb);
      return __all_sync(0xffffffffu, mbar_wait(mb, epi_ph, a.err));
    };
    // ATTN: fold this sequence's statistics (both pipelines') into its
    // partials (one warp per head, 4 entries per lane and pipeline, then the
    // lanes) and reset them
    auto flush = [&](int bb) -> bool {
      if (!epi_meet(base_addr + kOffBarEpi)) return false;
      const int slot = (int)blockIdx.x - tstart[bb] / per;
      for (int h = ew; h < H; h += kTcPipes * kTcEpiWarps) {
        float m = -INFINITY, l = 0.f;
#pragma unroll
        for (int q = 0; q < kTcPipes; ++q)
#pragma unroll
          for (int u = 0; u < kTcT / 32; ++u) {
            float2* e = stats_all + ((size_t)q * H + h) * kTcT + u * 32 + lane;
            const float2 pv = *e;
            if (pv.y > 0.f) {
              const float mn = fmaxf(m, pv.x);
              l = l * ex2(m - mn) + pv.y * ex2(pv.x - mn);
              m = mn;
            }
            *e = make_float2(-INFINITY, 0.f);
          }
        const float mw = warp_max(m);
        const float lw = warp_sum(l > 0.f ? l * ex2(m - mw) : 0.f);
        if (lane == 0) a.partials[((int64_t)bb * a.nslot + slot) * H + h] = make_float2(mw, lw);
      }
      const bool ok = epi_meet(base_addr + kOffBarEpi + 8);
      epi_ph ^= 1u;
      return ok;
    };
    int n = 0, k = 0;
    for (int item = it_lo, b = b_first; item < it_hi && !*abort_flag; ++k) {
      const int c = chunk_at(item, b);
      if (!RAW && b != cur_b) {   // both pipelines see every change of sequence
        if (cur_b >= 0 && !flush(cur_b)) {
          *abort_flag = 1;
          break;
        }
        cur_b = b;
      }
      if (k % kTcPipes != p) {
        next_chunk(item, b, c);
        continue;
      }
      const int j = (item - tstart[b]) * kTcSub + t;
      const bool valid = t < c * kTcSub && j < slen[b];
      float rs = 0.f;   // RAW: this token's sum over the chunk's KV heads
      // kTcBatch units (kTcU KV heads each) of the chunk per trip: their
      // waits, tensor-memory loads and epilogues overlap
      const int nunits = (nkv + kTcU - 1) / kTcU;
      for (int ui = 0; ui < nunits; ui += kTcBatch) {
        const int nb = min(kTcBatch, nunits - ui);
        bool ok = !*abort_flag;
#pragma unroll
        for (int w = 0; w < kTcBatch; ++w)
          if (w < nb && ok) ok = mbar_wait(bar(p, kBAccF + (n + w) % kTcAcc), (uint32_t)((n + w) / kTcAcc) & 1u, a.err);
        if (!__all_sync(0xffffffffu, ok)) {
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        // head slot x = w * kTcU + u: unit n + w, its u-th KV head
        constexpr int kX = kTcBatch * kTcU;
        uint32_t v[kX][16];
        float ksc[kX];
#pragma unroll
        for (int x = 0; x < kX; ++x) {
          const int w = x / kTcU, u = x % kTcU;
          const bool has = w < nb && (ui + w) * kTcU + u < nkv;
          if (has) tc_ld16(taddr_w + (uint32_t)((((n + w) % kTcAcc) * kTcU + u) * kTcN), v[x]);
          ksc[x] = has && valid ? __uint_as_float(lds32(base_addr + kOffScale +
                                                        (uint32_t)((p * kTcScSlots + (n + w) % kTcScSlots) * kTcScBytes) +
                                                        (u * kTcT + t) * 4))
                                : 0.f;
        }
        tc_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
#pragma unroll
          for (int w = 0; w < kTcBatch; ++w)
            if (w < nb) {
              mbar_arrive(bar(p, kBAccE + (n + w) % kTcAcc));
              mbar_arrive(bar(p, kBScE + (n + w) % kTcScSlots));
            }
        }
#pragma unroll
        for (int x = 0; x < kX; ++x) {
          const int w = x / kTcU, u = x % kTcU;
          const int gi = (ui + w) * kTcU + u;
          if (w >= nb || gi >= nkv) continue;
          const int g = a.goff + gi;
          const float* sqb = a.sq + (int64_t)b * H + g * a.G;
          if constexpr (RAW) {
            float sum = 0.f;
#pragma unroll
            for (int hl = 0; hl < kTcN; ++hl)
              if (hl < a.G) sum += __uint_as_float(v[x][hl]) * __ldg(sqb + hl);
            rs += sum * ksc[x];
          } else if (valid) {
            float* lg = a.logits + ((int64_t)b * H + g * a.G) * a.lstride + j;
#pragma unroll
            for (int hl = 0; hl < kTcN; ++hl) {
              if (hl >= a.G) break;
              const float z = __uint_as_float(v[x][hl]) * (__ldg(sqb + hl) * ksc[x]) * kLog2eInvSqrtD;
              st_global_hint(lg + (int64_t)hl * a.lstride, z, pol_keep);
              // this token's running (max, sum 2^(z2 - max)) of the head
              float2* st = stats + (g * a.G + hl) * kTcT + t;
              const float2 pv = *st;
              const float mn = fmaxf(pv.x, z);
              *st = make_float2(mn, pv.y * ex2(pv.x - mn) + ex2(z - mn));
            }
          }
        }
        n += nb;
      }
      if (RAW && valid && !*abort_flag) {
        const float val = rs * kInvSqrtD;
        const int64_t o = (int64_t)b * a.cap + j;
        if (a.scores) a.scores[o] = val;
        if (a.accum) a.accum[o] += val;
      }
      next_chunk(item, b, c);
    }
    if (!RAW && cur_b >= 0 && !*abort_flag && !flush(cur_b)) *abort_flag = 1;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTcCols);
  }
}

size_t tc_smem_bytes(int H) { return (size_t)kOffStats + (size_t)kTcPipes * H * kTcT * sizeof(float2) + 1024; }

}  // namespace

int score_tc_max_group() { return kTcN; }
int score_tc_max_heads() { return kTcMaxHeads; }

cudaError_t launch_quantize_q(const QuantQArgs& a, int dtype, cudaStream_t st) {
  const int64_t rows = (int64_t)a.B * a.Hkv * kTcN;
  const int grid = (int)((rows + 7) / 8);
  if (grid == 0) return cudaSuccess;
  return dtype == 0 ? launch_pdl(hill_quantize_q_kernel<0>, dim3(grid), dim3(256), 0, st, 0, a)
                    : launch_pdl(hill_quantize_q_kernel<1>, dim3(grid), dim3(256), 0, st, 0, a);
}

cudaError_t launch_score_tc(const ScoreTcArgs& a, bool raw, int grid, cudaStream_t st) {
  static int cache[2][64] = {{0}};
  if (a.B > kTcMaxBatch || a.G > kTcN || a.G < 1 || a.H > kTcMaxHeads) return cudaErrorInvalidValue;
  const size_t smem = tc_smem_bytes(a.H);
  auto kern = raw ? hill_score_tc_kernel<true> : hill_score_tc_kernel<false>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), (int)smem, cache[raw ? 1 : 0]);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(kTcThreads), smem, st, 0, a);
}

}  // namespace hill
