// attn.cu -- decode attention over the selected tokens only (Sec. 4.1, workflow step 6:
// only the critical KV reaches the attention; Eq. 1 restricted to the set).
//
// Gather + split-K flash decode on persistent CTAs.  The work is a list of
// batches: (sequence b, KV head g, batch bi of 32 consecutive entries of
// b's index list), ordered b, g, bi.  Every warp of the grid owns one
// contiguous segment of that list and streams it through a K region and a V
// region of shared memory.  A batch's 32 K rows and 32 V rows (tokens
// idx[b][32*bi + i]) are gathered with 16-byte asynchronous copies (a
// half-warp per 256-byte row; the K rows and the V rows are separate copy
// groups, so K of the next batch is in flight while this batch's softmax and
// P.V run, and V of the next batch while the next S runs) into an
// XOR-swizzled layout that ldmatrix reads without bank conflicts; rows of
// absent tokens are zero-filled by the copies themselves.  The index entries
// of the batch after next are loaded with the K copies and are checked only
// when that batch is issued.  (TMA
// alternatives were measured slower on the same layout: 256-byte bulk copies
// per row are bound by the copy engine's request rate, and tile::gather4 loads
// reached about 85 % of the cp.async throughput; neither depends on how
// scattered the rows are.)
// Both products run on mma.sync m16n8k16 with fp32 accumulation.  S = q . K^T
// takes the G query heads of the group as the rows of A (held in registers
// for all batches of a (b, g)) and K rows read with ldmatrix as B.  An online
// softmax per head, in base 2 (logits scaled by log2(e)/sqrt(d)), runs across
// the batches of one (b, g).  The output is accumulated transposed, O^T +=
// V^T . P^T: V rows read with transposed ldmatrix form A (16 dims x 16
// tokens), and the weights P -- already laid out as a B fragment by the S
// accumulators -- enter as a 16-bit high part plus its 16-bit residual, so
// every instruction covers 8 heads x 16 dims.  A group of 9 to 16 heads fills
// all 16 rows of A (two row blocks of 8 heads, each with its own softmax state
// and O^T accumulators), so the rows gathered once serve 16 heads; larger
// groups run in passes of 16.  When a warp's segment holds
// all batches of a (b, g) it writes the output; otherwise it writes a partial
// (max, sum, o) that hill_attn_combine_kernel merges.
#include <type_traits>

#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kAW = 8;                               // warps per CTA
constexpr int kAThreads = kAW * 32;
constexpr int kBatch = 32;                           // selected entries per batch
constexpr int kMaxBatchAttn = 512;                   // sequences in the per-CTA table

constexpr int kHalfBytes = kBatch * 128;             // 32 rows x 64 dims, swizzled

struct AttnCfg {
  // K dims 0-63 | K dims 64-127 | V dims 0-63 | V dims 64-127
  static constexpr int kSlotBytes = 4 * kHalfBytes;
  static constexpr int kSmem = kAW * kSlotBytes + 128;   // + alignment slack
};

// Position of a batch in the list: table unit u (a sequence b, or with
// per-KV-head selection a pair (b, g)), sequence, KV head, batch within (b, g).
struct Pos {
  int u, b, g, bi;
};

// Selected-token count of table unit u (count[] has one entry per unit).
__device__ __forceinline__ int clamp_count(const AttnArgs& a, int u) {
  const int n = a.count[u];
  return n < 0 ? 0 : (n > a.max_k ? a.max_k : n);
}

// Segment of the batch list owned by global warp w (balanced split).
__device__ __forceinline__ void warp_segment(int total, int nwarps, int w, int& t0, int& t1) {
  const int per = (total + nwarps - 1) / nwarps;
  t0 = min(total, w * per);
  t1 = min(total, t0 + per);
}

template <int DT, int G>
__global__ void __launch_bounds__(kAThreads, 1) hill_sparse_attn_kernel(const __grid_constant__ AttnArgs a) {
  extern __shared__ unsigned char asmem[];
  __shared__ int s_bstart[kMaxBatchAttn + 1];
  __shared__ int s_nbat[kMaxBatchAttn];
  __shared__ int s_cnt[kMaxBatchAttn];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait();
  // No early trigger (here and in the combine): the attention runs beside
  // the K stream of later layers, and a dependent launched early would hold
  // SMs idle while it waits (measured: the pipelined step is 2 % faster).

  // table units: sequences (every KV head reads the same set, Hkv * nbat
  // batches per unit, ordered g, bi), or with per-KV-head selection the pairs
  // (b, g) (nbat batches per unit)
  const int R = a.kvh ? a.B * a.Hkv : a.B;
  const int upb = a.kvh ? 1 : a.Hkv;   // KV heads per unit
  for (int u = threadIdx.x; u < R; u += kAThreads) {
    const int n = clamp_count(a, u);
    s_cnt[u] = n;
    s_nbat[u] = (n + kBatch - 1) / kBatch;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int u = 0; u < R; ++u) {
      s_bstart[u] = acc;
      acc += upb * s_nbat[u];
    }
    s_bstart[R] = acc;
  }
  __syncthreads();
  const int total = s_bstart[R];
  const int nwarps = gridDim.x * kAW;
  const int gw = blockIdx.x * kAW + warp;
  int t0, t1;
  warp_segment(total, nwarps, gw, t0, t1);
  if (t0 >= t1) return;

  // 128-byte aligned slots: every swizzled row is one bank-aligned line
  const uint32_t slot0 = ((smem_addr(asmem) + 127u) & ~127u) + warp * AttnCfg::kSlotBytes;
  const uint32_t sk = slot0, sv = slot0 + 2 * kHalfBytes;   // the warp's K rows | V rows
  const auto* kbase = static_cast<const uint16_t*>(a.k);
  const auto* vbase = static_cast<const uint16_t*>(a.v);
  const int ksn = (int)a.k_sn, vsn = (int)a.v_sn;   // the host checks both fit in 32 bits

  // position of batch t0 (binary search once), then advanced one batch at a time
  Pos first;
  {
    int lo = 0, hi = R;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (s_bstart[mid] <= t0) lo = mid; else hi = mid;
    }
    const int rem = t0 - s_bstart[lo];
    first.u = lo;
    if (a.kvh) {
      first.b = lo / a.Hkv;
      first.g = lo - first.b * a.Hkv;
      first.bi = rem;
    } else {
      first.b = lo;
      first.g = rem / s_nbat[lo];
      first.bi = rem - first.g * s_nbat[lo];
    }
  }
  auto advance = [&](Pos& p) {
    if (p.u >= R) return;
    if (++p.bi < s_nbat[p.u]) return;
    p.bi = 0;
    if (!a.kvh && ++p.g < a.Hkv) return;
    do {
      ++p.u;
    } while (p.u < R && s_nbat[p.u] == 0);
    p.b = a.kvh ? p.u / a.Hkv : p.u;
    p.g = a.kvh ? p.u - p.b * a.Hkv : 0;
  };

  // raw index entry of this lane for the batch at p (-1 past the count).
  // Nothing here depends on the loaded value, so the load stays in flight
  // until the batch is issued one iteration later, where it is checked.
  auto load_idx = [&](const Pos& p) -> int {
    const int e = p.bi * kBatch + lane;
    return e < s_cnt[p.u] ? a.idx[(int64_t)p.u * a.max_k + e] : -1;
  };
  // An entry of the batch at p that lies outside [0, cap) is reported and
  // skipped (-1: no token).
  auto check = [&](const Pos& p, int jj) -> int {
    if (p.bi * kBatch + lane < s_cnt[p.u] && (jj < 0 || jj >= a.cap)) {
      raise_error(a.err, kErrDevArg);
      jj = -1;
    }
    return jj;
  };
  // Gather the 32 rows of one cache (K or V) for the batch at p into the
  // 8 KB region dst: row r of the batch is token jj of lane r (-1: none,
  // zero-filled).  A half-warp copies one 256-byte row; chunk c (16 bytes)
  // of row r goes to 128-byte line r of half c / 8 at position
  // (c % 8) ^ (r % 8), so the ldmatrix reads below are conflict-free.  One
  // cp.async group per call.
  const int l16 = lane & 15, hrow = lane >> 4;
  const uint32_t dst_lane = (uint32_t)((l16 >> 3) * kHalfBytes + hrow * 128);
  const uint32_t swz_lane = (uint32_t)(((l16 & 7) ^ hrow) << 4);
  auto issue_rows = [&](const Pos& p, uint32_t dst, const uint16_t* base, int64_t sb, int64_t sh, int sn, int jj) {
    const uint16_t* rp = base + (int64_t)p.b * sb + (int64_t)p.g * sh + l16 * 8;
    dst += dst_lane;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int j = __shfl_sync(0xffffffffu, jj, 2 * i + hrow);
      const uint32_t nbytes = j >= 0 ? 16u : 0u;
      const int jc = j >= 0 ? j : 0;
      // row 2i + hrow: (2i + hrow) % 8 = (2i % 8) | hrow
      const uint32_t off = (uint32_t)(i * 256) + (swz_lane ^ (uint32_t)(((2 * i) & 7) << 4));
      cp_async16_zfill(dst + off, rp + (int64_t)jc * sn, nbytes);
    }
    cp_async_commit();
  };

  // Pipeline of one warp over its batches t0 .. t1-1, with one K region and
  // one V region: K rows of batch t + 1 are fetched once S(t) has read the K
  // region (while the softmax and O += P V of batch t run), V rows of batch
  // t + 1 once O += P V(t) has read the V region (while S(t + 1) runs).  The
  // cp.async groups complete in the order K(t), V(t), K(t + 1), V(t + 1), ...
  // The index entries of batch t + 2 are loaded when K(t + 1) is issued.
  Pos pc = first, pi = first, pl = first;
  int jcur = check(pi, load_idx(pl));           // entries of the batch being issued
  advance(pl);
  unsigned vm_cur = __ballot_sync(0xffffffffu, jcur >= 0), vm_next = 0u;
  issue_rows(pi, sk, kbase, a.k_sb, a.k_sh, ksn, jcur);
  issue_rows(pi, sv, vbase, a.v_sb, a.v_sh, vsn, jcur);
  advance(pi);
  int jnext = t0 + 1 < t1 ? load_idx(pl) : -1;
  advance(pl);

  // mma.sync fragments: grp = lane/4, tig = lane%4.  S accumulators: row grp
  // (+8 with 16 heads: row block rb = 1) = query head grp (+8) of the group
  // (rows >= Gn are zero, and rows 8..15 when G <= 8; Gn = G unless the
  // group has fewer heads than the power-of-two template), columns = tokens
  // nb*8 + 2*tig + {0,1}.  O^T accumulators, one set per row block: rows =
  // dims db*16 + grp (+8), columns = heads 8*rb + 2*tig, 8*rb + 2*tig + 1.
  constexpr int kRB = G > 8 ? 2 : 1;          // row blocks of 8 heads
  const int grp = lane >> 2, tig = lane & 3;
  const int Gn = G <= 2 ? G : a.Gn;
  bool head_ok[kRB];
#pragma unroll
  for (int rb = 0; rb < kRB; ++rb) head_ok[rb] = grp + 8 * rb < Gn;
  const int hA = 2 * tig, hB = 2 * tig + 1;   // heads of this lane's O^T columns (in a row block)
  float m_run[kRB], l_run[kRB];               // softmax state of head grp + 8*rb (base 2)
  float oacc[kRB][8][4];
  uint32_t qa[kRB][8][2];                     // q rows of the group as A fragments
  int cb = -1, cg = -1, cu = -1;              // the (b, g) being accumulated and its unit
  const int per = (total + nwarps - 1) / nwarps;

  auto reset = [&](int b, int g) {
    const auto* q32 = static_cast<const uint32_t*>(a.q);
#pragma unroll
    for (int rb = 0; rb < kRB; ++rb) {
      m_run[rb] = -INFINITY;
      l_run[rb] = 0.f;
#pragma unroll
      for (int db = 0; db < 8; ++db)
#pragma unroll
        for (int e = 0; e < 4; ++e) oacc[rb][db][e] = 0.f;
      const bool ok = head_ok[rb];
      const int64_t row =
          ok ? ((int64_t)b * a.q_sb + (int64_t)(g * a.Gs + a.hoff + 8 * rb + grp) * a.q_sh) / 2 : 0;
#pragma unroll
      for (int kb = 0; kb < 8; ++kb) {
        qa[rb][kb][0] = ok ? __ldg(q32 + row + kb * 8 + tig) : 0u;
        qa[rb][kb][1] = ok ? __ldg(q32 + row + kb * 8 + 4 + tig) : 0u;
      }
    }
  };

  // write the current (b, g): the output itself when this segment holds all
  // of its batches, else a partial for the combine kernel
  auto flush = [&]() {
    const int nb_ = s_nbat[cu];
    const int firstb = s_bstart[cu] + (a.kvh ? 0 : cg * nb_);   // first batch of (cb, cg) in the list
    const bool whole = firstb / per == (firstb + nb_ - 1) / per;   // one segment holds it all
    const int seg = gw - firstb / per;
#pragma unroll
    for (int rb = 0; rb < kRB; ++rb) {
      // (max, sum) of the heads in this lane's O^T columns of row block rb
      const float mA = __shfl_sync(0xffffffffu, m_run[rb], 8 * tig);
      const float lA = __shfl_sync(0xffffffffu, l_run[rb], 8 * tig);
      const float mB = __shfl_sync(0xffffffffu, m_run[rb], 8 * tig + 4);
      const float lB = __shfl_sync(0xffffffffu, l_run[rb], 8 * tig + 4);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int hl = 8 * rb + (c ? hB : hA);
        if (hl >= Gn) continue;
        const float m = c ? mB : mA, l = c ? lB : lA;
        const int h = cg * a.Gs + a.hoff + hl;
        if (whole) {
          float* op = a.out + ((int64_t)cb * a.H + h) * kHeadDim + grp;
          const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
          for (int db = 0; db < 8; ++db) {
            op[db * 16] = oacc[rb][db][c] * inv;
            op[db * 16 + 8] = oacc[rb][db][2 + c] * inv;
          }
        } else {
          float* pp = a.part + (((int64_t)cb * a.H + h) * a.splits + seg) * (2 + kHeadDim);
          if (grp == 0) {
            pp[0] = m;
            pp[1] = l;
          }
#pragma unroll
          for (int db = 0; db < 8; ++db) {
            pp[2 + db * 16 + grp] = oacc[rb][db][c];
            pp[2 + db * 16 + 8 + grp] = oacc[rb][db][2 + c];
          }
        }
      }
    }
  };

  for (int t = t0; t < t1; ++t) {
    if (pc.b != cb || pc.g != cg) {
      if (cb >= 0) flush();
      cb = pc.b;
      cg = pc.g;
      cu = pc.u;
      reset(cb, cg);
    }
    // K(t) is complete once at most V(t) is pending
    cp_async_wait<1>();
    __syncwarp();
    const unsigned vm = vm_cur;
    const bool more = t + 1 < t1;

    // S = q . K^T: A = q (16 rows = heads), B = K rows (n = 8 tokens)
    float sacc[4][4];
#pragma unroll
    for (int nb = 0; nb < 4; ++nb) {
#pragma unroll
      for (int e = 0; e < 4; ++e) sacc[nb][e] = 0.f;
      const int trow = nb * 8 + (lane & 7);
#pragma unroll
      for (int kp = 0; kp < 4; ++kp) {
        const int c = 4 * kp + (lane >> 3);
        uint32_t bk[4];
        ldmatrix_x4(sk + (c >> 3) * kHalfBytes + trow * 128 + (((c & 7) ^ (trow & 7)) << 4), bk);
        // rows 8..15 of A: the second row block of 16 heads, else zero
        const uint32_t a0[4] = {qa[0][2 * kp][0], kRB > 1 ? qa[kRB - 1][2 * kp][0] : 0u, qa[0][2 * kp][1],
                                kRB > 1 ? qa[kRB - 1][2 * kp][1] : 0u};
        const uint32_t a1[4] = {qa[0][2 * kp + 1][0], kRB > 1 ? qa[kRB - 1][2 * kp + 1][0] : 0u,
                                qa[0][2 * kp + 1][1], kRB > 1 ? qa[kRB - 1][2 * kp + 1][1] : 0u};
        mma_16816<DT>(sacc[nb], a0, bk[0], bk[1]);
        mma_16816<DT>(sacc[nb], a1, bk[2], bk[3]);
      }
    }
    // the K region is free: fetch K(t + 1), and the entries of batch t + 2
    __syncwarp();
    if (more) {
      jcur = check(pi, jnext);
      vm_next = __ballot_sync(0xffffffffu, jcur >= 0);
      issue_rows(pi, sk, kbase, a.k_sb, a.k_sh, ksn, jcur);
      jnext = t + 2 < t1 ? load_idx(pl) : -1;
      advance(pl);
    }
    // online softmax of head grp (+8 for row block 1) over the batch's tokens
    // nb*8 + 2*tig + {0,1}
    uint32_t pb[kRB][2][2][2];   // [row block][k block][hi/lo][tokens 0-7 | 8-15 of the block]
#pragma unroll
    for (int rb = 0; rb < kRB; ++rb) {
      float z[8];
      float tmax = -INFINITY;
#pragma unroll
      for (int nb = 0; nb < 4; ++nb)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int tkn = nb * 8 + 2 * tig + e;
          const float v = ((vm >> tkn) & 1u) ? sacc[nb][2 * rb + e] * kLog2eInvSqrtD : -INFINITY;
          z[nb * 2 + e] = v;
          tmax = fmaxf(tmax, v);
        }
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 1));
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 2));
      const float mn = fmaxf(m_run[rb], tmax);   // finite: every batch holds a token
      const float corr = ex2(m_run[rb] - mn);    // 0 on the first batch
      float p[8], psum = 0.f;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        p[u] = head_ok[rb] ? ex2(z[u] - mn) : 0.f;
        psum += p[u];
      }
      psum += __shfl_xor_sync(0xffffffffu, psum, 1);
      psum += __shfl_xor_sync(0xffffffffu, psum, 2);
      l_run[rb] = l_run[rb] * corr + psum;
      m_run[rb] = mn;
      // rescale O^T: columns hA, hB take the factor of their head
      const float cA = __shfl_sync(0xffffffffu, corr, 8 * tig);
      const float cB = __shfl_sync(0xffffffffu, corr, 8 * tig + 4);
#pragma unroll
      for (int db = 0; db < 8; ++db) {
        oacc[rb][db][0] *= cA;
        oacc[rb][db][2] *= cA;
        if constexpr (G > 1) {
          oacc[rb][db][1] *= cB;
          oacc[rb][db][3] *= cB;
        }
      }
      // P as B fragments (k = token, n = head grp), split into a 16-bit high
      // part and its 16-bit residual so the weights keep ~22 bits
#pragma unroll
      for (int kt = 0; kt < 2; ++kt)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          const float x = p[(2 * kt + hf) * 2], y = p[(2 * kt + hf) * 2 + 1];
          const uint32_t hi = pack2<DT>(x, y);
          const float2 hv = unpack2<DT>(hi);
          pb[rb][kt][0][hf] = hi;
          pb[rb][kt][1][hf] = pack2<DT>(x - hv.x, y - hv.y);
        }
    }
    // V(t) is complete once at most K(t + 1) is pending
    if (more) cp_async_wait<1>();
    else cp_async_wait<0>();
    __syncwarp();
    // O^T += V^T . P^T: A = V^T (16 dims x 16 tokens) by transposed ldmatrix
#pragma unroll
    for (int kt = 0; kt < 2; ++kt) {
      const int trow = kt * 16 + (lane & 7) + ((lane >> 4) & 1) * 8;
#pragma unroll
      for (int db = 0; db < 8; ++db) {
        const int c = 2 * db + ((lane >> 3) & 1);
        uint32_t av[4];
        ldmatrix_x4_trans(sv + (c >> 3) * kHalfBytes + trow * 128 + (((c & 7) ^ (trow & 7)) << 4), av);
#pragma unroll
        for (int rb = 0; rb < kRB; ++rb) {
          mma_16816<DT>(oacc[rb][db], av, pb[rb][kt][0][0], pb[rb][kt][0][1]);
          mma_16816<DT>(oacc[rb][db], av, pb[rb][kt][1][0], pb[rb][kt][1][1]);
        }
      }
    }
    // the V region is free: fetch V(t + 1)
    __syncwarp();
    if (more) {
      issue_rows(pi, sv, vbase, a.v_sb, a.v_sh, vsn, jcur);
      advance(pi);
    }
    vm_cur = vm_next;
    advance(pc);
  }
  flush();
}

// Merge the partials of one (b, h) whose batches were split over several
// warps: out = sum_s 2^{M_s - M} O_s / sum_s 2^{M_s - M} L_s (maxima in the
// base-2 scale of the attention kernel).  Pairs held whole by one warp were
// written directly; sequences with no selected token get zeros.  One CTA per
// (b, h): kCombGroups groups of kHeadDim threads (one per output dimension)
// each merge every kCombGroups-th partial with a running maximum, the loads
// of several partials in flight at once, and the group results are merged in
// shared memory.  A short budget split over many warps (one batch per warp)
// leaves dozens of partials per pair, so their loads must not be serialised.
constexpr int kCombGroups = 4;
constexpr int kCombThreads = kCombGroups * kHeadDim;

__global__ void __launch_bounds__(kCombThreads) hill_attn_combine_kernel(AttnArgs a, int total_warps) {
  __shared__ int s_first, s_nb, s_total;
  __shared__ float s_m[kCombGroups], s_l[kCombGroups];
  __shared__ float s_o[kCombGroups][kHeadDim];
  const int bh = blockIdx.x;
  const int b = bh / a.H, h = bh % a.H;
  const int G = a.H / a.Hkv, g = h / G;
  const int tid = threadIdx.x, dd = tid % kHeadDim, gi = tid / kHeadDim;
  __shared__ int s_nbu[kMaxBatchAttn];
  pdl_wait();
  // the batch layout of the attention kernel (see its table units)
  const int R = a.kvh ? a.B * a.Hkv : a.B;
  for (int u = tid; u < R; u += kCombThreads) s_nbu[u] = (clamp_count(a, u) + kBatch - 1) / kBatch;
  __syncthreads();
  if (tid == 0) {
    const int upb = a.kvh ? 1 : a.Hkv;
    const int mine = a.kvh ? b * a.Hkv + g : b;
    int acc = 0, first = 0, nb = 0;
    for (int u = 0; u < R; ++u) {
      const int nbu = s_nbu[u];
      if (u == mine) {
        first = acc + (a.kvh ? 0 : g * nbu);
        nb = nbu;
      }
      acc += upb * nbu;
    }
    s_first = first;
    s_nb = nb;
    s_total = acc;
  }
  __syncthreads();
  const int nb = s_nb, first = s_first, total = s_total;
  float* op = a.out + (int64_t)bh * kHeadDim + dd;
  if (nb == 0) {
    if (gi == 0) *op = 0.f;
    return;
  }
  const int per = (total + total_warps - 1) / total_warps;
  const int w0 = first / per, w1 = (first + nb - 1) / per;
  if (w0 == w1) return;   // one warp held every batch and wrote the output
  constexpr int kPS = 2 + kHeadDim;   // one partial: max, sum, o[kHeadDim]
  const float* pp = a.part + (int64_t)bh * a.splits * kPS;
  const int nseg = w1 - w0 + 1;
  float M = -INFINITY, L = 0.f, O = 0.f;
  // KU partials per group have their loads issued together; a pair with few
  // partials (nseg is the same for the whole CTA) takes the short variant
  auto merge = [&](auto ku) {
    constexpr int KU = decltype(ku)::value;
    for (int s0 = gi; s0 < nseg; s0 += kCombGroups * KU) {
      float ms[KU], ls[KU], os[KU];
#pragma unroll
      for (int u = 0; u < KU; ++u) {
        const int s = s0 + u * kCombGroups;
        const float* q = pp + (int64_t)s * kPS;
        ms[u] = s < nseg ? q[0] : -INFINITY;
        ls[u] = s < nseg ? q[1] : 0.f;
        os[u] = s < nseg ? q[2 + dd] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < KU; ++u) {
        if (ms[u] == -INFINITY) continue;   // past the end (every written partial holds a token)
        const float mn = fmaxf(M, ms[u]);
        const float c0 = ex2(M - mn), c1 = ex2(ms[u] - mn);   // partial maxima are in the base-2 scale
        L = L * c0 + ls[u] * c1;
        O = O * c0 + os[u] * c1;
        M = mn;
      }
    }
  };
  if (nseg <= kCombGroups * 2) merge(std::integral_constant<int, 2>{});
  else merge(std::integral_constant<int, 16>{});
  s_o[gi][dd] = O;
  if (dd == 0) {
    s_m[gi] = M;
    s_l[gi] = L;
  }
  __syncthreads();
  if (gi == 0) {
    float Mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < kCombGroups; ++i) Mx = fmaxf(Mx, s_m[i]);
    float Ls = 0.f, Os = 0.f;
    if (Mx != -INFINITY) {
#pragma unroll
      for (int i = 0; i < kCombGroups; ++i) {
        const float c = s_m[i] == -INFINITY ? 0.f : ex2(s_m[i] - Mx);
        Ls += s_l[i] * c;
        Os += s_o[i][dd] * c;
      }
    }
    *op = Ls > 0.f ? Os / Ls : 0.f;
  }
}

template <int DT, int G>
cudaError_t launch_attn_t(const AttnArgs& a, int grid, bool combine, cudaStream_t st) {
  static int cache[64] = {0};
  auto kern = hill_sparse_attn_kernel<DT, G>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), AttnCfg::kSmem, cache);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3(grid), dim3(kAThreads), AttnCfg::kSmem, st, 0, a);
  if (e != cudaSuccess || !combine) return e;
  return launch_pdl(hill_attn_combine_kernel, dim3(a.B * a.H), dim3(kCombThreads), 0, st, 0, a, grid * kAW);
}

template <int DT>
cudaError_t launch_attn_d(const AttnArgs& a, int G, int grid, bool combine, cudaStream_t st) {
  switch (G) {
    case 1: return launch_attn_t<DT, 1>(a, grid, combine, st);
    case 2: return launch_attn_t<DT, 2>(a, grid, combine, st);
    case 4: return launch_attn_t<DT, 4>(a, grid, combine, st);
    case 8: return launch_attn_t<DT, 8>(a, grid, combine, st);
    case 16: return launch_attn_t<DT, 16>(a, grid, combine, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int attn_batch_tokens() { return kBatch; }
int attn_max_batch() { return kMaxBatchAttn; }

// Partial slots per (b, h): a (b, g) of nb batches meets at most
// ceil(nb / per) + 1 warp segments, and per >= 1.
int attn_max_segments(int max_k) { return (max_k + kBatch - 1) / kBatch + 1; }

cudaError_t launch_sparse_attn(const AttnArgs& a, int dtype, int G, int grid, bool combine, cudaStream_t st) {
  return dtype == 0 ? launch_attn_d<0>(a, G, grid, combine, st) : launch_attn_d<1>(a, G, grid, combine, st);
}

}  // namespace hill
