// attn.cu -- decode attention over the selected tokens only (Sec. 4.1, workflow step 6:
// only the critical KV reaches the attention; Eq. 1 restricted to the set).
//
// Gather + split-K flash decode on persistent CTAs.  The work is a list of
// batches: (sequence b, KV head g, batch bi of 32 consecutive entries of
// b's index list), ordered b, g, bi.  Every warp of the grid owns one
// contiguous segment of that list and streams it through two shared-memory
// slots.  A batch's 32 K rows and 32 V rows (tokens idx[b][32*bi + i]) and
// the G query rows of the head group are gathered with 16-byte asynchronous
// copies (one cp.async group per batch, a half-warp per 256-byte row) into
// an XOR-swizzled layout that ldmatrix reads without bank conflicts; rows of
// absent tokens are zero-filled.  The index entries of the batch after next
// are loaded while the current one computes and are checked only when that
// batch is issued.  (TMA alternatives were measured slower on the same
// layout: 256-byte bulk copies per row are bound by the copy engine's
// request rate, and tile::gather4 loads reached about 85 % of the cp.async
// throughput; neither depends on how scattered the rows are.)
// Both products run on mma.sync m16n8k16 with fp32 accumulation: S^T =
// q . K^T (the G query heads are the rows, K rows read with ldmatrix), an
// online softmax per head across the batches of one (b, g), and O += P . V
// with V read by transposed ldmatrix; the weights P enter the tensor cores
// as a 16-bit high part plus its 16-bit residual.  When a warp's segment
// holds all batches of a (b, g) it writes the output; otherwise it writes a
// partial (max, sum, o) that hill_attn_combine_kernel merges.
#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kAW = 6;                               // warps per CTA
constexpr int kAThreads = kAW * 32;
constexpr int kBatch = 32;                           // selected entries per batch
constexpr int kMaxBatchAttn = 512;                   // sequences in the per-CTA table

constexpr int kHalfBytes = kBatch * 128;             // 32 rows x 64 dims, swizzled

template <int G>
struct AttnCfg {
  // K dims 0-63 | K dims 64-127 | V dims 0-63 | V dims 64-127 | q rows
  static constexpr int kSlotBytes = ((4 * kHalfBytes + G * kRowBytes + 1023) / 1024) * 1024;
  static constexpr int kSmem = kAW * 2 * kSlotBytes + 1024;   // + alignment slack
};

// Batch list bookkeeping shared by the attention and combine kernels.
struct BatchTable {
  const int* bstart;   // [B + 1]: first batch of sequence b
  const int* nbat;     // [B]: batches per (b, g)
  int B, Hkv;

  __device__ __forceinline__ void decode(int t, int& b, int& g, int& bi) const {
    int lo = 0, hi = B;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (bstart[mid] <= t) lo = mid; else hi = mid;
    }
    b = lo;
    const int rem = t - bstart[b];
    g = rem / nbat[b];
    bi = rem - g * nbat[b];
  }
};

__device__ __forceinline__ int clamp_count(const AttnArgs& a, int b) {
  const int n = a.count[b];
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
  using Cfg = AttnCfg<G>;
  extern __shared__ unsigned char asmem[];
  __shared__ int s_bstart[kMaxBatchAttn + 1];
  __shared__ int s_nbat[kMaxBatchAttn];
  __shared__ int s_cnt[kMaxBatchAttn];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait();
  pdl_launch_dependents();

  for (int b = threadIdx.x; b < a.B; b += kAThreads) {
    const int n = clamp_count(a, b);
    s_cnt[b] = n;
    s_nbat[b] = (n + kBatch - 1) / kBatch;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int b = 0; b < a.B; ++b) {
      s_bstart[b] = acc;
      acc += a.Hkv * s_nbat[b];
    }
    s_bstart[a.B] = acc;
  }
  __syncthreads();
  const BatchTable tab{s_bstart, s_nbat, a.B, a.Hkv};
  const int total = s_bstart[a.B];
  int t0, t1;
  warp_segment(total, gridDim.x * kAW, blockIdx.x * kAW + warp, t0, t1);
  if (t0 >= t1) return;

  const uint32_t base_addr = (smem_addr(asmem) + 1023u) & ~1023u;
  const uint32_t slot0 = base_addr + warp * 2 * Cfg::kSlotBytes;
  const auto* qbase = static_cast<const uint16_t*>(a.q);

  // raw index entry of this lane for batch t (-1 past the count).  Nothing
  // here depends on the loaded value, so the load stays in flight until the
  // batch is issued one iteration later, where it is checked.
  auto load_idx = [&](int t) -> int {
    int b, g, bi;
    tab.decode(t, b, g, bi);
    const int e = bi * kBatch + lane;
    return e < s_cnt[b] ? a.idx[(int64_t)b * a.max_k + e] : -1;
  };
  // gather batch t into slot s: row r of the batch is token jj of lane r
  // (-1: none, zero-filled).  A half-warp copies one 256-byte row; chunk c
  // (16 bytes) of row r goes to 128-byte line r of half c / 8 at position
  // (c % 8) ^ (r % 8), so the ldmatrix reads below are conflict-free.
  auto issue = [&](int t, int s, int jj) {
    int b, g, bi;
    tab.decode(t, b, g, bi);
    if (bi * kBatch + lane < s_cnt[b] && (jj < 0 || jj >= a.cap)) {
      raise_error(a.err, kErrDevArg);   // a listed entry outside [0, cap): skipped
      jj = -1;
    }
    const unsigned vm = __ballot_sync(0xffffffffu, jj >= 0);
    const uint32_t sk = slot0 + s * Cfg::kSlotBytes;
    const uint16_t* kr = static_cast<const uint16_t*>(a.k) + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh;
    const uint16_t* vr = static_cast<const uint16_t*>(a.v) + (int64_t)b * a.v_sb + (int64_t)g * a.v_sh;
    const int l16 = lane & 15, hf = l16 >> 3, cc = l16 & 7;
#pragma unroll 4
    for (int i = 0; i < 16; ++i) {
      const int row = 2 * i + (lane >> 4);
      const int j = __shfl_sync(0xffffffffu, jj, row);
      const uint32_t off = hf * kHalfBytes + row * 128 + ((cc ^ (row & 7)) << 4);
      if (j >= 0) {
        cp_async16(sk + off, kr + (int64_t)j * a.k_sn + l16 * 8);
        cp_async16(sk + 2 * kHalfBytes + off, vr + (int64_t)j * a.v_sn + l16 * 8);
      } else {
        sts128_zero(sk + off);
        sts128_zero(sk + 2 * kHalfBytes + off);
      }
    }
    const uint16_t* qr = qbase + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh;
#pragma unroll
    for (int hh = lane >> 4; hh < G; hh += 2)
      cp_async16(sk + 4 * kHalfBytes + hh * kRowBytes + l16 * 16, qr + (int64_t)hh * a.q_sh + l16 * 8);
    cp_async_commit();
    return vm;
  };

  // prologue: batches t0 and t0 + 1, and the indices of t0 + 2
  unsigned vmask[2] = {0u, 0u};
  int jnext = -1;
  {
    int j0 = load_idx(t0);
    int j1 = t0 + 1 < t1 ? load_idx(t0 + 1) : -1;
    vmask[0] = issue(t0, 0, j0);
    if (t0 + 1 < t1) vmask[1] = issue(t0 + 1, 1, j1);
    if (t0 + 2 < t1) jnext = load_idx(t0 + 2);
  }

  // mma.sync fragments: row grp = lane/4 of the 16-row tiles is query head
  // grp of the group (rows >= G and 8..15 are zero); tig = lane%4.
  const int grp = lane >> 2, tig = lane & 3;
  const bool head_ok = grp < G;
  // running softmax of head grp (the 4 lanes of a group hold the same values)
  // and its output tile O[grp][nb*8 + 2*tig + {0,1}] for the 16 dim blocks nb
  float m_run = -INFINITY, l_run = 0.f;
  float oacc[16][4];
  auto reset = [&]() {
    m_run = -INFINITY;
    l_run = 0.f;
#pragma unroll
    for (int nb = 0; nb < 16; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) oacc[nb][e] = 0.f;
  };
  reset();
  int cb = -1, cg = -1;   // the (b, g) being accumulated

  // write the current (b, g): the output itself when this segment holds all
  // of its batches, else a partial for the combine kernel
  auto flush = [&]() {
    const int nb_ = s_nbat[cb];
    const int first = s_bstart[cb] + cg * nb_;   // first batch of (cb, cg) in the list
    const int per = (total + gridDim.x * kAW - 1) / (gridDim.x * kAW);
    const bool whole = first / per == (first + nb_ - 1) / per;   // one segment holds it all
    const int seg = (blockIdx.x * kAW + warp) - first / per;
    if (!head_ok) return;
    const int h = cg * G + grp;
    if (whole) {
      float* op = a.out + ((int64_t)cb * a.H + h) * kHeadDim + 2 * tig;
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
#pragma unroll
      for (int nb = 0; nb < 16; ++nb) {
        op[nb * 8] = oacc[nb][0] * inv;
        op[nb * 8 + 1] = oacc[nb][1] * inv;
      }
    } else {
      float* pp = a.part + (((int64_t)cb * a.H + h) * a.splits + seg) * (2 + kHeadDim);
      if (tig == 0) {
        pp[0] = m_run;
        pp[1] = l_run;
      }
#pragma unroll
      for (int nb = 0; nb < 16; ++nb) {
        pp[2 + nb * 8 + 2 * tig] = oacc[nb][0];
        pp[2 + nb * 8 + 2 * tig + 1] = oacc[nb][1];
      }
    }
  };

  for (int t = t0; t < t1; ++t) {
    const int s = (t - t0) & 1;
    const uint32_t sk = slot0 + s * Cfg::kSlotBytes;
    const uint32_t sv = sk + 2 * kHalfBytes;
    const uint32_t sq = sk + 4 * kHalfBytes;
    int b, g, bi;
    tab.decode(t, b, g, bi);
    if (b != cb || g != cg) {
      if (cb >= 0) flush();
      reset();
      cb = b;
      cg = g;
    }
    const unsigned vm = vmask[s];
    if (t + 1 < t1) cp_async_wait<1>(); else cp_async_wait<0>();
    __syncwarp();

    // S^T = q . K^T: A = q (16 rows = heads), B = K rows (n = 8 tokens)
    uint32_t qa[8][2];
#pragma unroll
    for (int kb = 0; kb < 8; ++kb) {
      if (head_ok) {
        const uint32_t qaddr = sq + grp * kRowBytes + (kb * 16 + tig * 2) * 2;
        qa[kb][0] = lds32(qaddr);
        qa[kb][1] = lds32(qaddr + 16);
      } else {
        qa[kb][0] = 0u;
        qa[kb][1] = 0u;
      }
    }
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
        const uint32_t a0[4] = {qa[2 * kp][0], 0u, qa[2 * kp][1], 0u};
        const uint32_t a1[4] = {qa[2 * kp + 1][0], 0u, qa[2 * kp + 1][1], 0u};
        mma_16816<DT>(sacc[nb], a0, bk[0], bk[1]);
        mma_16816<DT>(sacc[nb], a1, bk[2], bk[3]);
      }
    }
    // online softmax of head grp over the batch's tokens nb*8 + 2*tig + {0,1}
    float z[8];
    float tmax = -INFINITY;
#pragma unroll
    for (int nb = 0; nb < 4; ++nb)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int tkn = nb * 8 + 2 * tig + e;
        const float v = ((vm >> tkn) & 1u) ? sacc[nb][e] * kInvSqrtD : -INFINITY;
        z[nb * 2 + e] = v;
        tmax = fmaxf(tmax, v);
      }
    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 1));
    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 2));
    const float mn = fmaxf(m_run, tmax);
    const float corr = (m_run == -INFINITY) ? 0.f : expf(m_run - mn);
    float p[8], psum = 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      p[u] = (mn == -INFINITY || z[u] == -INFINITY) ? 0.f : expf(z[u] - mn);
      psum += p[u];
    }
    psum += __shfl_xor_sync(0xffffffffu, psum, 1);
    psum += __shfl_xor_sync(0xffffffffu, psum, 2);
    l_run = l_run * corr + psum;
    m_run = mn;
#pragma unroll
    for (int nb = 0; nb < 16; ++nb) {
      oacc[nb][0] *= corr;
      oacc[nb][1] *= corr;
    }
    // O += P . V: A = P (heads x 16 tokens per k block), split into a 16-bit
    // high part and the 16-bit residual so the weights keep ~22 bits; B = V
    // rows read transposed (k = token, n = dim)
    uint32_t pa[2][2][2];   // [k block][hi/lo][token pair 0-7 | 8-15]
#pragma unroll
    for (int kt = 0; kt < 2; ++kt)
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const float x = p[(2 * kt + hf) * 2], y = p[(2 * kt + hf) * 2 + 1];
        const uint32_t hi = pack2<DT>(x, y);
        const float2 hv = unpack2<DT>(hi);
        pa[kt][0][hf] = hi;
        pa[kt][1][hf] = pack2<DT>(x - hv.x, y - hv.y);
      }
#pragma unroll
    for (int kt = 0; kt < 2; ++kt) {
      const int trow = kt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
      const uint32_t ahi[4] = {pa[kt][0][0], 0u, pa[kt][0][1], 0u};
      const uint32_t alo[4] = {pa[kt][1][0], 0u, pa[kt][1][1], 0u};
#pragma unroll
      for (int np = 0; np < 8; ++np) {
        const int c = 2 * np + (lane >> 4);
        uint32_t bv[4];
        ldmatrix_x4_trans(sv + (c >> 3) * kHalfBytes + trow * 128 + (((c & 7) ^ (trow & 7)) << 4), bv);
        mma_16816<DT>(oacc[2 * np], ahi, bv[0], bv[1]);
        mma_16816<DT>(oacc[2 * np], alo, bv[0], bv[1]);
        mma_16816<DT>(oacc[2 * np + 1], ahi, bv[2], bv[3]);
        mma_16816<DT>(oacc[2 * np + 1], alo, bv[2], bv[3]);
      }
    }
    // the slot is free: refill it with batch t + 2, prefetch the indices of t + 3
    __syncwarp();
    if (t + 2 < t1) {
      vmask[s] = issue(t + 2, s, jnext);
      jnext = t + 3 < t1 ? load_idx(t + 3) : -1;
    }
  }
  if (cb >= 0) flush();
}

// Merge the partials of one (b, h) whose batches were split over several
// warps: out = sum_s e^{M_s - M} O_s / sum_s e^{M_s - M} L_s.  Pairs held
// whole by one warp were written directly; sequences with no selected token
// get zeros.
__global__ void __launch_bounds__(kHeadDim) hill_attn_combine_kernel(AttnArgs a, int total_warps) {
  __shared__ int s_first, s_nb, s_total;
  const int bh = blockIdx.x;
  const int b = bh / a.H, h = bh % a.H;
  const int G = a.H / a.Hkv, g = h / G;
  const int dd = threadIdx.x;
  pdl_wait();
  pdl_launch_dependents();
  if (dd == 0) {
    int acc = 0, first = 0, nb = 0;
    for (int bb = 0; bb < a.B; ++bb) {
      const int nbb = (clamp_count(a, bb) + kBatch - 1) / kBatch;
      if (bb == b) {
        first = acc + g * nbb;
        nb = nbb;
      }
      acc += a.Hkv * nbb;
    }
    s_first = first;
    s_nb = nb;
    s_total = acc;
  }
  __syncthreads();
  const int nb = s_nb, first = s_first, total = s_total;
  float* op = a.out + (int64_t)bh * kHeadDim + dd;
  if (nb == 0) {
    *op = 0.f;
    return;
  }
  const int per = (total + total_warps - 1) / total_warps;
  const int w0 = first / per, w1 = (first + nb - 1) / per;
  if (w0 == w1) return;   // one warp held every batch and wrote the output
  const float* pp = a.part + (int64_t)bh * a.splits * (2 + kHeadDim);
  const int nseg = w1 - w0 + 1;
  float M = -INFINITY;
  for (int s = 0; s < nseg; ++s) M = fmaxf(M, pp[s * (2 + kHeadDim)]);
  float L = 0.f, O = 0.f;
  if (M != -INFINITY) {
    for (int s = 0; s < nseg; ++s) {
      const float* q = pp + s * (2 + kHeadDim);
      const float c = q[0] == -INFINITY ? 0.f : expf(q[0] - M);
      L += q[1] * c;
      O += q[2 + dd] * c;
    }
  }
  *op = L > 0.f ? O / L : 0.f;
}

template <int DT, int G>
cudaError_t launch_attn_t(const AttnArgs& a, int grid, cudaStream_t st) {
  static int cache[64] = {0};
  auto kern = hill_sparse_attn_kernel<DT, G>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), AttnCfg<G>::kSmem, cache);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3(grid), dim3(kAThreads), AttnCfg<G>::kSmem, st, 0, a);
  if (e != cudaSuccess) return e;
  return launch_pdl(hill_attn_combine_kernel, dim3(a.B * a.H), dim3(kHeadDim), 0, st, 0, a, grid * kAW);
}

template <int DT>
cudaError_t launch_attn_d(const AttnArgs& a, int G, int grid, cudaStream_t st) {
  switch (G) {
    case 1: return launch_attn_t<DT, 1>(a, grid, st);
    case 2: return launch_attn_t<DT, 2>(a, grid, st);
    case 4: return launch_attn_t<DT, 4>(a, grid, st);
    case 8: return launch_attn_t<DT, 8>(a, grid, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int attn_batch_tokens() { return kBatch; }
int attn_max_batch() { return kMaxBatchAttn; }

// Partial slots per (b, h): a (b, g) of nb batches meets at most
// ceil(nb / per) + 1 warp segments, and per >= 1.
int attn_max_segments(int max_k) { return (max_k + kBatch - 1) / kBatch + 1; }

cudaError_t launch_sparse_attn(const AttnArgs& a, int dtype, int G, int grid, cudaStream_t st) {
  return dtype == 0 ? launch_attn_d<0>(a, G, grid, st) : launch_attn_d<1>(a, G, grid, st);
}

}  // namespace hill
