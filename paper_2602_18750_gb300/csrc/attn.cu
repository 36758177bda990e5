// attn.cu -- decode attention over the selected tokens only (Sec. 4.1, workflow step 6:
// only the critical KV reaches the attention; Eq. 1 restricted to the set).
//
// Gather + split-K flash decode on persistent CTAs.  The work is a list of
// batches: (sequence b, KV head g, batch bi of 32 consecutive entries of
// b's index list), ordered b, g, bi.  Every warp of the grid owns one
// contiguous segment of that list and streams it through two shared-memory
// slots: each batch's 32 K rows, 32 V rows (tokens idx[b][32*bi + i]) and the
// G query rows of the head group are gathered with 16-byte asynchronous
// copies (one cp.async group per batch, a half-warp per 256-byte row); the
// indices of the batch after next are loaded while the current one computes.
// (Per-row bulk TMA copies were measured slower here: at 256 bytes each the
// copy engine's per-request cost, not DRAM, bounds the gather.)  Lanes then own
// 16 bytes of a row (a half-warp covers one row), partial dots for 16 rows
// finish with the transposed reduction, an online softmax keeps (max, sum,
// o) per query head across the batches of one (b, g), and the V rows are
// accumulated with the weights shuffled back to the lanes that read them.
// When a warp's segment holds all batches of a (b, g) it writes the output;
// otherwise it writes a partial (max, sum, o) that hill_attn_combine_kernel
// merges.
#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kAW = 6;                               // warps per CTA
constexpr int kAThreads = kAW * 32;
constexpr int kBatch = 32;                           // selected entries per batch
constexpr int kMaxBatchAttn = 512;                   // sequences in the per-CTA table

template <int G>
struct AttnCfg {
  static constexpr int kSlotBytes = 2 * kBatch * kRowBytes + G * kRowBytes;   // K, V, q
  static constexpr int kSmem = kAW * 2 * kSlotBytes;
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
__global__ void __launch_bounds__(kAThreads, 1) hill_sparse_attn_kernel(AttnArgs a) {
  using Cfg = AttnCfg<G>;
  extern __shared__ __align__(128) unsigned char asmem[];
  __shared__ int s_bstart[kMaxBatchAttn + 1];
  __shared__ int s_nbat[kMaxBatchAttn];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int l16 = lane & 15, half = lane >> 4;
  const int tok = 2 * l16 + half;
  pdl_wait();
  pdl_launch_dependents();

  for (int b = threadIdx.x; b < a.B; b += kAThreads) s_nbat[b] = (clamp_count(a, b) + kBatch - 1) / kBatch;
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

  const uint32_t slot0 = smem_addr(asmem) + warp * 2 * Cfg::kSlotBytes;
  const auto* qbase = static_cast<const uint16_t*>(a.q);
  const auto* kbase = static_cast<const uint16_t*>(a.k);
  const auto* vbase = static_cast<const uint16_t*>(a.v);

  // token index of this lane for batch t (-1 if none)
  auto load_idx = [&](int t) -> int {
    int b, g, bi;
    tab.decode(t, b, g, bi);
    const int e = bi * kBatch + lane;
    int j = e < clamp_count(a, b) ? a.idx[(int64_t)b * a.max_k + e] : -1;
    if (j >= a.cap || (j < 0 && e < clamp_count(a, b))) {
      raise_error(a.err, kErrDevArg);
      j = -1;
    }
    return j;
  };
  // gather batch t into slot s: row r of the batch is token jj of lane r
  // (-1: nothing to copy); one cp.async group per batch
  auto issue = [&](int t, int s, int jj) {
    int b, g, bi;
    tab.decode(t, b, g, bi);
    const unsigned vm = __ballot_sync(0xffffffffu, jj >= 0);
    const uint32_t sk = slot0 + s * Cfg::kSlotBytes;
    const uint16_t* kr = kbase + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh + l16 * 8;
    const uint16_t* vr = vbase + (int64_t)b * a.v_sb + (int64_t)g * a.v_sh + l16 * 8;
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      const int row = 2 * it + half;
      const int j = __shfl_sync(0xffffffffu, jj, row);
      if (j >= 0) {
        cp_async16(sk + row * kRowBytes + l16 * 16, kr + (int64_t)j * a.k_sn);
        cp_async16(sk + (kBatch + row) * kRowBytes + l16 * 16, vr + (int64_t)j * a.v_sn);
      }
    }
    const uint16_t* qr = qbase + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh + l16 * 8;
#pragma unroll
    for (int hh = half; hh < G; hh += 2)
      cp_async16(sk + (2 * kBatch + hh) * kRowBytes + l16 * 16, qr + (int64_t)hh * a.q_sh);
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

  float m[G], l[G], o[G][8];
  auto reset = [&]() {
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
      m[hh] = -INFINITY;
      l[hh] = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) o[hh][e] = 0.f;
    }
  };
  reset();
  int cb = -1, cg = -1;   // the (b, g) being accumulated

  // write the current (b, g): the output itself when this segment holds all
  // of its batches, else a partial for the combine kernel
  auto flush = [&]() {
    const int nb = s_nbat[cb];
    const int first = s_bstart[cb] + cg * nb;   // first batch of (cb, cg) in the list
    const int per = (total + gridDim.x * kAW - 1) / (gridDim.x * kAW);
    const bool whole = first / per == (first + nb - 1) / per;   // one segment holds it all
    const int seg = (blockIdx.x * kAW + warp) - first / per;
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
      float oo[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) oo[e] = o[hh][e] + __shfl_xor_sync(0xffffffffu, o[hh][e], 16);
      const int h = cg * G + hh;
      if (whole) {
        if (half == 0) {
          float* op = a.out + ((int64_t)cb * a.H + h) * kHeadDim + l16 * 8;
          const float inv = l[hh] > 0.f ? 1.f / l[hh] : 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) op[e] = oo[e] * inv;
        }
      } else {
        float* pp = a.part + (((int64_t)cb * a.H + h) * a.splits + seg) * (2 + kHeadDim);
        if (lane == 0) {
          pp[0] = m[hh];
          pp[1] = l[hh];
        }
        if (half == 0) {
#pragma unroll
          for (int e = 0; e < 8; ++e) pp[2 + l16 * 8 + e] = oo[e];
        }
      }
    }
  };

  for (int t = t0; t < t1; ++t) {
    const int s = (t - t0) & 1;
    const uint32_t sk = slot0 + s * Cfg::kSlotBytes;
    const uint32_t sv = sk + kBatch * kRowBytes;
    const uint32_t sq = sk + 2 * kBatch * kRowBytes;
    int b, g, bi;
    tab.decode(t, b, g, bi);
    if (b != cb || g != cg) {
      if (cb >= 0) flush();
      reset();
      cb = b;
      cg = g;
    }
    const unsigned vm = vmask[s];
    // batch t is the older of at most two outstanding groups
    if (t + 1 < t1) cp_async_wait<1>(); else cp_async_wait<0>();
    __syncwarp();

    float qf[G][8];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) to_float8<DT>(lds128(sq + hh * kRowBytes + l16 * 16), qf[hh]);
    float acc[G][16];
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      float kf[8];
      to_float8<DT>(lds128(sk + (2 * it + half) * kRowBytes + l16 * 16), kf);
#pragma unroll
      for (int hh = 0; hh < G; ++hh) {
        float sum = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) sum = fmaf(qf[hh][e], kf[e], sum);
        acc[hh][it] = sum;
      }
    }
    const bool valid = (vm >> tok) & 1u;
    float p[G];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
      const float z = half_transpose_reduce(acc[hh], lane) * kInvSqrtD;
      const float bm = warp_max(valid ? z : -INFINITY);
      const float mn = fmaxf(m[hh], bm);
      const float corr = m[hh] == -INFINITY ? 0.f : expf(m[hh] - mn);
      p[hh] = valid ? expf(z - mn) : 0.f;
      l[hh] = l[hh] * corr + warp_sum(p[hh]);
      m[hh] = mn;
#pragma unroll
      for (int e = 0; e < 8; ++e) o[hh][e] *= corr;
    }
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      const int row = 2 * it + half;
      const int src = (row & 1) << 4 | (row >> 1);   // lane holding token `row`
      float w[G];
#pragma unroll
      for (int hh = 0; hh < G; ++hh) w[hh] = __shfl_sync(0xffffffffu, p[hh], src);
      if ((vm >> row) & 1u) {   // rows that were not gathered hold stale bytes
        float vf[8];
        to_float8<DT>(lds128(sv + row * kRowBytes + l16 * 16), vf);
#pragma unroll
        for (int hh = 0; hh < G; ++hh)
#pragma unroll
          for (int e = 0; e < 8; ++e) o[hh][e] = fmaf(w[hh], vf[e], o[hh][e]);
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
