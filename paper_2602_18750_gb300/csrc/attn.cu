// attn.cu -- decode attention over the selected tokens only (Sec. 3.1 step 6:
// only the critical KV reaches the attention; Eq. 1 restricted to the set).
//
// Gather + split-K flash decode.  The grid is (chunks, Hkv, B): a CTA takes
// kChunk consecutive entries of one sequence's index list for one KV head
// and all G query heads that read it; each of its warps owns 32 entries.  A
// warp reads its 32 token indices and every lane issues two bulk TMA copies
// (that token's K row and V row, 256 B each) into the warp's shared-memory
// slot, all completing on one mbarrier: the gather holds no registers and the
// whole CTA has 64 KB in flight at once.  Lanes then own 16 bytes of a row (a
// half-warp covers one row); partial dots for 16 rows finish with the
// transposed reduction, a softmax over the warp's tokens gives (max, sum) per
// head, and the V rows are accumulated with the weights shuffled back to the
// lanes that read them.  Warps merge in shared memory; chunks merge in
// hill_attn_combine_kernel (not launched when one chunk covers max_k).
#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kAttnWarps = 4;
constexpr int kAttnThreads = kAttnWarps * 32;
constexpr int kBatch = 32;                           // selected tokens per warp
constexpr int kChunk = kAttnWarps * kBatch;          // selected tokens per CTA
constexpr int kSlotBytes = 2 * kBatch * kRowBytes;   // K rows then V rows
constexpr int kAttnSmem = kAttnWarps * kSlotBytes;

template <int DT, int G>
__global__ void __launch_bounds__(kAttnThreads) hill_sparse_attn_kernel(AttnArgs a) {
  extern __shared__ __align__(128) unsigned char asmem[];
  __shared__ __align__(8) uint64_t bar[kAttnWarps];
  __shared__ float sm_m[kAttnWarps][G], sm_l[kAttnWarps][G];

  const int ch = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int l16 = lane & 15, half = lane >> 4;
  const int tok = 2 * l16 + half;

  int n = a.count[b];
  n = n < 0 ? 0 : (n > a.max_k ? a.max_k : n);
  if (a.splits > 1 && ch * kChunk >= n) return;      // the combine reads only used chunks
  const int tb = ch * kChunk + warp * kBatch;        // this warp's first entry
  const int nb = max(0, min(kBatch, n - tb));        // entries this warp holds

  const auto* qp = static_cast<const uint16_t*>(a.q) + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh;
  const auto* kp = static_cast<const uint16_t*>(a.k) + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh;
  const auto* vp = static_cast<const uint16_t*>(a.v) + (int64_t)b * a.v_sb + (int64_t)g * a.v_sh;
  const int32_t* ip = a.idx + (int64_t)b * a.max_k;
  unsigned char* slot = asmem + warp * kSlotBytes;
  const uint32_t sk = smem_addr(slot);
  const uint32_t sv = sk + kBatch * kRowBytes;
  const uint32_t mb = smem_addr(&bar[warp]);

  // ---- gather: one K row and one V row per lane, completing on the warp's barrier
  int jj = lane < nb ? ip[tb + lane] : -1;
  if (lane < nb && (jj < 0 || jj >= a.cap)) {
    raise_error(a.err, kErrDevArg);
    jj = -1;
  }
  const unsigned vmask = __ballot_sync(0xffffffffu, jj >= 0);
  if (vmask) {
    if (lane == 0) {
      mbar_init(mb, 1);
      fence_barrier_init();
      mbar_arrive_expect_tx(mb, (uint32_t)__popc(vmask) * 2u * kRowBytes);
    }
    __syncwarp();
    if (jj >= 0) {
      bulk_g2s(sk + lane * kRowBytes, kp + (int64_t)jj * a.k_sn, kRowBytes, mb);
      bulk_g2s(sv + lane * kRowBytes, vp + (int64_t)jj * a.v_sn, kRowBytes, mb);
    }
  }

  float qf[G][8];
#pragma unroll
  for (int hh = 0; hh < G; ++hh) to_float8<DT>(ldg_nc128(qp + (int64_t)hh * a.q_sh + l16 * 8), qf[hh]);

  float m[G], l[G], o[G][8];
#pragma unroll
  for (int hh = 0; hh < G; ++hh) {
    m[hh] = -INFINITY;
    l[hh] = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) o[hh][e] = 0.f;
  }

  bool have = false;
  if (vmask) {
    have = mbar_wait(mb, 0, a.err);
    // after a timeout, give the copies one more bounded wait before the slot
    // is reused or the CTA exits
    if (!have) (void)mbar_wait(mb, 0, a.err);
  }
  if (have) {
    float acc[G][16];
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      float kf[8];
      to_float8<DT>(lds128(sk + (2 * it + half) * kRowBytes + l16 * 16), kf);
#pragma unroll
      for (int hh = 0; hh < G; ++hh) {
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) s = fmaf(qf[hh][e], kf[e], s);
        acc[hh][it] = s;
      }
    }
    const bool valid = (vmask >> tok) & 1u;
    float p[G];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
      const float z = half_transpose_reduce(acc[hh], lane) * kInvSqrtD;
      m[hh] = warp_max(valid ? z : -INFINITY);
      p[hh] = valid ? expf(z - m[hh]) : 0.f;
      l[hh] = warp_sum(p[hh]);
    }
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      const int row = 2 * it + half;
      const int src = (row & 1) << 4 | (row >> 1);   // lane holding token `row`
      float w[G];
#pragma unroll
      for (int hh = 0; hh < G; ++hh) w[hh] = __shfl_sync(0xffffffffu, p[hh], src);
      if ((vmask >> row) & 1u) {   // rows that were not gathered hold stale bytes
        float vf[8];
        to_float8<DT>(lds128(sv + row * kRowBytes + l16 * 16), vf);
#pragma unroll
        for (int hh = 0; hh < G; ++hh)
#pragma unroll
          for (int e = 0; e < 8; ++e) o[hh][e] = fmaf(w[hh], vf[e], o[hh][e]);
      }
    }
  }
  // the two half-warps accumulated disjoint rows: add them
#pragma unroll
  for (int hh = 0; hh < G; ++hh)
#pragma unroll
    for (int e = 0; e < 8; ++e) o[hh][e] += __shfl_xor_sync(0xffffffffu, o[hh][e], 16);

  // ---- merge the warps of this CTA (slots are reused as scratch)
  __syncthreads();
  float* so = reinterpret_cast<float*>(asmem) + warp * (kSlotBytes / 4);   // [G][128]
  if (lane == 0) {
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
      sm_m[warp][hh] = m[hh];
      sm_l[warp][hh] = l[hh];
    }
  }
  if (half == 0) {
#pragma unroll
    for (int hh = 0; hh < G; ++hh)
#pragma unroll
      for (int e = 0; e < 8; ++e) so[hh * kHeadDim + l16 * 8 + e] = o[hh][e];
  }
  __syncthreads();
  for (int t = threadIdx.x; t < G * kHeadDim; t += kAttnThreads) {
    const int hh = t / kHeadDim, dd = t % kHeadDim;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, sm_m[w][hh]);
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kAttnWarps; ++w) {
        const float c = expf(sm_m[w][hh] - M);
        L += sm_l[w][hh] * c;
        O += reinterpret_cast<const float*>(asmem)[w * (kSlotBytes / 4) + hh * kHeadDim + dd] * c;
      }
    }
    const int h = g * G + hh;
    if (a.splits == 1) {
      a.out[((int64_t)b * a.H + h) * kHeadDim + dd] = L > 0.f ? O / L : 0.f;
    } else {
      float* pp = a.part + (((int64_t)b * a.H + h) * a.splits + ch) * (2 + kHeadDim);
      if (dd == 0) {
        pp[0] = M;
        pp[1] = L;
      }
      pp[2 + dd] = O;
    }
  }
}

// Merge the used chunks of one (b, h): out = sum_c e^{M_c - M} O_c / sum_c e^{M_c - M} L_c.
__global__ void __launch_bounds__(kHeadDim) hill_attn_combine_kernel(AttnArgs a) {
  const int bh = blockIdx.x;
  const int b = bh / a.H;
  const int dd = threadIdx.x;
  int n = a.count[b];
  n = n < 0 ? 0 : (n > a.max_k ? a.max_k : n);
  const int used = (n + kChunk - 1) / kChunk;
  const float* pp = a.part + (int64_t)bh * a.splits * (2 + kHeadDim);
  float M = -INFINITY;
  for (int s = 0; s < used; ++s) M = fmaxf(M, pp[s * (2 + kHeadDim)]);
  float L = 0.f, O = 0.f;
  if (M != -INFINITY) {
    for (int s = 0; s < used; ++s) {
      const float* q = pp + s * (2 + kHeadDim);
      const float c = expf(q[0] - M);
      L += q[1] * c;
      O += q[2 + dd] * c;
    }
  }
  a.out[(int64_t)bh * kHeadDim + dd] = L > 0.f ? O / L : 0.f;
}

template <int DT, int G>
cudaError_t launch_attn_t(const AttnArgs& a, cudaStream_t st) {
  static int cache[64] = {0};
  auto kern = hill_sparse_attn_kernel<DT, G>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), kAttnSmem, cache);
  if (e != cudaSuccess) return e;
  dim3 grid(a.splits, a.Hkv, a.B);
  kern<<<grid, kAttnThreads, kAttnSmem, st>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess || a.splits == 1) return e;
  hill_attn_combine_kernel<<<a.B * a.H, kHeadDim, 0, st>>>(a);
  return cudaGetLastError();
}

template <int DT>
cudaError_t launch_attn_d(const AttnArgs& a, int G, cudaStream_t st) {
  switch (G) {
    case 1: return launch_attn_t<DT, 1>(a, st);
    case 2: return launch_attn_t<DT, 2>(a, st);
    case 4: return launch_attn_t<DT, 4>(a, st);
    case 8: return launch_attn_t<DT, 8>(a, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int attn_chunk_tokens() { return kChunk; }

cudaError_t launch_sparse_attn(const AttnArgs& a, int dtype, int G, cudaStream_t st) {
  return dtype == 0 ? launch_attn_d<0>(a, G, st) : launch_attn_d<1>(a, G, st);
}

}  // namespace hill
