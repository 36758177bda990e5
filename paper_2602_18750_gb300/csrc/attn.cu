// attn.cu -- decode attention over the selected tokens only (Sec. 3.1 step 6:
// only the critical KV reaches the attention; Eq. 1 restricted to the set).
//
// Split-K flash decode with a gather: the grid is (splits, Hkv, B); a CTA
// takes a slice of one sequence's selected positions for one KV head and all
// G query heads that read it.  A warp handles batches of 32 selected tokens:
// lanes own 16 bytes of a row (a half-warp covers one row), the token index
// is broadcast with a shuffle and the K rows are gathered with 128-bit
// loads, partial dots for 16 rows finish with the transposed reduction, the
// online softmax (running max / sum) is updated per head, and the V rows of
// the same batch are accumulated with the weights shuffled back to the
// lanes that read them.  Warps of a CTA merge in shared memory; splits merge
// in hill_attn_combine_kernel.
#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kAttnWarps = 4;
constexpr int kAttnThreads = kAttnWarps * 32;

template <int DT, int G>
__global__ void __launch_bounds__(kAttnThreads) hill_sparse_attn_kernel(AttnArgs a) {
  const int sp = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int l16 = lane & 15, half = lane >> 4;
  const int tok = 2 * l16 + half;

  int n = a.count[b];
  n = n < 0 ? 0 : (n > a.max_k ? a.max_k : n);
  const int t0 = sp * a.per_split;
  const int t1 = min(t0 + a.per_split, n);

  const auto* qp = static_cast<const uint16_t*>(a.q) + (int64_t)b * a.q_sb + (int64_t)(g * G) * a.q_sh;
  const auto* kp = static_cast<const uint16_t*>(a.k) + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh;
  const auto* vp = static_cast<const uint16_t*>(a.v) + (int64_t)b * a.v_sb + (int64_t)g * a.v_sh;
  const int32_t* ip = a.idx + (int64_t)b * a.max_k;

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

  for (int tb = t0 + warp * 32; tb < t1; tb += kAttnWarps * 32) {
    const int nb = min(32, t1 - tb);
    int jj = lane < nb ? ip[tb + lane] : -1;
    if (lane < nb && (jj < 0 || jj >= a.cap)) {
      raise_error(a.err, kErrDevArg);
      jj = -1;
    }
    uint4 kv[16];
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      const int j = __shfl_sync(0xffffffffu, jj, 2 * it + half);
      kv[it] = j >= 0 ? ldg_nc128(kp + (int64_t)j * a.k_sn + l16 * 8) : make_uint4(0, 0, 0, 0);
    }
    float acc[G][16];
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      float kf[8];
      to_float8<DT>(kv[it], kf);
#pragma unroll
      for (int hh = 0; hh < G; ++hh) {
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) s = fmaf(qf[hh][e], kf[e], s);
        acc[hh][it] = s;
      }
    }
    // V rows of the batch (issued before the softmax arithmetic)
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      const int j = __shfl_sync(0xffffffffu, jj, 2 * it + half);
      kv[it] = j >= 0 ? ldg_nc128(vp + (int64_t)j * a.v_sn + l16 * 8) : make_uint4(0, 0, 0, 0);
    }
    const int jt = __shfl_sync(0xffffffffu, jj, tok);
    const bool valid = jt >= 0;
    float p[G];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
      const float z = half_transpose_reduce(acc[hh], lane) * kInvSqrtD;
      const float bm = warp_max(valid ? z : -INFINITY);
      const float mn = fmaxf(m[hh], bm);
      if (mn == -INFINITY) {  // nothing valid yet
        p[hh] = 0.f;
        continue;
      }
      const float corr = expf(m[hh] - mn);
      p[hh] = valid ? expf(z - mn) : 0.f;
      l[hh] = l[hh] * corr + warp_sum(p[hh]);
      m[hh] = mn;
#pragma unroll
      for (int e = 0; e < 8; ++e) o[hh][e] *= corr;
    }
#pragma unroll
    for (int it = 0; it < 16; ++it) {
      float vf[8];
      to_float8<DT>(kv[it], vf);
      const int src = ((2 * it + half) & 1) << 4 | ((2 * it + half) >> 1);  // lane holding token 2*it+half
#pragma unroll
      for (int hh = 0; hh < G; ++hh) {
        const float w = __shfl_sync(0xffffffffu, p[hh], src);
#pragma unroll
        for (int e = 0; e < 8; ++e) o[hh][e] = fmaf(w, vf[e], o[hh][e]);
      }
    }
  }
  // the two half-warps hold disjoint rows: add them
#pragma unroll
  for (int hh = 0; hh < G; ++hh)
#pragma unroll
    for (int e = 0; e < 8; ++e) o[hh][e] += __shfl_xor_sync(0xffffffffu, o[hh][e], 16);

  // merge the warps of this CTA
  __shared__ float sm_m[kAttnWarps][G], sm_l[kAttnWarps][G];
  __shared__ float sm_o[kAttnWarps][G][kHeadDim];
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
      for (int e = 0; e < 8; ++e) sm_o[warp][hh][l16 * 8 + e] = o[hh][e];
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
        O += sm_o[w][hh][dd] * c;
      }
    }
    const int h = g * G + hh;
    if (a.splits == 1) {
      a.out[((int64_t)b * a.H + h) * kHeadDim + dd] = L > 0.f ? O / L : 0.f;
    } else {
      float* pp = a.part + (((int64_t)b * a.H + h) * a.splits + sp) * (2 + kHeadDim);
      if (dd == 0) {
        pp[0] = M;
        pp[1] = L;
      }
      pp[2 + dd] = O;
    }
  }
}

__global__ void __launch_bounds__(kHeadDim) hill_attn_combine_kernel(AttnArgs a) {
  const int bh = blockIdx.x;
  const int dd = threadIdx.x;
  const float* pp = a.part + (int64_t)bh * a.splits * (2 + kHeadDim);
  float M = -INFINITY;
  for (int s = 0; s < a.splits; ++s) M = fmaxf(M, pp[s * (2 + kHeadDim)]);
  float L = 0.f, O = 0.f;
  if (M != -INFINITY) {
    for (int s = 0; s < a.splits; ++s) {
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
  dim3 grid(a.splits, a.Hkv, a.B);
  hill_sparse_attn_kernel<DT, G><<<grid, kAttnThreads, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
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

cudaError_t launch_sparse_attn(const AttnArgs& a, int dtype, int G, cudaStream_t st) {
  return dtype == 0 ? launch_attn_d<0>(a, G, st) : launch_attn_d<1>(a, G, st);
}

}  // namespace hill
