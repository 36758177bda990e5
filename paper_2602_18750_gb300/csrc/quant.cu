// quant.cu -- the 8-bit key shadow used by the asymmetric-precision scoring
// (Sec. 4.4: the evaluation ranks tokens with low-precision inner products;
// the attention keeps the original 16-bit keys and values).
//
// Each (b, g, j) row of K (128 dims) becomes 128 E4M3 codes and one float32
// scale: amax = max |K|, r = 448 / amax, code_i = e4m3(K_i * r) (float32
// product, round to nearest even, saturating), scale = amax / 448.  One warp
// per row: every lane converts 4 dims, a shuffle reduction gives amax, and
// the warp stores the row's 128 bytes in one coalesced transaction.
#include "hill_internal.h"

namespace hill {
namespace {

constexpr int kQWarps = 8;

template <int DT>
__global__ void __launch_bounds__(kQWarps * 32) hill_quantize_k_kernel(QuantArgs a) {
  pdl_wait();
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.z, g = blockIdx.y;
  int j0 = a.row_begin[b], j1 = a.row_end[b];
  j0 = j0 < 0 ? 0 : (j0 > a.cap ? a.cap : j0);
  j1 = j1 < j0 ? j0 : (j1 > a.cap ? a.cap : j1);
  const int j = j0 + blockIdx.x * kQWarps + warp;
  if (j >= j1) return;
  const auto* kr = static_cast<const uint16_t*>(a.k) + (int64_t)b * a.k_sb + (int64_t)g * a.k_sh +
                   (int64_t)j * a.k_sn + lane * 4;
  const uint2 raw = *reinterpret_cast<const uint2*>(kr);
  float x[4];
  {
    const uint4 v{raw.x, raw.y, 0u, 0u};
    float f[8];
    to_float8<DT>(v, f);
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = f[i];
  }
  float amax = fmaxf(fmaxf(fabsf(x[0]), fabsf(x[1])), fmaxf(fabsf(x[2]), fabsf(x[3])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const int64_t row = ((int64_t)b * a.Hkv + g) * a.cap + j;
  uint32_t w = 0u;
  if (amax > 0.f) {
    const float r = __fdiv_rn(448.f, amax);
    w = e4m3x2(__fmul_rn(x[0], r), __fmul_rn(x[1], r)) | (e4m3x2(__fmul_rn(x[2], r), __fmul_rn(x[3], r)) << 16);
  }
  reinterpret_cast<uint32_t*>(a.k8 + row * kHeadDim)[lane] = w;
  if (lane == 0) a.kscale[((int64_t)b * a.Hkv + g) * a.cap32 + j] = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
}

}  // namespace

cudaError_t launch_quantize_k(const QuantArgs& a, int dtype, int max_rows, cudaStream_t st) {
  const dim3 grid((max_rows + kQWarps - 1) / kQWarps, a.Hkv, a.B);
  if (dtype == 0) return launch_pdl(hill_quantize_k_kernel<0>, grid, dim3(kQWarps * 32), 0, st, 0, a);
  return launch_pdl(hill_quantize_k_kernel<1>, grid, dim3(kQWarps * 32), 0, st, 0, a);
}

}  // namespace hill
