// select.cu -- per-sequence top-k selection (Sec. 3.1 top-alpha retention;
// Sec. 4.2: the global top-alpha after merging every score source).
//
// A sequence's scores are held on chip as 32-bit order-preserving keys, by
// one CTA when they fit (up to kChunkMax keys), otherwise by a thread-block
// cluster of C CTAs, each holding a contiguous chunk.  The exact k-th largest
// key is found by an MSD radix select with digits of 11, 11 and 10 bits.  In
// each pass every CTA histograms the keys that match the digits fixed so
// far; CTA r merges bins [r*W, (r+1)*W) of all CTAs' histograms through
// distributed shared memory and publishes its bin total; every CTA then finds
// the crossing bin itself by reading the owner's merged bins.  A pass ends
// the search early when the crossing bin is taken whole.  This is the GPU
// form of the paper's merge of chunked <position, score> blocks (Sec. 4.2):
// the chunks stay on chip and only bin counts cross between CTAs.
//
// Ties at the boundary go to the lowest token index: with tau the k-th key
// and r_eq the number of keys equal to tau that must be taken, a token is
// selected iff key > tau, or key == tau and fewer than r_eq keys equal to tau
// precede it.  Output positions come from prefix counts over (CTA, thread,
// element) in index order, so idx is ascending without a sort.
#include <cooperative_groups.h>

#include "hill_internal.h"

namespace cg = cooperative_groups;

namespace hill {
namespace {

constexpr int kSelThreads = 512;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kBins = 2048;
constexpr int kMaxCluster = 8;
constexpr int kChunkMax = 16384;   // keys per CTA before the cluster grows

// Exclusive prefix sum over the block (thread order); *total gets the sum.
// wsum needs kSelWarps + 1 entries.
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* wsum, uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();  // wsum may still be read by a previous scan
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    const uint32_t t = lane < kSelWarps ? wsum[lane] : 0u;
    uint32_t u = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, u, o);
      if (lane >= o) u += y;
    }
    if (lane < kSelWarps) wsum[lane] = u - t;
    if (lane == 31) wsum[kSelWarps] = u;
  }
  __syncthreads();
  *total = wsum[kSelWarps];
  return wsum[warp] + x - v;
}

template <bool CL>
__global__ void __launch_bounds__(kSelThreads) hill_select_kernel(SelectArgs a) {
  int C = 1, r = 0;
  cg::cluster_group cluster = cg::this_cluster();
  if (CL) {
    C = (int)cluster.num_blocks();
    r = (int)cluster.block_rank();
  }
  auto csync = [&]() {
    if (CL) cluster.sync(); else __syncthreads();
  };
  auto remote = [&](uint32_t* p, int c) -> uint32_t* {
    return CL ? cluster.map_shared_rank(p, c) : p;
  };
  const int b = blockIdx.y;
  const int tid = threadIdx.x;
  pdl_wait();
  pdl_launch_dependents();

  extern __shared__ uint32_t sm[];
  uint32_t* keys = sm;                   // [chunk]
  uint32_t* hist = keys + a.chunk;       // [kBins]
  uint32_t* merged = hist + kBins;       // [kBins] (only [0, nb / C) used)
  __shared__ uint32_t wsum[kSelWarps + 1];
  __shared__ uint32_t tot[kMaxCluster];
  __shared__ uint32_t cgt[kMaxCluster], ceq[kMaxCluster];
  __shared__ uint32_t bc[3];

  int len = a.lens[b];
  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  int kk = a.k[b];
  kk = kk < 0 ? 0 : (kk > len ? len : kk);
  if (kk > a.max_k) {
    if (r == 0 && tid == 0) raise_error(a.err, kErrDevArg);
    kk = a.max_k;
  }
  int32_t* out = a.idx + (int64_t)b * a.max_k;
  const int j_lo = r * a.chunk;
  const int j_hi = min(j_lo + a.chunk, len);
  const int n = max(0, j_hi - j_lo);

  // padding and count (every path)
  for (int p = kk + r * kSelThreads + tid; p < a.max_k; p += C * kSelThreads) out[p] = -1;
  if (r == 0 && tid == 0) a.count[b] = kk;
  if (kk == 0) return;
  if (kk == len) {  // everything is selected
    for (int i = tid; i < n; i += kSelThreads) out[j_lo + i] = j_lo + i;
    return;
  }

  const float* kp = a.key + (int64_t)b * a.cap + j_lo;
  for (int i = tid; i < n; i += kSelThreads) keys[i] = ordered_key(kp[i]);

  uint32_t prefix = 0, pmask = 0;
  uint32_t remaining = (uint32_t)kk;
  bool take_bucket = false;    // the crossing bucket is taken whole
#pragma unroll 1
  for (int pass = 0; pass < 3; ++pass) {
    const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
    const int nb = pass == 2 ? 1024 : 2048;
    const uint32_t dmask = (uint32_t)nb - 1u;
    for (int i = tid; i < nb; i += kSelThreads) hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < n; i += kSelThreads) {
      const uint32_t kv = keys[i];
      if ((kv & pmask) == prefix) atomicAdd(&hist[(kv >> shift) & dmask], 1u);
    }
    csync();  // (A) every local histogram is complete

    int W = nb;
    uint32_t above = 0;
    int owner = 0;
    const uint32_t* om = hist;
    if (CL) {
      W = nb / C;
      const int base = r * W;
      uint32_t part = 0;
      for (int i = tid; i < W; i += kSelThreads) {
        uint32_t s = 0;
        for (int c = 0; c < C; ++c) s += remote(hist, c)[base + i];
        merged[i] = s;
        part += s;
      }
      uint32_t mine;
      (void)block_excl_scan(part, wsum, &mine);
      if (tid == 0)
        for (int c = 0; c < C; ++c) remote(tot, c)[r] = mine;
      csync();  // (B) merged bins and totals published; remote histogram reads done
      // which CTA's bin range holds the remaining-th largest matching key?
      for (int c = C - 1; c >= 0; --c) {
        if (above + tot[c] >= remaining) {
          owner = c;
          break;
        }
        above += tot[c];
      }
      om = remote(merged, owner);
    }
    // positions p = 0.. run over the owner's bins from the top down
    const int per = (W + kSelThreads - 1) / kSelThreads;
    const int p0 = tid * per;
    const int p1 = min(p0 + per, W);
    uint32_t s = 0;
    for (int p = p0; p < p1; ++p) s += om[W - 1 - p];
    uint32_t tall;
    const uint32_t ex = block_excl_scan(s, wsum, &tall);
    if (above + ex < remaining && remaining <= above + ex + s) {
      uint32_t cum = above + ex;
      for (int p = p0; p < p1; ++p) {
        const uint32_t c = om[W - 1 - p];
        if (cum + c >= remaining) {
          bc[0] = (uint32_t)(owner * W + W - 1 - p);
          bc[1] = remaining - cum;
          bc[2] = c;
          break;
        }
        cum += c;
      }
    }
    __syncthreads();
    prefix |= bc[0] << shift;
    pmask |= dmask << shift;
    remaining = bc[1];
    if (remaining == bc[2]) {
      take_bucket = true;
      break;
    }
  }
  // Selection rule: take_bucket -> key >= prefix (every key of the crossing
  // bucket and above); otherwise tau = prefix is the k-th key itself and
  // `remaining` of the keys equal to tau are taken, lowest index first.
  const uint32_t tau = prefix;

  // ---------------------------------------------------------------- compaction
  const int per = (n + kSelThreads - 1) / kSelThreads;
  const int i0 = tid * per, i1 = min(i0 + per, n);
  uint32_t my_gt = 0, my_eq = 0;
  for (int i = i0; i < i1; ++i) {
    const uint32_t kv = keys[i];
    if (take_bucket) {
      my_gt += kv >= tau;
    } else {
      my_gt += kv > tau;
      my_eq += kv == tau;
    }
  }
  uint32_t tgt, teq;
  const uint32_t gt_ex = block_excl_scan(my_gt, wsum, &tgt);
  const uint32_t eq_ex = block_excl_scan(my_eq, wsum, &teq);
  if (CL) {
    if (tid == 0)
      for (int c = 0; c < C; ++c) {
        remote(cgt, c)[r] = tgt;
        remote(ceq, c)[r] = teq;
      }
    csync();
  }
  uint32_t gt_before = 0, eq_before = 0;
  for (int c = 0; c < r; ++c) {
    gt_before += cgt[c];
    eq_before += ceq[c];
  }
  uint32_t eq_rank = eq_before + eq_ex;   // ties before this thread's segment
  uint32_t pos = gt_before + gt_ex + min(eq_rank, remaining);
  for (int i = i0; i < i1; ++i) {
    const uint32_t kv = keys[i];
    bool take;
    if (take_bucket) {
      take = kv >= tau;
    } else {
      take = kv > tau;
      if (kv == tau) {
        take = eq_rank < remaining;
        ++eq_rank;
      }
    }
    if (take) {
      if (pos < (uint32_t)kk) out[pos] = j_lo + i;
      else raise_error(a.err, kErrDevArg);   // cannot happen: more picks than the budget
      ++pos;
    }
  }
}

}  // namespace

int select_cluster_size(int cap) {
  int C = 1;
  while (C < kMaxCluster && (cap + C - 1) / C > kChunkMax) C <<= 1;
  return C;
}

size_t select_smem_bytes(int cap, int C) {
  const int chunk = (cap + C - 1) / C;
  return (size_t)chunk * 4 + 2 * kBins * 4;
}

cudaError_t launch_select(const SelectArgs& a0, cudaStream_t st) {
  SelectArgs a = a0;
  const int C = select_cluster_size(a.cap);
  a.chunk = (a.cap + C - 1) / C;
  const size_t smem = select_smem_bytes(a.cap, C);
  const dim3 grid(C, a.B, 1), block(kSelThreads, 1, 1);
  if (C == 1) {
    static int cache[64] = {0};
    cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(hill_select_kernel<false>), (int)smem, cache);
    if (e != cudaSuccess) return e;
    return launch_pdl(hill_select_kernel<false>, grid, block, smem, st, 0, a);
  }
  static int cache[64] = {0};
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(hill_select_kernel<true>), (int)smem, cache);
  if (e != cudaSuccess) return e;
  return launch_pdl(hill_select_kernel<true>, grid, block, smem, st, C, a);
}

}  // namespace hill
