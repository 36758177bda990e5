// select.cu -- per-sequence top-k selection (Sec. 3.1 top-alpha retention;
// Sec. 4.2: the global top-alpha after merging every score source).
//
// A sequence's scores are held on chip as 32-bit order-preserving keys, by
// one CTA when they fit (up to kChunkMax keys), otherwise by a thread-block
// cluster of C CTAs, each holding a contiguous chunk.  The exact k-th largest
// key is found by an MSD radix select with digits of 11, 11 and 10 bits.  In
// each pass every CTA histograms the keys that match the digits fixed so
// far; after one cluster barrier every CTA adds up all C histograms through
// distributed shared memory and searches the merged bins itself, so all CTAs
// reach the same digit without further exchange.  The crossing bin is found
// in two levels -- every warp sums its slice of the bins, one warp scans the
// 32 slice sums and then the bins of the crossing slice.  A pass ends the
// search early when the crossing bin is taken whole.  The first pass can
// start from a histogram of the leading digit that the score normalisation
// already accumulated (SelectArgs::hist0).  With 8-CTA clusters the keys of
// the first pass's crossing bucket, when few, are gathered into every CTA so
// that the later passes need no exchange.  This is the GPU form of the
// paper's merge of chunked <position, score> blocks (Sec. 4.2): the chunks
// stay on chip and only bin counts (or the few candidate keys) cross between
// CTAs.  All global reads are issued before the first use of any of them.
//
// Ties at the boundary go to the lowest token index: with tau the k-th key
// and r_eq the number of keys equal to tau that must be taken, a token is
// selected iff key > tau, or key == tau and fewer than r_eq keys equal to tau
// precede it.  Every thread owns a contiguous run of keys; a block scan of
// the per-thread counts (and a cluster exchange of the CTA totals) gives each
// run its output position, so idx comes out in ascending order without a
// sort.
#include <cooperative_groups.h>

#include "hill_internal.h"

namespace cg = cooperative_groups;

namespace hill {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kBins = 2048;
constexpr int kMaxCluster = 8;
constexpr int kChunkMax = 16384;   // keys per CTA before the cluster grows
constexpr int kCand = kBins;       // crossing-bucket keys a cluster gathers into each CTA
constexpr int kCandMinCluster = 8; // cluster size from which it gathers them
constexpr int kHistBufs = 3;       // one per pass: no buffer is rewritten while a peer may read it

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
  // row = one key row; with per-KV-head selection a sequence has
  // rows_per_seq rows that share its length and budget
  const int row = blockIdx.y;
  const int b = row / a.rows_per_seq;
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  pdl_wait();
  pdl_launch_dependents();

  extern __shared__ __align__(16) uint32_t sm[];
  uint32_t* keys = sm;                       // [chunk]
  uint32_t* histbuf = keys + a.chunk;        // [kHistBufs][kBins], pass p uses buffer p
  uint32_t* merged = histbuf + kHistBufs * kBins;   // [kBins]: the cluster's sum for this pass
  __shared__ uint32_t wtot[kSelWarps];
  __shared__ uint32_t cnt[kMaxCluster];
  __shared__ uint32_t cnt2[kMaxCluster];
  __shared__ uint32_t s_nc;
  __shared__ uint32_t bc[3];

  // Every global read the search needs is issued before the first use of
  // any of them, so the kernel pays one memory round trip, not one per
  // input: the length and budget, the upstream leading-digit histogram, and
  // this CTA's chunk of keys.  The keys are read up to the capacity (valid
  // memory); rows at or beyond the length are never counted.
  int len = a.lens[b];
  int kk = a.k[b];
  constexpr int kH0 = kBins / kSelThreads;
  uint32_t h0v[kH0];
  if (a.hist0) {
    const uint32_t* h0 = a.hist0 + (int64_t)row * kBins;
#pragma unroll
    for (int j = 0; j < kH0; ++j) h0v[j] = h0[tid + j * kSelThreads];
  }
  const int j_lo = r * a.chunk;
  const int ncap = max(0, min(a.chunk, a.cap - j_lo));
  const float* kp = a.key + (int64_t)row * a.cap + j_lo;
  int i_tail = 0;
  if ((reinterpret_cast<uintptr_t>(kp) & 15u) == 0) {
    // 16-byte loads when the chunk starts on a 16-byte boundary
    const int n4 = ncap >> 2;
    const float4* kp4 = reinterpret_cast<const float4*>(kp);
    uint4* k4 = reinterpret_cast<uint4*>(keys);
#pragma unroll 4
    for (int i = tid; i < n4; i += kSelThreads) {
      const float4 v = kp4[i];
      k4[i] = make_uint4(ordered_key(v.x), ordered_key(v.y), ordered_key(v.z), ordered_key(v.w));
    }
    i_tail = n4 << 2;
  }
#pragma unroll 8
  for (int i = i_tail + tid; i < ncap; i += kSelThreads) keys[i] = ordered_key(kp[i]);
  for (int i = tid; i < kHistBufs * kBins; i += kSelThreads) histbuf[i] = 0;

  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  // BKP temporal pinning (Sec. 4.2): the most recent tokens [older, len) are
  // kept outright; the ranking runs over [0, older)
  const int rec = a.recent > 0 ? a.recent : 0;
  const int rfull = rec < len ? rec : len;
  const int older = len - rfull;
  int win = rfull;
  kk = kk < 0 ? 0 : (kk > older ? older : kk);
  if (win > a.max_k || kk > a.max_k - min(win, a.max_k)) {
    if (r == 0 && tid == 0) raise_error(a.err, kErrDevArg);
    win = min(win, a.max_k);           // the most recent max_k tokens of the window
    kk = min(kk, a.max_k - win);
  }
  int32_t* out = a.idx + (int64_t)row * a.max_k;
  uint16_t* hits = a.hits ? a.hits + (int64_t)row * a.cap : nullptr;
  auto hit = [&](int j) {   // the hit-rate table: +1 per kept token, saturating
    if (hits && hits[j] != 0xffffu) hits[j] = (uint16_t)(hits[j] + 1u);
  };
  const int n = max(0, min(j_lo + a.chunk, older) - j_lo);

  // padding, count and the pinned window (every path)
  for (int p = kk + win + r * kSelThreads + tid; p < a.max_k; p += C * kSelThreads) out[p] = -1;
  if (r == 0 && tid == 0) a.count[row] = kk + win;
  for (int j = max(j_lo, len - win) + tid; j < min(j_lo + a.chunk, len); j += kSelThreads) {
    out[kk + j - (len - win)] = j;
    hit(j);
  }
  if (kk == 0) return;
  if (kk == older) {  // every older token is selected
    for (int i = tid; i < n; i += kSelThreads) {
      out[j_lo + i] = j_lo + i;
      hit(j_lo + i);
    }
    return;
  }
  __syncthreads();

  uint32_t prefix = 0, pmask = 0;
  uint32_t remaining = (uint32_t)kk;
  bool take_bucket = false;    // the crossing bucket is taken whole
  const uint32_t* src = keys;  // the keys histogrammed by passes 1 and 2
  int nsrc = n;
  bool local = !CL;            // a pass needs no exchange between CTAs
#pragma unroll 1
  for (int pass = 0; pass < 3; ++pass) {
    const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
    const int nb = pass == 2 ? 1024 : 2048;
    const uint32_t dmask = (uint32_t)nb - 1u;
    uint32_t* hist = histbuf + pass * kBins;
    const uint32_t* om = merged;
    if (pass == 0 && a.hist0) {
      // leading-digit counts over the whole sequence, accumulated upstream
#pragma unroll
      for (int j = 0; j < kH0; ++j) merged[tid + j * kSelThreads] = h0v[j];
    } else {
      for (int i = tid; i < nsrc; i += kSelThreads) {
        const uint32_t kv = src[i];
        if ((kv & pmask) == prefix) atomicAdd(&hist[(kv >> shift) & dmask], 1u);
      }
      if (local) {
        __syncthreads();
      } else {
        csync();  // every CTA's histogram of this pass is complete
        // all peer reads are issued before any sum is stored
        uint32_t v[kH0] = {};
#pragma unroll
        for (int c = 0; c < kMaxCluster; ++c) {
          if (c < C) {
            const uint32_t* h = remote(hist, c);
#pragma unroll
            for (int j = 0; j < kH0; ++j)
              if (tid + j * kSelThreads < nb) v[j] += h[tid + j * kSelThreads];
          }
        }
#pragma unroll
        for (int j = 0; j < kH0; ++j)
          if (tid + j * kSelThreads < nb) merged[tid + j * kSelThreads] = v[j];
      }
      if (local) om = hist;
    }
    __syncthreads();
    // Two-level search over positions p = 0..nb-1 (bins from the top down):
    // warp w sums positions [w*S, (w+1)*S), then warp 0 scans the 32 sums
    // and the positions of the crossing slice.
    const int S = nb / kSelWarps;   // 64 or 32
    {
      uint32_t v = 0;
      for (int p = warp * S + lane; p < (warp + 1) * S; p += 32) v += om[nb - 1 - p];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) wtot[warp] = v;
    }
    __syncthreads();
    if (warp == 0) {
      const uint32_t t = wtot[lane];
      uint32_t inc = t;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
      }
      const uint32_t need = remaining;   // >= 1
      const unsigned hit = __ballot_sync(0xffffffffu, inc >= need);
      const int ws = hit ? __ffs(hit) - 1 : 31;    // slice holding the crossing
      uint32_t cum = __shfl_sync(0xffffffffu, inc - t, ws);
      for (int p0 = ws * S; p0 < (ws + 1) * S; p0 += 32) {
        const int p = p0 + lane;
        const uint32_t c = om[nb - 1 - p];
        uint32_t ci = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, ci, o);
          if (lane >= o) ci += y;
        }
        const unsigned h = __ballot_sync(0xffffffffu, cum + ci >= need);
        if (h) {
          if (lane == __ffs(h) - 1) {
            bc[0] = (uint32_t)(nb - 1 - p);
            bc[1] = need - (cum + ci - c);
            bc[2] = c;
          }
          break;
        }
        cum += __shfl_sync(0xffffffffu, ci, 31);
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
    if (!local && pass == 0 && C >= kCandMinCluster && bc[2] <= (uint32_t)kCand) {
      // The keys of the crossing bucket are few (typically 1-4 % of the
      // sequence): every CTA gathers all of them from the cluster once, and
      // the two remaining passes then run on that copy inside each CTA, with
      // no further histogram exchange.  All CTAs hold the same multiset, so
      // they reach the same digits.  (Measured: this pays off against the
      // exchange of 2 x C histograms at C = 8 and loses at C = 2.)  The
      // buffers: this CTA's own candidates go to `merged` (free after the
      // search above; peers read it until the compaction's cluster barrier),
      // the gathered copy to histogram buffer 0 (peers have finished reading
      // it once they pass the barrier below).
      uint32_t* cand = merged;
      if (tid == 0) s_nc = 0;
      __syncthreads();
      for (int w0 = warp * 32; w0 < n; w0 += kSelThreads) {   // warp-uniform trip count
        const int i = w0 + lane;
        const uint32_t kv = i < n ? keys[i] : 0u;
        const bool m = i < n && (kv & pmask) == prefix;
        const unsigned bal = __ballot_sync(0xffffffffu, m);
        if (bal) {
          uint32_t base = 0;
          if (lane == 0) base = atomicAdd(&s_nc, (uint32_t)__popc(bal));
          base = __shfl_sync(0xffffffffu, base, 0) + (uint32_t)__popc(bal & ((1u << lane) - 1u));
          if (m && base < (uint32_t)kCand) cand[base] = kv;
        }
      }
      __syncthreads();
      if (tid < C) remote(cnt2, tid)[r] = s_nc;
      csync();  // every CTA's candidates and count are in place
      uint32_t offs[kMaxCluster + 1];
      offs[0] = 0;
#pragma unroll
      for (int c = 0; c < kMaxCluster; ++c) offs[c + 1] = offs[c] + (c < C ? min(cnt2[c], (uint32_t)kCand) : 0u);
      const uint32_t tot = offs[kMaxCluster];
      if (tot != bc[2] && tid == 0) raise_error(a.err, kErrDevArg);   // cannot happen: counts disagree
      uint32_t* all = histbuf;
      constexpr int kCandPer = kCand / kSelThreads;
      uint32_t v[kCandPer];
#pragma unroll
      for (int j = 0; j < kCandPer; ++j) {   // every peer read is issued before any store
        const uint32_t i = (uint32_t)(tid + j * kSelThreads);
        int c = 0;
        uint32_t base = 0;
#pragma unroll
        for (int cc = 1; cc < kMaxCluster; ++cc)
          if (i >= offs[cc]) {
            c = cc;
            base = offs[cc];
          }
        v[j] = i < tot ? remote(cand, c)[i - base] : 0u;
      }
#pragma unroll
      for (int j = 0; j < kCandPer; ++j)
        if ((uint32_t)(tid + j * kSelThreads) < tot) all[tid + j * kSelThreads] = v[j];
      src = all;
      nsrc = (int)min(tot, (uint32_t)kCand);
      local = true;
      __syncthreads();
    }
  }
  // Selection rule: take_bucket -> key >= prefix (every key of the crossing
  // bucket and above); otherwise tau = prefix is the k-th key itself and
  // `remaining` of the keys equal to tau are taken, lowest index first.
  const uint32_t tau = prefix;
  auto is_gt = [&](uint32_t kv) { return take_bucket ? kv >= tau : kv > tau; };
  auto is_eq = [&](uint32_t kv) { return !take_bucket && kv == tau; };

  // ---------------------------------------------------------------- compaction
  // thread t owns keys [t*m, t*m + m) of the chunk (m odd: conflict-free
  // strided reads); counts are packed as (above tau) << 16 | (equal to tau),
  // a chunk holding fewer than 2^16 keys
  const int m = ((n + kSelThreads - 1) / kSelThreads) | 1;
  const int i0 = min(n, tid * m), i1 = min(n, i0 + m);
  uint32_t mine = 0;
  for (int i = i0; i < i1; ++i) {
    const uint32_t kv = keys[i];
    mine += is_gt(kv) ? (1u << 16) : (is_eq(kv) ? 1u : 0u);
  }
  // exclusive block scan of the packed counts
  uint32_t inc = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wtot[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    const uint32_t t = wtot[lane];
    uint32_t wi = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += y;
    }
    wtot[lane] = wi - t;                       // exclusive prefix of warp totals
    if (lane == 31) bc[0] = wi;                // the CTA total
  }
  __syncthreads();
  const uint32_t before = wtot[warp] + inc - mine;   // this thread's exclusive prefix in the CTA
  uint32_t gt_before = 0, eq_before = 0;
  if (CL) {
    if (tid < C) remote(cnt, tid)[r] = bc[0];
    csync();
    for (int c = 0; c < r; ++c) {
      gt_before += cnt[c] >> 16;
      eq_before += cnt[c] & 0xffffu;
    }
  }
  uint32_t eq_rank = eq_before + (before & 0xffffu);   // ties before this run
  uint32_t pos = gt_before + (before >> 16) + min(eq_rank, remaining);
  for (int i = i0; i < i1; ++i) {
    const uint32_t kv = keys[i];
    bool take = is_gt(kv);
    if (is_eq(kv)) {
      take = eq_rank < remaining;
      ++eq_rank;
    }
    if (take) {
      if (pos < (uint32_t)kk) {
        out[pos] = j_lo + i;
        hit(j_lo + i);
      } else {
        raise_error(a.err, kErrDevArg);   // cannot happen: more picks than the budget
      }
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
  return (size_t)chunk * 4 + (kHistBufs + 1) * kBins * 4;
}

int select_hist_bins() { return kBins; }

cudaError_t launch_select(const SelectArgs& a0, cudaStream_t st) {
  SelectArgs a = a0;
  const int C = select_cluster_size(a.cap);
  a.chunk = (a.cap + C - 1) / C;
  const size_t smem = select_smem_bytes(a.cap, C);
  const dim3 grid(C, a.B * a.rows_per_seq, 1), block(kSelThreads, 1, 1);
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
