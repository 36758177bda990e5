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

// ---------------------------------------------------------------------------
// Lean selection: the same result as hill_select_kernel (first min(k, len)
// tokens by key descending, lower index first on ties, written in ascending
// index order), from a kernel small enough to run beside the scoring kernel
// on one SM (256 threads at most 64 registers, ~25 KB of shared memory), so
// that the selection of one layer can overlap the K stream of the next one
// (the layer pipelining of Sec. 4.3).  A row is split over a cluster of C
// CTAs; thread t of a CTA owns the contiguous run [t * run, (t + 1) * run) of
// its chunk.  While the K stream of another layer keeps HBM busy, every
// dependent round trip to global memory costs microseconds, so the kernel
// reads each key once and keeps what it learnt about it in registers:
//
//   1. The crossing bin of the leading 11 key bits comes from the histogram
//      the normalisation accumulated (SelectArgs::hist0, read together with
//      the length and budget), or from one this kernel builds (every CTA
//      histograms its chunk; the C histograms are added through distributed
//      shared memory).
//   2. One pass over the run classifies every key into two 64-bit masks
//      (above the crossing bin; in it) and stores the keys in the bin (the
//      candidates) in shared memory, each thread's in a contiguous slot range
//      that it can recompute later (per load group: a warp-reserved base plus
//      a warp scan of the per-thread counts).
//   3. The candidates of all CTAs, when they fit kLeanCand, are gathered into
//      every CTA, which finds the exact k-th key tau and the number r_eq of
//      keys equal to tau to take by two radix passes over them; otherwise the
//      radix passes run over each CTA's own candidates with cluster-merged
//      histograms.
//   4. Each thread classifies its candidates against tau (keys read back from
//      shared memory), one block scan and one cluster exchange give the
//      position of its first pick, and it writes its picks in order.
constexpr int kLeanThreads = 256;
constexpr int kLeanWarps = kLeanThreads / 32;
constexpr int kLeanCand = 2048;            // crossing-bucket keys a CTA holds (8 KB)
constexpr int kLeanBinsPerThread = kBins / kLeanThreads;   // 8
constexpr int kLeanGroup = 16;             // keys per load group (four 16-byte loads)
constexpr int kLeanRunMax = 64;            // keys per thread: the class masks are 64-bit
constexpr int kLeanGroupsMax = kLeanRunMax / kLeanGroup;
constexpr int kLeanMaxCluster = 8;         // CTAs per key row (measured: 16-CTA clusters run slower beside the K stream)

__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Block-wide search of the bin where the count from the top reaches `need`:
// on entry thread t holds the counts of bins [NBT*t, NBT*t + NBT) in v[].
// Returns, in res, the bin, the count of keys in bins above it, and the bin's
// own count; res[3] = 0 if the bins hold fewer than `need` keys.  Uses
// wtot[kLeanWarps]; ends with a __syncthreads.
template <int NBT>
__device__ __forceinline__ void lean_crossing(const uint32_t (&v)[NBT], uint32_t need, uint32_t* wtot,
                                              uint32_t* res) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t s = 0;
#pragma unroll
  for (int i = 0; i < NBT; ++i) s += v[i];
  // inclusive suffix sum over the lanes of the warp (higher lanes hold higher bins)
  uint32_t suf = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_down_sync(0xffffffffu, suf, o);
    if (lane + o < 32) suf += y;
  }
  if (lane == 0) wtot[warp] = suf;   // the warp's total
  if (tid == 0) res[3] = 0;          // found flag
  __syncthreads();
  uint32_t above = suf - s;          // keys in this warp's higher lanes
#pragma unroll
  for (int w = 0; w < kLeanWarps; ++w)
    if (w > warp) above += wtot[w];
  if (above < need && above + s >= need) {
    uint32_t cum = above;
#pragma unroll
    for (int i = NBT - 1; i >= 0; --i) {
      if (cum + v[i] >= need) {
        res[0] = (uint32_t)(NBT * tid + i);
        res[1] = cum;
        res[2] = v[i];
        res[3] = 1;
        break;
      }
      cum += v[i];
    }
  }
  __syncthreads();
}

// Warp-aggregated shared-memory histogram count: the lanes adding to one bin
// are combined into a single atomic, so keys crowding into a few bins do not
// serialise on them.  Every lane of the warp calls it.
__device__ __forceinline__ void hist_add(uint32_t* hist, uint32_t bin, bool valid) {
  const unsigned act = __ballot_sync(0xffffffffu, valid);
  if (!valid) return;
  const unsigned same = __match_any_sync(act, bin);
  if ((int)(threadIdx.x & 31) == __ffs(same) - 1) atomicAdd(&hist[bin], (uint32_t)__popc(same));
}

template <bool CL>
__global__ void __launch_bounds__(kLeanThreads, 4) hill_select_lean_kernel(SelectArgs a) {
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
  // The C CTAs' histograms h summed into dst (this CTA's shared memory):
  // consecutive threads read consecutive 16-byte pieces of every peer's
  // histogram (coalesced distributed-shared-memory loads), four peers' loads
  // in flight at a time.
  auto merge_hist = [&](uint32_t* h, uint32_t* dst) {
    uint4 acc[2] = {make_uint4(0u, 0u, 0u, 0u), make_uint4(0u, 0u, 0u, 0u)};
    for (int c0 = 0; c0 < C; c0 += 4) {
      uint4 x[4][2];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (c0 + u < C) {
          const uint4* p = reinterpret_cast<const uint4*>(remote(h, c0 + u));
          x[u][0] = p[threadIdx.x];
          x[u][1] = p[kLeanThreads + threadIdx.x];
        }
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (c0 + u < C)
#pragma unroll
          for (int v = 0; v < 2; ++v) {
            acc[v].x += x[u][v].x;
            acc[v].y += x[u][v].y;
            acc[v].z += x[u][v].z;
            acc[v].w += x[u][v].w;
          }
    }
    reinterpret_cast<uint4*>(dst)[threadIdx.x] = acc[0];
    reinterpret_cast<uint4*>(dst)[kLeanThreads + threadIdx.x] = acc[1];
  };
  __shared__ __align__(16) uint32_t cand[kLeanCand];   // this CTA's candidates, per thread in run order
  __shared__ __align__(16) uint32_t work[kLeanCand];   // every CTA's candidates, in CTA order
  __shared__ __align__(16) uint32_t hist[kBins];
  __shared__ uint32_t wtot[kLeanWarps];
  __shared__ uint32_t res[4];
  __shared__ uint32_t s_nc;                            // candidate slots reserved (may exceed kLeanCand)
  __shared__ uint32_t s_cnt[2];                        // picks above tau, keys equal to tau (this CTA)
  __shared__ uint32_t gbase[kLeanGroupsMax][kLeanWarps];
  __shared__ uint32_t p_nc[kLeanMaxCluster];

  const int row = blockIdx.y;
  const int b = row / a.rows_per_seq;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_wait();
  pdl_launch_dependents();

  // length, budget and the upstream histogram: one round trip
  int len = a.lens[b];
  int kk = a.k[b];
  uint32_t hv[kLeanBinsPerThread];
  if (a.hist0) {
    const uint4* h0 = reinterpret_cast<const uint4*>(a.hist0 + (int64_t)row * kBins + kLeanBinsPerThread * tid);
    const uint4 x = h0[0], y = h0[1];
    hv[0] = x.x; hv[1] = x.y; hv[2] = x.z; hv[3] = x.w;
    hv[4] = y.x; hv[5] = y.y; hv[6] = y.z; hv[7] = y.w;
  }
  len = len < 0 ? 0 : (len > a.cap ? a.cap : len);
  const int rec = a.recent > 0 ? a.recent : 0;
  const int rfull = rec < len ? rec : len;
  const int older = len - rfull;
  int win = rfull;
  kk = kk < 0 ? 0 : (kk > older ? older : kk);
  if (win > a.max_k || kk > a.max_k - min(win, a.max_k)) {
    if (r == 0 && tid == 0) raise_error(a.err, kErrDevArg);
    win = min(win, a.max_k);
    kk = min(kk, a.max_k - win);
  }
  int32_t* out = a.idx + (int64_t)row * a.max_k;
  uint16_t* hits = a.hits ? a.hits + (int64_t)row * a.cap : nullptr;
  auto hit = [&](int j) {
    if (hits && hits[j] != 0xffffu) hits[j] = (uint16_t)(hits[j] + 1u);
  };
  const int j_lo = r * a.chunk;
  const int n = max(0, min(j_lo + a.chunk, older) - j_lo);   // ranked keys of this chunk
  for (int p = kk + win + r * kLeanThreads + tid; p < a.max_k; p += C * kLeanThreads) out[p] = -1;
  if (r == 0 && tid == 0) a.count[row] = kk + win;
  for (int j = max(j_lo, len - win) + tid; j < min(j_lo + a.chunk, len); j += kLeanThreads) {
    out[kk + j - (len - win)] = j;
    hit(j);
  }
  if (kk == 0) return;
  if (kk == older) {
    for (int i = tid; i < n; i += kLeanThreads) {
      out[j_lo + i] = j_lo + i;
      hit(j_lo + i);
    }
    return;
  }

  // this thread's run of keys: chunk positions [i0, i0 + nv)
  const int m = a.run;
  const int i0 = tid * m;
  const int nv = max(0, min(m, n - i0));
  const float* rowk = a.key + (int64_t)row * a.cap + j_lo;
  const float* kp = rowk + i0;
  const bool vec = (reinterpret_cast<uintptr_t>(rowk) & 15u) == 0;   // runs start 4 keys apart
  const int ngroups = (m + kLeanGroup - 1) / kLeanGroup;
  auto load_group = [&](int g, uint32_t (&kv)[kLeanGroup]) {
    const int base = g * kLeanGroup;
    if (vec && base + kLeanGroup <= nv) {
      const float4* p4 = reinterpret_cast<const float4*>(kp + base);
#pragma unroll
      for (int q = 0; q < kLeanGroup / 4; ++q) {
        const float4 v = p4[q];
        kv[4 * q] = ordered_key(v.x);
        kv[4 * q + 1] = ordered_key(v.y);
        kv[4 * q + 2] = ordered_key(v.z);
        kv[4 * q + 3] = ordered_key(v.w);
      }
    } else {
#pragma unroll
      for (int e = 0; e < kLeanGroup; ++e) kv[e] = base + e < nv ? ordered_key(kp[base + e]) : 0u;
    }
  };

  // ---------------------------------------------------------------- 1. crossing bin
  if (!a.hist0) {
    for (int i = tid; i < kBins; i += kLeanThreads) hist[i] = 0u;
    __syncthreads();
    for (int g = 0; g < ngroups; ++g) {
      uint32_t kv[kLeanGroup];
      load_group(g, kv);
#pragma unroll
      for (int e = 0; e < kLeanGroup; ++e) hist_add(hist, kv[e] >> 21, g * kLeanGroup + e < nv);
    }
    csync();   // every CTA's histogram is complete
    merge_hist(hist, work);
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kLeanBinsPerThread; ++i) hv[i] = work[kLeanBinsPerThread * tid + i];
    csync();   // every peer has read this CTA's histogram
  }
  lean_crossing(hv, (uint32_t)kk, wtot, res);
  if (!res[3]) {   // the histogram holds fewer keys than the budget: inconsistent input
    if (r == 0 && tid == 0) raise_error(a.err, kErrDevArg);
    return;
  }
  const uint32_t bstar = res[0];
  uint32_t remaining = (uint32_t)kk - res[1];   // keys to take from the crossing bin (>= 1)
  const uint32_t bucket = res[2];

  // ---------------------------------------------------------------- 2. classify
  if (tid == 0) s_nc = 0;
  __syncthreads();
  uint64_t above_m = 0, cand_m = 0;
  // slot of this thread's first candidate of group g: the warp's reserved base
  // plus the warp's exclusive prefix of the per-thread counts (recomputable)
  auto group_slot = [&](int g, uint32_t cnt) -> uint32_t {
    uint32_t inc = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    return gbase[g][warp] + inc - cnt;
  };
  uint32_t kva[kLeanGroup], kvb[kLeanGroup];
  load_group(0, kva);
#pragma unroll
  for (int g = 0; g < kLeanGroupsMax; ++g) {
    if (g >= ngroups) break;
    // the next group's loads go out before this group is classified
    uint32_t (&kv)[kLeanGroup] = (g & 1) ? kvb : kva;
    if (g + 1 < ngroups) load_group(g + 1, (g & 1) ? kva : kvb);
    uint32_t mine = 0;
#pragma unroll
    for (int e = 0; e < kLeanGroup; ++e) {
      const int i = g * kLeanGroup + e;
      if (i < nv) {
        const uint32_t dg = kv[e] >> 21;
        if (dg > bstar) above_m |= 1ull << i;
        if (dg == bstar) {
          cand_m |= 1ull << i;
          ++mine;
        }
      }
    }
    uint32_t inc = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    uint32_t gb = 0;
    const uint32_t wsum = __shfl_sync(0xffffffffu, inc, 31);
    if (lane == 0) {
      gb = wsum ? atomicAdd(&s_nc, wsum) : 0u;
      gbase[g][warp] = gb;
    }
    uint32_t slot = __shfl_sync(0xffffffffu, gb, 0) + inc - mine;
#pragma unroll
    for (int e = 0; e < kLeanGroup; ++e) {
      const int i = g * kLeanGroup + e;
      if (i < nv && (kv[e] >> 21) == bstar) {
        if (slot < (uint32_t)kLeanCand) cand[slot] = kv[e];
        ++slot;
      }
    }
  }
  // f(i, key) over this thread's candidates in run order (keys from `cand`,
  // or from global memory past its capacity)
  auto for_my_cands = [&](auto&& f) {
    for (int g = 0; g < ngroups; ++g) {
      const uint32_t bits = (uint32_t)(cand_m >> (g * kLeanGroup)) & 0xffffu;
      uint32_t slot = group_slot(g, (uint32_t)__popc(bits));
      for (uint32_t mk = bits; mk; mk &= mk - 1) {
        const int i = g * kLeanGroup + __ffs(mk) - 1;
        f(i, slot < (uint32_t)kLeanCand ? cand[slot] : ordered_key(kp[i]));
        ++slot;
      }
    }
  };

  // ---------------------------------------------------------------- 3. tau
  csync();   // every CTA's candidates and count are in place
  if (tid < C) p_nc[tid] = *remote(&s_nc, tid);
  __syncthreads();
  uint32_t offs[kLeanMaxCluster + 1];
  offs[0] = 0;
#pragma unroll
  for (int c = 0; c < kLeanMaxCluster; ++c) offs[c + 1] = offs[c] + (c < C ? p_nc[c] : 0u);
  const uint32_t total = offs[kLeanMaxCluster];
  if (total != bucket && r == 0 && tid == 0) raise_error(a.err, kErrDevArg);   // cannot happen
  const bool fast = total <= (uint32_t)kLeanCand;
  uint32_t prefix = bstar << 21, pmask = 0xffe00000u;
  bool take_bucket = remaining == bucket;
  if (fast) {
    // gather every CTA's candidates; all of a thread's peer reads are issued
    // before its stores
    constexpr int kPer = kLeanCand / kLeanThreads;
    uint32_t v[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const uint32_t i = (uint32_t)(tid + u * kLeanThreads);
      int c = 0;
#pragma unroll
      for (int cc = 1; cc < kLeanMaxCluster; ++cc)
        if (cc < C && i >= offs[cc]) c = cc;
      v[u] = i < total ? remote(cand, c)[i - offs[c]] : 0u;
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u)
      if ((uint32_t)(tid + u * kLeanThreads) < total) work[tid + u * kLeanThreads] = v[u];
    __syncthreads();
  }
  if (!take_bucket) {
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {
      const int shift = pass == 0 ? 10 : 0;
      const uint32_t dmask = pass == 0 ? 2047u : 1023u;
      for (int i = tid; i < kBins; i += kLeanThreads) hist[i] = 0u;
      __syncthreads();
      uint32_t v[kLeanBinsPerThread];
      if (fast) {
        for (uint32_t i0w = (uint32_t)warp * 32; i0w < total; i0w += kLeanThreads) {   // warp-uniform trips
          const uint32_t i = i0w + lane;
          const uint32_t kv = i < total ? work[i] : 0u;
          hist_add(hist, (kv >> shift) & dmask, i < total && (kv & pmask) == prefix);
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kLeanBinsPerThread; ++i) v[i] = hist[kLeanBinsPerThread * tid + i];
      } else {
        for_my_cands([&](int, uint32_t kv) {
          if ((kv & pmask) == prefix) atomicAdd(&hist[(kv >> shift) & dmask], 1u);
        });
        csync();   // every CTA's histogram of this pass is complete
        merge_hist(hist, work);   // `work` holds no gathered keys on this path
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kLeanBinsPerThread; ++i) v[i] = work[kLeanBinsPerThread * tid + i];
        csync();   // every peer has read this CTA's histogram
      }
#pragma unroll
      for (int i = 0; i < kLeanBinsPerThread; ++i)
        if (kLeanBinsPerThread * tid + i > (int)dmask) v[i] = 0u;
      lean_crossing(v, remaining, wtot, res);
      if (!res[3]) {   // cannot happen: the candidates hold the rest of the budget
        if (r == 0 && tid == 0) raise_error(a.err, kErrDevArg);
        take_bucket = true;
        break;
      }
      prefix |= res[0] << shift;
      pmask |= dmask << shift;
      remaining -= res[1];
      if (remaining == res[2]) {
        take_bucket = true;
        break;
      }
    }
  }
  // Selection rule: take_bucket -> key >= prefix; otherwise tau = prefix is
  // the k-th key and the first `remaining` keys equal to it are taken.
  const uint32_t tau = prefix;

  // ---------------------------------------------------------------- 4. picks
  uint64_t sel_m = above_m, eq_m = 0;
  for_my_cands([&](int i, uint32_t kv) {
    if (take_bucket ? kv >= tau : kv > tau) sel_m |= 1ull << i;
    else if (!take_bucket && kv == tau) eq_m |= 1ull << i;
  });
  // (picks above tau) << 16 | (keys equal to tau): at most 16384 each per CTA
  const uint32_t mine = ((uint32_t)__popcll(sel_m) << 16) | (uint32_t)__popcll(eq_m);
  uint32_t inc = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wtot[warp] = inc;
  __syncthreads();
  uint32_t wbefore = 0, cta_tot = 0;
#pragma unroll
  for (int w = 0; w < kLeanWarps; ++w) {
    const uint32_t x = wtot[w];
    wbefore += w < warp ? x : 0u;
    cta_tot += x;
  }
  if (tid == 0) {
    s_cnt[0] = cta_tot >> 16;
    s_cnt[1] = cta_tot & 0xffffu;
  }
  csync();   // every CTA's counts are in place
  uint32_t gt_before = 0, eq_before = 0;
  for (int c = 0; c < r; ++c) {
    const uint32_t* pc = remote(s_cnt, c);
    gt_before += pc[0];
    eq_before += pc[1];
  }
  if (CL) cluster_arrive();   // this CTA's last read of a peer; the wait comes before exit
  const uint32_t before = wbefore + inc - mine;
  uint32_t gpos = gt_before + (before >> 16);
  uint32_t eqr = eq_before + (before & 0xffffu);
  for (uint64_t mk = sel_m | eq_m; mk; mk &= mk - 1) {
    const int i = __ffsll((long long)mk) - 1;
    const int j = j_lo + i0 + i;
    bool take;
    uint32_t pos;
    if ((sel_m >> i) & 1ull) {
      take = true;
      pos = gpos + min(eqr, remaining);
      ++gpos;
    } else {
      take = eqr < remaining;
      pos = gpos + eqr;
      ++eqr;
    }
    if (take) {
      if (pos < (uint32_t)kk) {
        out[pos] = j;
        hit(j);
      } else {
        raise_error(a.err, kErrDevArg);   // cannot happen: more picks than the budget
      }
    }
  }
  if (CL) cluster_wait();   // no peer reads this CTA's shared memory any more
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

int select_lean_cluster_size(int cap) {
  int C = 1;
  while (C < kLeanMaxCluster && (cap + C - 1) / C > 4096) C <<= 1;
  return C;
}

cudaError_t launch_select_lean(const SelectArgs& a0, cudaStream_t st) {
  SelectArgs a = a0;
  const int C = select_lean_cluster_size(a.cap);
  a.chunk = ((a.cap + C - 1) / C + 3) & ~3;
  a.run = ((a.chunk + kLeanThreads - 1) / kLeanThreads + 3) & ~3;
  // rows too long for 64 keys per thread in the largest cluster take the
  // cluster select that holds the keys in shared memory
  if (a.run > kLeanRunMax) return launch_select(a0, st);
  const dim3 grid(C, a.B * a.rows_per_seq, 1), block(kLeanThreads, 1, 1);
  if (C == 1) return launch_pdl(hill_select_lean_kernel<false>, grid, block, 0, st, 0, a);
  return launch_pdl(hill_select_lean_kernel<true>, grid, block, 0, st, C, a);
}

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
