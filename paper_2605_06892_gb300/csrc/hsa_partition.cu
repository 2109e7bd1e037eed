// Token partition (Sec. 2.2, Eq. 3; App. B "dynamic token selection", Eq. 7)
// and the per-iteration active set (Sec. 2.2 modular rule, Sec. 2.3, Sec. 2.5
// caching window).
//
// Partition = a stable rank of the statistic.  Each fp32 value is mapped to an
// unsigned key whose integer order is the float order (-0 folded onto +0); the
// rank of a token is its position in the (key, token) order, which is the tie
// rule, and rank r maps to its group.  Three paths give the same groups:
//   N <= 12032    one launch ranks every token by counting the pairs before it;
//   N <= 360448   one launch of a cluster of 8 CTAs (keys spread over their
//                 shared memory) finds the pair at each group boundary by radix
//                 select and compares every token with those pairs;
//   larger N      a least-significant-digit radix sort of the (key, token)
//                 pairs: four passes of 8 bits, each a per-tile histogram, one
//                 exclusive scan of the (digit, tile) counts in digit-major
//                 order, and a stable scatter (the pairs start in token order,
//                 so equal keys stay in token order), then rank -> group.
//
// The active set needs no workspace.  Up to 2097152 tokens one cluster of 8
// CTAs marks and counts the active tokens of its ranges, exchanges the counts
// through distributed shared memory and compacts; above that, block b owns one
// chunk of tokens, counts the active tokens of all earlier chunks itself, then
// compacts its own chunk with warp ballots and a block scan.
#include <cooperative_groups.h>

#include <algorithm>
#include <atomic>

#include "hsa_internal.cuh"

namespace hsa {
namespace {

constexpr int kSortThreads = 256;
constexpr int kItems = 16;                              // per thread per tile
constexpr int kTile = kSortThreads * kItems;            // 4096 tokens
constexpr int kWarps = kSortThreads / 32;
constexpr int kWarpItems = kTile / kWarps;              // 512 consecutive tokens
constexpr int kMaxGroups = 32;

struct GroupStarts {
  int start[kMaxGroups];   // first rank of group k (ranks ascend with the statistic)
  int count[kMaxGroups];
};

constexpr size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }

struct SortLayout {
  size_t keys0, keys1, vals0, vals1, hist, total;
  int tiles;
};

// Workspace layout of the radix-sort path; constexpr so that the fixed
// scratch array of hsa_partition_static is sized by this same formula.
constexpr SortLayout sort_layout(int N) {
  SortLayout L{};
  L.tiles = (N + kTile - 1) / kTile;
  const size_t a = align256((size_t)N * 4);
  L.keys0 = 0;
  L.keys1 = a;
  L.vals0 = 2 * a;
  L.vals1 = 3 * a;
  L.hist = 4 * a;
  L.total = L.hist + align256((size_t)256 * L.tiles * 4);
  return L;
}

__global__ void __launch_bounds__(kSortThreads)
radix_key_kernel(const float *__restrict__ stat, int N, uint32_t *__restrict__ keys,
           int32_t *__restrict__ vals, unsigned *err) {
  for (int n = blockIdx.x * blockDim.x + threadIdx.x; n < N; n += gridDim.x * blockDim.x) {
    const float f = stat[n];
    uint32_t u = __float_as_uint(f);
    if (!isfinite(f)) set_error(err, kErrNonfinite);
    if (u == 0x80000000u) u = 0u;                          // -0 ranks with +0
    keys[n] = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // float order as uint order
    vals[n] = n;
  }
}

__global__ void __launch_bounds__(kSortThreads)
radix_hist_kernel(const uint32_t *__restrict__ keys, int N, int shift, uint32_t *__restrict__ hist,
            int tiles) {
  __shared__ uint32_t h[256];
  h[threadIdx.x] = 0;
  __syncthreads();
  const int base = blockIdx.x * kTile;
#pragma unroll
  for (int i = 0; i < kItems; ++i) {
    const int n = base + i * kSortThreads + threadIdx.x;
    if (n < N) atomicAdd(&h[(keys[n] >> shift) & 255u], 1u);
  }
  __syncthreads();
  hist[threadIdx.x * tiles + blockIdx.x] = h[threadIdx.x];
}

// Exclusive scan, in place, of the 256*tiles counts in digit-major order, by
// one block of 1024 threads, each owning a contiguous run.
__global__ void __launch_bounds__(1024) radix_scan_kernel(uint32_t *__restrict__ hist, int total) {
  __shared__ uint32_t warp_sum[32];
  const int per = (total + 1023) / 1024;
  const int b = threadIdx.x * per;
  const int e = min(total, b + per);
  uint32_t s = 0;
  for (int i = b; i < e; ++i) s += hist[i];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t incl = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_sum[w] = incl;
  __syncthreads();
  if (w == 0) {
    uint32_t v = warp_sum[lane], inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    warp_sum[lane] = inc - v;
  }
  __syncthreads();
  uint32_t run = warp_sum[w] + incl - s;
  for (int i = b; i < e; ++i) {
    const uint32_t c = hist[i];
    hist[i] = run;
    run += c;
  }
}

// Stable scatter of one tile.  Warp w owns tokens [w*512, w*512+512) of the
// tile and walks them 32 at a time in order; lanes holding the same digit find
// each other with __match_any_sync, so a token's rank among equal digits in
// the tile is (earlier warps' count) + (this warp's running count) + (earlier
// lanes of this step).
__global__ void __launch_bounds__(kSortThreads)
radix_scatter_kernel(const uint32_t *__restrict__ kin, const int32_t *__restrict__ vin,
               uint32_t *__restrict__ kout, int32_t *__restrict__ vout, int N, int shift,
               const uint32_t *__restrict__ offsets, int tiles) {
  __shared__ uint32_t cnt[kWarps][256];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int d = threadIdx.x; d < kWarps * 256; d += kSortThreads) (&cnt[0][0])[d] = 0;
  __syncthreads();
  const unsigned lt_mask = (1u << lane) - 1u;
  const int base = blockIdx.x * kTile + w * kWarpItems;
  uint32_t key[kItems];
  int32_t val[kItems];
  uint32_t local[kItems];
#pragma unroll
  for (int it = 0; it < kItems; ++it) {
    const int n = base + it * 32 + lane;
    const bool valid = n < N;
    key[it] = valid ? kin[n] : 0u;
    val[it] = valid ? vin[n] : 0;
    const uint32_t d = (key[it] >> shift) & 255u;
    const unsigned peers = __match_any_sync(0xffffffffu, valid ? d : 256u + lane);
    const uint32_t before = valid ? cnt[w][d] : 0u;
    local[it] = before + __popc(peers & lt_mask);
    __syncwarp();
    if (valid && lane == __ffs(peers) - 1) cnt[w][d] = before + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
  // exclusive prefix over warps, one digit per thread (blockDim == 256)
  {
    const int d = threadIdx.x;
    uint32_t run = offsets[d * tiles + blockIdx.x];
    for (int ww = 0; ww < kWarps; ++ww) {
      const uint32_t c = cnt[ww][d];
      cnt[ww][d] = run;
      run += c;
    }
  }
  __syncthreads();
#pragma unroll
  for (int it = 0; it < kItems; ++it) {
    const int n = base + it * 32 + lane;
    if (n < N) {
      const uint32_t d = (key[it] >> shift) & 255u;
      const uint32_t p = cnt[w][d] + local[it];
      kout[p] = key[it];
      vout[p] = val[it];
    }
  }
}

// ------------------------------------------------ small layers: rank by count
//
// For N <= kRankMaxN every block holds all N keys in shared memory, and a
// token's rank is the number of tokens ordered before it by (key, index):
// exactly the ranks of the stable sort, in one launch instead of fourteen.
// A block takes 32 tokens (its lanes) and splits the key range over its 8
// warps; the partial counts are summed in shared memory.  The keys are the
// same order-preserving transform as radix_key_kernel's.
constexpr int kRankThreads = 256;
constexpr int kRankTokens = 32;
// The keys (dynamic) and the partial counts (static) stay within the 48 KB a
// block gets without opting in to more shared memory.
constexpr int kRankMaxN = (48 * 1024 - (kRankThreads / 32) * kRankTokens * 4) / 4;   // 12032
static_assert(kRankMaxN * 4 + (kRankThreads / 32) * kRankTokens * 4 <= 48 * 1024,
              "rank partition shared memory");

__global__ void __launch_bounds__(kRankThreads)
rank_partition_kernel(const float *__restrict__ stat, int N, int K, GroupStarts gs,
                      int32_t *__restrict__ group_of, unsigned *err) {
  extern __shared__ uint32_t skey[];
  __shared__ int part[kRankThreads / 32][kRankTokens];
  for (int m = threadIdx.x; m < N; m += kRankThreads) {
    const float f = stat[m];
    uint32_t u = __float_as_uint(f);
    if (blockIdx.x == 0 && !isfinite(f)) set_error(err, kErrNonfinite);
    if (u == 0x80000000u) u = 0u;                          // -0 ranks with +0
    skey[m] = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // float order as uint order
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int n = blockIdx.x * kRankTokens + lane;
  const uint32_t kn = n < N ? skey[n] : 0u;
  const int per = (N + kRankThreads / 32 - 1) / (kRankThreads / 32);
  const int m0 = w * per, m1 = min(N, m0 + per);
  int r = 0;
#pragma unroll 4
  for (int m = m0; m < m1; ++m) {
    const uint32_t km = skey[m];                           // the same word for every lane
    r += (km < kn) + ((km == kn) & (m < n));
  }
  part[w][lane] = r;
  __syncthreads();
  if (w == 0 && n < N) {
    int rank = 0;
#pragma unroll
    for (int i = 0; i < kRankThreads / 32; ++i) rank += part[i][lane];
    int g = 0;
    for (int k = 0; k < K; ++k)
      if (rank >= gs.start[k] && rank < gs.start[k] + gs.count[k]) g = k;
    group_of[n] = g;
  }
}

// ------------------------------------------------ larger layers: select
//
// A token's group depends only on which group boundaries its rank passes:
// rank >= start[k] for k = 0 .. K-2 (group K-1 holds the lowest ranks), and
// rank >= b holds exactly when (key, token) >= the pair of rank b in the
// (key, token) order.  So it is enough to find the pair of each boundary rank
// (a radix select: four 8-bit digit passes, each a histogram of the keys that
// share the boundary's digits so far, then the boundary's position among the
// keys equal to its key, counted in token order) and to compare every token
// with those pairs: one launch instead of a sort's fourteen, and the same
// ranks as the stable sort.
constexpr int kMaxBounds = kMaxGroups - 1;

__device__ __forceinline__ uint32_t order_key(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;                          // -0 ranks with +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);     // float order as uint order
}

// The select runs on a thread-block cluster of
// kCsCtas CTAs (one launch).  CTA c holds the keys of tokens [c*chunk,
// (c+1)*chunk) in its shared memory; each digit pass builds one histogram per
// CTA, and every CTA then sums the cluster's histograms through distributed
// shared memory and takes the same digit decisions (identical integer work on
// identical data, so no broadcast is needed).  The boundary token is found in
// the CTA whose token range holds it (counts of equal keys are exchanged the
// same way, in CTA order = token order); that CTA writes the boundary pair into
// every CTA's shared memory.  Cluster barriers are hardware barriers: every
// thread of every CTA reaches each of them, so none can wait forever.
constexpr int kCsCtas = 8;
constexpr int kCsThreads = 1024;
constexpr int kCsMaxChunk = 44 * 1024;                 // keys per CTA: 176 KB
constexpr int kCsMaxN = kCsCtas * kCsMaxChunk;         // 360448 tokens

__global__ void __cluster_dims__(kCsCtas, 1, 1) __launch_bounds__(kCsThreads, 1)
cluster_select_kernel(const float *__restrict__ stat, int N, int chunk, int K, GroupStarts gs,
                      int32_t *__restrict__ group_of, unsigned *err) {
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  extern __shared__ uint4 ckey4[];                     // this CTA's keys, padded to uint4
  uint32_t *skey = reinterpret_cast<uint32_t *>(ckey4);
  __shared__ __align__(16) uint32_t hist[kMaxBounds * 256];   // [prefix slot][digit]
  __shared__ uint32_t pre[kMaxBounds];                 // boundary key digits found so far
  __shared__ int below[kMaxBounds];                    // keys ordered below that prefix
  __shared__ int slot[kMaxBounds];                     // histogram of the boundary's prefix
  __shared__ uint32_t dpre[kMaxBounds];                // distinct prefixes, ascending
  __shared__ int nd;
  __shared__ int eqc[kMaxBounds];                      // local keys equal to a boundary key
  __shared__ unsigned long long thr[kMaxBounds];       // boundary pair (key << 32 | token)
  __shared__ int warp_tot[kCsThreads / 32];
  const int cta = (int)cl.block_rank();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int nb = K - 1;
  const int lo = min(N, cta * chunk), hi = min(N, lo + chunk);
  const int n_loc = hi - lo;
  const int n4 = (n_loc + 3) >> 2;
  auto searched = [&](int j) { return gs.start[j] > 0 && gs.start[j] < N; };

  // keys of [lo, hi); chunk is a multiple of 4, so a 16-byte aligned stat
  // gives 16-byte aligned rows
  const bool vec = (reinterpret_cast<uintptr_t>(stat) & 15) == 0;
  for (int i = threadIdx.x; i < n4; i += kCsThreads) {
    float f[4];
    if (vec && 4 * i + 3 < n_loc) {
      const float4 v = __ldg(reinterpret_cast<const float4 *>(stat + lo) + i);
      f[0] = v.x, f[1] = v.y, f[2] = v.z, f[3] = v.w;
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) f[e] = 4 * i + e < n_loc ? __ldg(stat + lo + 4 * i + e) : 0.f;
    }
    if (!(isfinite(f[0]) && isfinite(f[1]) && isfinite(f[2]) && isfinite(f[3])))
      set_error(err, kErrNonfinite);
    ckey4[i] = make_uint4(order_key(f[0]), order_key(f[1]), order_key(f[2]), order_key(f[3]));
  }
  if (threadIdx.x == 0) {
    nd = 1;
    dpre[0] = 0u;
  }
  if (threadIdx.x < kMaxBounds) {
    pre[threadIdx.x] = 0u;
    below[threadIdx.x] = 0;
    slot[threadIdx.x] = 0;
    eqc[threadIdx.x] = 0;
  }
  __syncthreads();
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    const int n_hist = nd;
    for (int i = threadIdx.x; i < n_hist * 256; i += kCsThreads) hist[i] = 0u;
    __syncthreads();
    // Local histogram.  Every lane of a warp runs the same number of rounds,
    // so the warp can merge equal bins (__match_any_sync) and add each bin's
    // count once: in early passes most keys share a few bins.
    for (int b4 = 0; b4 < n4; b4 += kCsThreads) {
      const int i = b4 + threadIdx.x;
      uint4 k4 = make_uint4(0u, 0u, 0u, 0u);
      if (i < n4) k4 = ckey4[i];
      const uint32_t kk[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        uint32_t bin = 0xffffffffu;                    // no histogram
        if (i < n4 && 4 * i + e < n_loc) {
          const uint32_t key = kk[e];
          const uint32_t hp = pass == 0 ? 0u : key >> (shift + 8);
          for (int q = 0; q < n_hist; ++q) {           // few distinct prefixes
            const uint32_t v = dpre[q];
            if (v >= hp) {
              if (v == hp) bin = (uint32_t)q * 256u + ((key >> shift) & 255u);
              break;
            }
          }
        }
        const unsigned peers = __match_any_sync(0xffffffffu, bin);
        if (bin != 0xffffffffu && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
      }
    }
    cl.sync();                                         // every CTA's histogram is complete
    // warp j picks boundary j's digit from the cluster's summed histogram
    if (w < nb && searched(w)) {
      const int target = gs.start[w] - below[w];       // rank among the prefix's keys
      // bins 8*lane .. 8*lane+7 of every CTA's histogram: all 16 remote
      // 16-byte loads are issued before they are summed
      uint4 hv[kCsCtas][2];
#pragma unroll
      for (int r = 0; r < kCsCtas; ++r) {
        const uint4 *h = reinterpret_cast<const uint4 *>(cl.map_shared_rank(hist, r) +
                                                         slot[w] * 256 + 8 * lane);
        hv[r][0] = h[0];
        hv[r][1] = h[1];
      }
      int c[8], sum = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) c[i] = 0;
#pragma unroll
      for (int r = 0; r < kCsCtas; ++r) {
        c[0] += (int)hv[r][0].x; c[1] += (int)hv[r][0].y; c[2] += (int)hv[r][0].z;
        c[3] += (int)hv[r][0].w; c[4] += (int)hv[r][1].x; c[5] += (int)hv[r][1].y;
        c[6] += (int)hv[r][1].z; c[7] += (int)hv[r][1].w;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) sum += c[i];
      int incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      const int excl = incl - sum;
      if (target >= excl && target < incl) {           // exactly one lane
        int cum = excl, d = 8 * lane;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (target < cum + c[i]) { d = 8 * lane + i; break; }
          cum += c[i];
        }
        pre[w] = (pre[w] << 8) | (uint32_t)d;
        below[w] += cum;                               // keys below the longer prefix
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {                            // distinct prefixes, ascending
      int m = 0;
      for (int j = 0; j < nb; ++j) {
        if (!searched(j)) continue;
        const uint32_t v = pre[j];
        int p = 0;
        while (p < m && dpre[p] < v) ++p;
        if (p == m || dpre[p] != v) {
          for (int q = m; q > p; --q) dpre[q] = dpre[q - 1];
          dpre[p] = v;
          ++m;
        }
      }
      for (int j = 0; j < nb; ++j) {
        if (!searched(j)) continue;
        int p = 0;
        while (dpre[p] != pre[j]) ++p;
        slot[j] = p;
      }
      nd = m > 0 ? m : 1;
    }
    cl.sync();                // no CTA clears its histogram while another reads it
  }
  // Keys equal to each boundary key in this CTA: one sweep over a contiguous
  // run of tokens per thread (an odd run length spreads a warp's reads over
  // the shared-memory banks).
  const int run = ((n_loc + kCsThreads - 1) / kCsThreads) | 1;
  const int r0 = min(n_loc, threadIdx.x * run), r1 = min(n_loc, r0 + run);
  for (int j = 0; j < nb; ++j) {
    if (!searched(j)) continue;
    const uint32_t kj = pre[j];
    int eq = 0;
    for (int n = r0; n < r1; ++n) eq += skey[n] == kj;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) eq += __shfl_xor_sync(0xffffffffu, eq, o);
    if (lane == 0 && eq) atomicAdd(&eqc[j], eq);
  }
  for (int j = threadIdx.x; j < nb; j += kCsThreads)
    if (!searched(j)) thr[j] = gs.start[j] <= 0 ? 0ull : ~0ull;
  cl.sync();                                           // every CTA's eqc is complete
  for (int j = 0; j < nb; ++j) {
    if (!searched(j)) continue;                        // the same in every thread
    int before_cta = 0;                                // equal keys in earlier CTAs
    for (int r = 0; r < cta; ++r) before_cta += *cl.map_shared_rank(&eqc[j], r);
    const int need = gs.start[j] - below[j] - before_cta;
    if (need < 0 || need >= eqc[j]) continue;          // another CTA holds it
    const uint32_t kj = pre[j];
    int eq = 0;
    for (int n = r0; n < r1; ++n) eq += skey[n] == kj;
    int incl = eq;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) warp_tot[w] = incl;
    __syncthreads();
    if (w == 0) {
      const int x = warp_tot[lane];
      int inc = x;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
      }
      warp_tot[lane] = inc - x;
    }
    __syncthreads();
    const int before = warp_tot[w] + incl - eq;
    if (need >= before && need < before + eq) {
      int seen = before;
      for (int n = r0; n < r1; ++n) {
        if (skey[n] != kj) continue;
        if (seen == need) {
          const unsigned long long pair = ((unsigned long long)kj << 32) | (unsigned)(lo + n);
          for (int r = 0; r < kCsCtas; ++r) *cl.map_shared_rank(&thr[j], r) = pair;
          break;
        }
        ++seen;
      }
    }
    __syncthreads();                                   // warp_tot is reused
  }
  cl.sync();                  // the boundary pairs have reached every CTA
  for (int n = threadIdx.x; n < n_loc; n += kCsThreads) {
    const unsigned long long kn = ((unsigned long long)skey[n] << 32) | (unsigned)(lo + n);
    int passed = 0;
    for (int j = 0; j < nb; ++j) passed += kn >= thr[j];
    group_of[lo + n] = K - 1 - passed;
  }
}

__global__ void __launch_bounds__(kSortThreads)
group_assign_kernel(const int32_t *__restrict__ sorted_tokens, int N, int K, GroupStarts gs,
              int32_t *__restrict__ group_of) {
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < N; r += gridDim.x * blockDim.x) {
    int g = 0;
    for (int k = 0; k < K; ++k)
      if (r >= gs.start[k] && r < gs.start[k] + gs.count[k]) g = k;
    group_of[sorted_tokens[r]] = g;
  }
}

// ------------------------------------------------------------- active set

constexpr int kActThreads = 1024;

template <bool kVec>
__global__ void __launch_bounds__(kActThreads)
active_set_kernel(const int32_t *__restrict__ group_of, int N, int K, uint32_t mask, int chunk,
              int32_t *__restrict__ idx, int32_t *__restrict__ pos, unsigned *err) {
  __shared__ int warp_cnt[32];
  __shared__ int block_base;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int start = blockIdx.x * chunk;
  const int end = min(N, start + chunk);
  auto act = [&](int g) -> int {
    return (g >= 0 && g < K) ? (int)((mask >> g) & 1u) : 0;
  };
  // 1. active tokens before this chunk
  int c = 0;
  if (kVec) {
    const int4 *g4 = reinterpret_cast<const int4 *>(group_of);
    for (int i = threadIdx.x; i < start / 4; i += kActThreads) {
      const int4 v = __ldg(g4 + i);
      c += act(v.x) + act(v.y) + act(v.z) + act(v.w);
    }
  } else {
    for (int i = threadIdx.x; i < start; i += kActThreads) c += act(__ldg(group_of + i));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) warp_cnt[w] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int i = 0; i < kActThreads / 32; ++i) s += warp_cnt[i];
    block_base = s;
  }
  __syncthreads();
  int base = block_base;
  // 2. compact this chunk, 1024 tokens at a time
  for (int b0 = start; b0 < end; b0 += kActThreads) {
    const int n = b0 + threadIdx.x;
    int flag = 0;
    if (n < end) {
      const int g = group_of[n];
      if (g < 0 || g >= K) set_error(err, kErrIndex);
      flag = act(g);
    }
    const unsigned bal = __ballot_sync(0xffffffffu, flag);
    __syncthreads();                                   // warp_cnt reuse
    if (lane == 0) warp_cnt[w] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int i = 0; i < kActThreads / 32; ++i) {
      const int v = warp_cnt[i];
      before += (i < w) ? v : 0;
      total += v;
    }
    const int r = base + before + __popc(bal & ((1u << lane) - 1u));
    if (n < end) {
      if (flag) idx[r] = n;
      if (pos) pos[n] = flag ? r : -1;
    }
    base += total;
  }
}

// Active set of layers up to kAcMaxN tokens in one cluster of kCsCtas CTAs:
// CTA c owns tokens [c*chunk, (c+1)*chunk).  First pass: each CTA marks its
// active tokens (one bit each, in shared memory) and counts them.  The CTAs
// exchange their counts through distributed shared memory (CTA order is token
// order), so CTA c learns how many active tokens come before its range; the
// second pass compacts from the bits.  Group ids are read once, and no global
// scratch or inter-CTA spin is needed.
constexpr int kAcThreads = 1024;
constexpr int kAcMaxChunk = 256 * 1024;                // tokens per CTA: 32 KB of bits
constexpr int kAcMaxN = kCsCtas * kAcMaxChunk;         // 2097152 tokens

__global__ void __cluster_dims__(kCsCtas, 1, 1) __launch_bounds__(kAcThreads, 1)
active_set_cluster_kernel(const int32_t *__restrict__ group_of, int N, int K, uint32_t mask,
                          int chunk, int32_t *__restrict__ idx, int32_t *__restrict__ pos,
                          unsigned *err) {
  pdl_wait();
  pdl_trigger();
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  __shared__ uint32_t bits[kAcMaxChunk / 32];          // bit t: token lo + t is active
  __shared__ int warp_cnt[kAcThreads / 32];
  __shared__ int cta_count;
  __shared__ int cta_base;
  const int cta = (int)cl.block_rank();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int lo = min(N, cta * chunk), hi = min(N, lo + chunk);
  const int n_loc = hi - lo;
  const int rounds = (n_loc + kAcThreads - 1) / kAcThreads;
  auto act = [&](int g) -> int { return (g >= 0 && g < K) ? (int)((mask >> g) & 1u) : 0; };
  // pass 1: bits and count; four rounds' loads are issued before their ballots
  int c = 0;
  for (int r0 = 0; r0 < rounds; r0 += 4) {
    int g[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int t = (r0 + u) * kAcThreads + threadIdx.x;
      g[u] = t < n_loc ? __ldg(group_of + lo + t) : 0;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (r0 + u >= rounds) break;                     // uniform across the block
      const int t = (r0 + u) * kAcThreads + threadIdx.x;
      int flag = 0;
      if (t < n_loc) {
        if (g[u] < 0 || g[u] >= K) set_error(err, kErrIndex);
        flag = act(g[u]);
      }
      const unsigned bal = __ballot_sync(0xffffffffu, flag);
      if (lane == 0) {
        bits[(r0 + u) * (kAcThreads / 32) + w] = bal;
        c += __popc(bal);
      }
    }
  }
  if (lane == 0) warp_cnt[w] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int i = 0; i < kAcThreads / 32; ++i) s += warp_cnt[i];
    cta_count = s;
  }
  cl.sync();                                           // every CTA's count is known
  if (threadIdx.x == 0) {
    int b = 0;
    for (int r = 0; r < cta; ++r) b += *cl.map_shared_rank(&cta_count, r);
    cta_base = b;
  }
  cl.sync();                  // no CTA exits while another still reads its count
  // pass 2: compact from the bits, one round of kAcThreads tokens at a time
  int base = cta_base;
  for (int r = 0; r < rounds; ++r) {
    const int t = r * kAcThreads + threadIdx.x;
    const unsigned bal = bits[r * (kAcThreads / 32) + w];
    // active tokens of the round's earlier warps: lane i holds warp i's count,
    // an inclusive warp scan gives every prefix
    const int cnt = __popc(bits[r * (kAcThreads / 32) + lane]);
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    const int before = __shfl_sync(0xffffffffu, incl - cnt, w);
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    const int flag = (bal >> lane) & 1u;
    const int rank = base + before + __popc(bal & ((1u << lane) - 1u));
    if (t < n_loc) {
      if (flag) idx[rank] = lo + t;
      if (pos) pos[lo + t] = flag ? rank : -1;
    }
    base += total;
  }
}

}  // namespace
}  // namespace hsa

using namespace hsa;

namespace {

// Opts the cluster kernel in to its shared memory on the current device and
// checks that one cluster of kCsCtas such CTAs can be resident; otherwise the
// partition takes the radix-sort path.  Resolved once per device.
bool cluster_select_ready() {
  static std::atomic<int> state[64];            // 0 unknown, 1 ready, 2 unavailable
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  int st = state[dev].load();
  if (st == 0) {
    st = 2;
    const int smem = kCsMaxChunk * (int)sizeof(uint32_t);
    if (cudaFuncSetAttribute(cluster_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem) == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(kCsCtas);
      cfg.blockDim = dim3(kCsThreads);
      cfg.dynamicSmemBytes = smem;
      int clusters = 0;
      if (cudaOccupancyMaxActiveClusters(&clusters, cluster_select_kernel, &cfg) == cudaSuccess &&
          clusters >= 1)
        st = 1;
    }
    cudaGetLastError();                          // a refused query leaves no sticky error
    state[dev].store(st);
  }
  return st == 1;
}

// The same check for the active-set cluster (8 CTAs of 1024 threads, 33 KB of
// static shared memory each); otherwise the active set takes the per-block
// scheme.
bool cluster_active_ready() {
  static std::atomic<int> state[64];            // 0 unknown, 1 ready, 2 unavailable
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  int st = state[dev].load();
  if (st == 0) {
    st = 2;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kCsCtas);
    cfg.blockDim = dim3(kAcThreads);
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, active_set_cluster_kernel, &cfg) ==
            cudaSuccess &&
        clusters >= 1)
      st = 1;
    cudaGetLastError();                          // a refused query leaves no sticky error
    state[dev].store(st);
  }
  return st == 1;
}

}  // namespace

extern "C" size_t hsa_partition_workspace_bytes(int N) {
  if (N <= 0) return 0;
  return sort_layout(N).total;
}

extern "C" int hsa_partition(const float *stat, int N, int T, const int *budgets,
                             const int *counts, int K, int32_t *group_of, void *workspace,
                             size_t workspace_bytes, hsa_stream_t stream) {
  if (!budgets || !counts || K < 1) return HSA_ERR_INVALID_ARG;
  if (K > kMaxGroups) return HSA_ERR_UNSUPPORTED;
  const int st = hsa_check_budgets(T, budgets, counts, K, N);
  if (st != HSA_OK) return st;
  if (N == 0) return HSA_OK;
  if (!stat || !group_of) return HSA_ERR_INVALID_ARG;
  const SortLayout L = sort_layout(N);
  if (!workspace || workspace_bytes < L.total || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return HSA_ERR_WORKSPACE;
  char *ws = static_cast<char *>(workspace);
  uint32_t *keys[2] = {reinterpret_cast<uint32_t *>(ws + L.keys0),
                       reinterpret_cast<uint32_t *>(ws + L.keys1)};
  int32_t *vals[2] = {reinterpret_cast<int32_t *>(ws + L.vals0),
                      reinterpret_cast<int32_t *>(ws + L.vals1)};
  uint32_t *hist = reinterpret_cast<uint32_t *>(ws + L.hist);
  cudaStream_t s = (cudaStream_t)stream;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  GroupStarts gs{};
  int r = 0;
  for (int k = K - 1; k >= 0; --k) {
    gs.start[k] = r;
    gs.count[k] = counts[k];
    r += counts[k];
  }
  if (N <= kRankMaxN) {
    count_launches(1);
    rank_partition_kernel<<<(N + kRankTokens - 1) / kRankTokens, kRankThreads,
                            (size_t)N * sizeof(uint32_t), s>>>(stat, N, K, gs, group_of, err);
    return launch_status();
  }
  if (N <= kCsMaxN && cluster_select_ready()) {
    const int chunk = (((N + kCsCtas - 1) / kCsCtas) + 3) & ~3;   // keys per CTA, whole uint4
    count_launches(1);
    cluster_select_kernel<<<kCsCtas, kCsThreads, (size_t)chunk * sizeof(uint32_t), s>>>(
        stat, N, chunk, K, gs, group_of, err);
    return launch_status();
  }
  const int ew_blocks = (int)std::min<long long>((N + kSortThreads - 1) / kSortThreads,
                                                 (long long)sm_count() * 8);
  count_launches(1);
  radix_key_kernel<<<ew_blocks, kSortThreads, 0, s>>>(stat, N, keys[0], vals[0], err);
  for (int pass = 0; pass < 4; ++pass) {
    const int in = pass & 1, out = in ^ 1;
    count_launches(1);
    radix_hist_kernel<<<L.tiles, kSortThreads, 0, s>>>(keys[in], N, 8 * pass, hist, L.tiles);
    count_launches(1);
    radix_scan_kernel<<<1, 1024, 0, s>>>(hist, 256 * L.tiles);
    count_launches(1);
    radix_scatter_kernel<<<L.tiles, kSortThreads, 0, s>>>(keys[in], vals[in], keys[out], vals[out], N,
                                                     8 * pass, hist, L.tiles);
  }
  count_launches(1);
  group_assign_kernel<<<ew_blocks, kSortThreads, 0, s>>>(vals[0], N, K, gs, group_of);
  return launch_status();
}

extern "C" int hsa_partition_active(const int32_t *group_of, int N, int T, const int *budgets,
                                    int K, int iter, int window_pct, int32_t *idx,
                                    int32_t *pos, hsa_stream_t stream) {
  if (!budgets || K < 1) return HSA_ERR_INVALID_ARG;
  if (K > kMaxGroups) return HSA_ERR_UNSUPPORTED;
  const int st = hsa_check_budgets(T, budgets, nullptr, K, N);
  if (st != HSA_OK) return st;
  const int m = hsa_window_margin(T, window_pct);
  if (m < 0 || iter < 0 || iter >= T) return HSA_ERR_INVALID_ARG;
  if (N == 0) return HSA_OK;
  if (!group_of || !idx) return HSA_ERR_INVALID_ARG;
  uint32_t mask = 0;
  for (int k = 0; k < K; ++k) {
    const bool full = iter < m || iter > T - m - 1;
    if (full || iter % (T / budgets[k]) == 0) mask |= 1u << k;
  }
  cudaStream_t s = (cudaStream_t)stream;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  if (N <= kAcMaxN && cluster_active_ready()) {
    const int chunk = (N + kCsCtas - 1) / kCsCtas;
    count_launches(1);
    launch_pdl(active_set_cluster_kernel, dim3(kCsCtas), dim3(kAcThreads), 0, s, group_of, N, K,
               mask, chunk, idx, pos, err);
    return launch_status();
  }
  // Larger layers: chunks of whole 1024-token rounds, at most one block per
  // SM; block b counts the active tokens of the chunks before its own.
  const int sms = sm_count();
  long long chunk = ((long long)N + sms - 1) / sms;
  chunk = ((chunk + kActThreads - 1) / kActThreads) * kActThreads;
  const int blocks = (int)(((long long)N + chunk - 1) / chunk);
  count_launches(1);
  if (aligned16(group_of))
    active_set_kernel<true><<<blocks, kActThreads, 0, s>>>(group_of, N, K, mask, (int)chunk, idx,
                                                        pos, err);
  else
    active_set_kernel<false><<<blocks, kActThreads, 0, s>>>(group_of, N, K, mask, (int)chunk, idx,
                                                         pos, err);
  return launch_status();
}

// ------------------------------------------------------- token reordering
//
// Sec. 2.5: new position r holds old token order[r]; non-baseline tokens
// (group != 0) first, then the baseline group, each in token order.  Same
// workspace-free scheme as the active set: block b counts the non-baseline
// tokens before its chunk, then ranks its chunk with warp ballots.

template <bool kVec>
__global__ void __launch_bounds__(kActThreads)
reorder_kernel(const int32_t *__restrict__ group_of, int N, int M, int chunk,
               int32_t *__restrict__ order, int32_t *__restrict__ where,
               int32_t *__restrict__ group_new, unsigned *err) {
  __shared__ int warp_cnt[32];
  __shared__ int block_base;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int start = blockIdx.x * chunk;
  const int end = min(N, start + chunk);
  int c = 0;
  if (kVec) {
    const int4 *g4 = reinterpret_cast<const int4 *>(group_of);
    for (int i = threadIdx.x; i < start / 4; i += kActThreads) {
      const int4 v = __ldg(g4 + i);
      c += (v.x != 0) + (v.y != 0) + (v.z != 0) + (v.w != 0);
    }
  } else {
    for (int i = threadIdx.x; i < start; i += kActThreads) c += __ldg(group_of + i) != 0;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) warp_cnt[w] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int i = 0; i < kActThreads / 32; ++i) s += warp_cnt[i];
    block_base = s;
  }
  __syncthreads();
  int nb_base = block_base;             // non-baseline tokens before b0
  for (int b0 = start; b0 < end; b0 += kActThreads) {
    const int n = b0 + threadIdx.x;
    int g = 0, flag = 0;
    if (n < end) {
      g = group_of[n];
      flag = g != 0;
    }
    const unsigned bal = __ballot_sync(0xffffffffu, flag);
    __syncthreads();
    if (lane == 0) warp_cnt[w] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int i = 0; i < kActThreads / 32; ++i) {
      const int v = warp_cnt[i];
      before += (i < w) ? v : 0;
      total += v;
    }
    if (n < end) {
      const int nb_rank = nb_base + before + __popc(bal & ((1u << lane) - 1u));
      // baseline rank = tokens before n that are baseline
      const int r = flag ? nb_rank : M + (n - nb_rank);
      if ((flag && nb_rank < M) || (!flag && r < N)) {
        order[r] = n;
        if (where) where[n] = r;
        if (group_new) group_new[r] = g;
      } else {
        set_error(err, kErrIndex);
      }
    }
    nb_base += total;
  }
}

// ------------------------------------------------- allocation strategies
//
// Statistics whose ranking by hsa_partition gives the other token allocation
// strategies of App. B.  Uniform (U): stat[n] = top 24 bits of the 32-bit
// product (n+1) * 2654435769 (the golden ratio times 2^32), an integer exactly
// representable in fp32; each group then takes the tokens of one interval of
// the golden-ratio sequence, spaced by at most three distinct gaps.
// First-frame reservation (F): the first frame's tokens get FLT_MAX, so they
// rank into the baseline group.

__global__ void uniform_stat_kernel(float *__restrict__ stat, int N) {
  for (int n = blockIdx.x * blockDim.x + threadIdx.x; n < N; n += gridDim.x * blockDim.x)
    stat[n] = (float)(((uint32_t)(n + 1) * 2654435769u) >> 8);
}

__global__ void reserve_frame_kernel(float *__restrict__ stat, int frame_tokens) {
  for (int n = blockIdx.x * blockDim.x + threadIdx.x; n < frame_tokens;
       n += gridDim.x * blockDim.x)
    stat[n] = 3.40282347e38f;
}

// ----------------------------------------------- partition without allocation
//
// Variant of hsa_partition for callers that cannot hand the library a
// workspace: a plugin running inside a host framework that owns all device
// memory and exposes no allocator to it, or a latency-critical loop where
// cudaMalloc/cudaFree (which may synchronise the device) are not acceptable.
// Its scratch is a fixed file-scope device array sized for
// HSA_PARTITION_STATIC_MAX_TOKENS tokens (the radix sort of layers above
// kCsMaxN tokens works in it; smaller layers need no scratch); every GPU that
// loads the library holds it until the process exits.

namespace {

constexpr size_t kStaticScratchBytes = sort_layout(HSA_PARTITION_STATIC_MAX_TOKENS).total;
static_assert(kStaticScratchBytes % 256 == 0, "scratch array size");
static_assert(HSA_PARTITION_STATIC_MAX_TOKENS > kCsMaxN,
              "the fixed scratch must serve the sizes that need one");

// The host cannot use this symbol as a device address; the set-up below asks
// the runtime for the device address once per device.
static __device__ __align__(256) unsigned char g_partition_scratch[kStaticScratchBytes];

std::atomic<void *> g_scratch_ptr[64];

// Device address of g_partition_scratch on the current device (nullptr on
// failure).  The first call on a device resolves it.
void *static_scratch() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  void *p = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (!p) {
    if (cudaGetSymbolAddress(&p, g_partition_scratch) != cudaSuccess || !p) return nullptr;
    g_scratch_ptr[dev].store(p, std::memory_order_release);
  }
  return p;
}

}  // namespace

extern "C" int hsa_partition_static(const float *stat, int N, int T, const int *budgets,
                                    const int *counts, int K, int32_t *group_of,
                                    hsa_stream_t stream) {
  if (N > HSA_PARTITION_STATIC_MAX_TOKENS) return HSA_ERR_UNSUPPORTED;
  if (N >= 0 && hsa_partition_workspace_bytes(N) > kStaticScratchBytes) return HSA_ERR_UNSUPPORTED;
  void *scratch = static_scratch();
  if (!scratch) return HSA_ERR_CUDA;
  return hsa_partition(stat, N, T, budgets, counts, K, group_of, scratch, kStaticScratchBytes,
                       stream);
}

extern "C" int hsa_uniform_stat(float *stat, int N, hsa_stream_t stream) {
  if (N < 0) return HSA_ERR_INVALID_ARG;
  if (N == 0) return HSA_OK;
  if (!stat) return HSA_ERR_INVALID_ARG;
  const int blocks = (int)std::min<long long>((N + 255) / 256, (long long)sm_count() * 8);
  count_launches(1);
  uniform_stat_kernel<<<blocks, 256, 0, (cudaStream_t)stream>>>(stat, N);
  return launch_status();
}

extern "C" int hsa_reserve_first_frame(float *stat, int N, int frame_tokens,
                                       hsa_stream_t stream) {
  if (N < 0 || frame_tokens < 0 || frame_tokens > N) return HSA_ERR_INVALID_ARG;
  if (frame_tokens == 0) return HSA_OK;
  if (!stat) return HSA_ERR_INVALID_ARG;
  const int blocks = (int)std::min<long long>((frame_tokens + 255) / 256, (long long)sm_count() * 8);
  count_launches(1);
  reserve_frame_kernel<<<blocks, 256, 0, (cudaStream_t)stream>>>(stat, frame_tokens);
  return launch_status();
}

extern "C" int hsa_reorder_tokens(const int32_t *group_of, int N, int n_baseline,
                                  int32_t *order, int32_t *where, int32_t *group_new,
                                  hsa_stream_t stream) {
  if (N < 0 || n_baseline < 0 || n_baseline > N) return HSA_ERR_INVALID_ARG;
  if (N == 0) return HSA_OK;
  if (!group_of || !order) return HSA_ERR_INVALID_ARG;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const int sms = sm_count();
  long long chunk = ((long long)N + sms - 1) / sms;
  chunk = ((chunk + kActThreads - 1) / kActThreads) * kActThreads;
  if (chunk < 4096) chunk = 4096;
  const int blocks = (int)(((long long)N + chunk - 1) / chunk);
  const int M = N - n_baseline;
  cudaStream_t s = (cudaStream_t)stream;
  count_launches(1);
  if (aligned16(group_of))
    reorder_kernel<true><<<blocks, kActThreads, 0, s>>>(group_of, N, M, (int)chunk, order, where,
                                                         group_new, err);
  else
    reorder_kernel<false><<<blocks, kActThreads, 0, s>>>(group_of, N, M, (int)chunk, order, where,
                                                          group_new, err);
  return launch_status();
}
