// Token partition (Sec. 2.2, Eq. 3; App. B "dynamic token selection", Eq. 7)
// and the per-iteration active set (Sec. 2.2 modular rule, Sec. 2.3, Sec. 2.5
// caching window).
//
// Partition = a stable rank of the statistic.  Each fp32 value is mapped to an
// unsigned key whose integer order is the float order (-0 folded onto +0); the
// rank of a token is its position in the (key, token) order, which is the tie
// rule, and rank r maps to its group.  Three paths give the same groups:
//   N <= 12032   one launch ranks every token by counting the pairs before it;
//   N <= 49152   one block finds the pair at each group boundary (radix select
//                over keys held in shared memory) and compares every token with
//                those pairs;
//   larger N     a least-significant-digit radix sort of the (key, token)
//                pairs: four passes of 8 bits, each a per-tile histogram, one
//                exclusive scan of the (digit, tile) counts in digit-major
//                order, and a stable scatter (the pairs start in token order,
//                so equal keys stay in token order), then rank -> group.
//
// The active set needs no workspace: block b owns one chunk of tokens, counts
// the active tokens of all earlier chunks itself (an L2-resident re-read that
// is cheap at the token counts of a video DiT), then compacts its own chunk
// with warp ballots and a block scan.
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

// ------------------------------------------------ mid-size layers: select
//
// A token's group depends only on which group boundaries its rank passes:
// rank >= start[k] for k = 0 .. K-2 (group K-1 holds the lowest ranks), and
// rank >= b holds exactly when (key, token) >= the pair of rank b in the
// (key, token) order.  So for kRankMaxN < N <= kSelectMaxN one block loads the
// N keys into shared memory, finds the pair of each boundary rank (a radix
// select: four 8-bit digit passes, each a histogram of the keys that share
// the boundary's digits so far, then the boundary's position among the keys
// equal to its key, counted in token order) and compares every token with
// those pairs.  One launch instead of fourteen, and the same ranks as the
// stable sort.
constexpr int kSelectThreads = 1024;
constexpr int kSelectMaxN = 49152;                     // keys: 192 KB of shared memory
constexpr int kMaxBounds = kMaxGroups - 1;

__device__ __forceinline__ uint32_t order_key(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;                          // -0 ranks with +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);     // float order as uint order
}

__global__ void __launch_bounds__(kSelectThreads)
select_partition_kernel(const float *__restrict__ stat, int N, int K, GroupStarts gs,
                        int32_t *__restrict__ group_of, unsigned *err) {
  extern __shared__ uint4 skey4[];                      // the N keys, padded to whole uint4
  uint32_t *skey = reinterpret_cast<uint32_t *>(skey4);
  __shared__ uint32_t hist[kMaxBounds][256];
  __shared__ uint32_t pre[kMaxBounds];      // boundary key digits found so far
  __shared__ int below[kMaxBounds];         // keys ordered below that digit prefix
  __shared__ int slot[kMaxBounds];          // histogram of the boundary's prefix
  __shared__ uint32_t dpre[kMaxBounds];     // distinct prefixes, ascending
  __shared__ int nd;
  __shared__ unsigned long long thr[kMaxBounds];   // boundary pair (key << 32 | token)
  __shared__ int warp_tot[kSelectThreads / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int nb = K - 1;
  const int n4 = (N + 3) >> 2;
  // boundary j is searched when 0 < start[j] < N (rank 0 is passed by every
  // token, rank N by none)
  auto searched = [&](int j) { return gs.start[j] > 0 && gs.start[j] < N; };
  if ((reinterpret_cast<uintptr_t>(stat) & 15) == 0) {
    for (int i = threadIdx.x; i < n4; i += kSelectThreads) {
      float4 f;
      if (4 * i + 3 < N) {
        f = reinterpret_cast<const float4 *>(stat)[i];
      } else {
        f.x = stat[4 * i];
        f.y = 4 * i + 1 < N ? stat[4 * i + 1] : 0.f;
        f.z = 4 * i + 2 < N ? stat[4 * i + 2] : 0.f;
        f.w = 0.f;
      }
      if (!(isfinite(f.x) && isfinite(f.y) && isfinite(f.z) && isfinite(f.w)))
        set_error(err, kErrNonfinite);
      skey4[i] = make_uint4(order_key(f.x), order_key(f.y), order_key(f.z), order_key(f.w));
    }
  } else {
    for (int n = threadIdx.x; n < 4 * n4; n += kSelectThreads) {
      const float f = n < N ? stat[n] : 0.f;
      if (!isfinite(f)) set_error(err, kErrNonfinite);
      skey[n] = order_key(f);
    }
  }
  if (threadIdx.x == 0) {
    nd = 1;
    dpre[0] = 0u;
  }
  if (threadIdx.x < kMaxBounds) {
    pre[threadIdx.x] = 0u;
    below[threadIdx.x] = 0;
    slot[threadIdx.x] = 0;
  }
  __syncthreads();
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    const int n_hist = nd;
    for (int i = threadIdx.x; i < n_hist * 256; i += kSelectThreads) hist[i >> 8][i & 255] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n4; i += kSelectThreads) {
      const uint4 k4 = skey4[i];
      const uint32_t kk[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (4 * i + e >= N) break;                     // padding
        const uint32_t key = kk[e];
        const uint32_t hi = pass == 0 ? 0u : key >> (shift + 8);
        for (int q = 0; q < n_hist; ++q) {             // few distinct prefixes
          const uint32_t v = dpre[q];
          if (v >= hi) {
            if (v == hi) atomicAdd(&hist[q][(key >> shift) & 255u], 1u);
            break;
          }
        }
      }
    }
    __syncthreads();
    // warp j picks boundary j's digit: the bin where its rank falls
    if (w < nb && searched(w)) {
      const int target = gs.start[w] - below[w];       // rank among the prefix's keys
      const uint32_t *h = hist[slot[w]];
      int c[8], sum = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) { c[i] = (int)h[8 * lane + i]; sum += c[i]; }
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
        int pos = 0;
        while (pos < m && dpre[pos] < v) ++pos;
        if (pos == m || dpre[pos] != v) {
          for (int q = m; q > pos; --q) dpre[q] = dpre[q - 1];
          dpre[pos] = v;
          ++m;
        }
      }
      for (int j = 0; j < nb; ++j) {
        if (!searched(j)) continue;
        int pos = 0;
        while (dpre[pos] != pre[j]) ++pos;
        slot[j] = pos;
      }
      nd = m > 0 ? m : 1;
    }
    __syncthreads();
  }
  // Boundary j's pair: its key pre[j] and the token of rank start[j] - below[j]
  // among the tokens with that key in token order.  Thread t counts a
  // contiguous run of tokens; an odd run length keeps the threads of a warp
  // on different shared-memory banks.
  const int run = ((N + kSelectThreads - 1) / kSelectThreads) | 1;
  const int r0 = min(N, threadIdx.x * run), r1 = min(N, r0 + run);
  for (int j = 0; j < nb; ++j) {
    const int b = gs.start[j];
    if (!searched(j)) {                                // the same for every thread
      if (threadIdx.x == 0) thr[j] = b <= 0 ? 0ull : ~0ull;
      continue;
    }
    const uint32_t kj = pre[j];
    int eq = 0;
    for (int n = r0; n < r1; ++n) eq += skey[n] == kj;
    // exclusive block sum of eq
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
    const int need = b - below[j];
    if (need >= before && need < before + eq) {
      int seen = before;
      for (int n = r0; n < r1; ++n) {
        if (skey[n] != kj) continue;
        if (seen == need) {
          thr[j] = ((unsigned long long)kj << 32) | (unsigned)n;
          break;
        }
        ++seen;
      }
    }
    __syncthreads();                                   // warp_tot is reused
  }
  __syncthreads();
  for (int n = threadIdx.x; n < N; n += kSelectThreads) {
    const unsigned long long kn = ((unsigned long long)skey[n] << 32) | (unsigned)n;
    int passed = 0;
    for (int j = 0; j < nb; ++j) passed += kn >= thr[j];
    group_of[n] = K - 1 - passed;
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

}  // namespace
}  // namespace hsa

using namespace hsa;

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
  if (N <= kSelectMaxN) {
    static std::atomic<int> configured[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return HSA_ERR_CUDA;
    if (!configured[dev].load()) {
      if (cudaFuncSetAttribute(select_partition_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               kSelectMaxN * (int)sizeof(uint32_t)) != cudaSuccess)
        return HSA_ERR_CUDA;
      configured[dev].store(1);
    }
    count_launches(1);
    select_partition_kernel<<<1, kSelectThreads, (size_t)((N + 3) / 4) * sizeof(uint4), s>>>(
        stat, N, K, gs, group_of, err);
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
  // Chunks of whole 1024-token rounds, at most one block per SM: a layer of
  // up to 152 * 1024 tokens is compacted in one round per block.
  const int sms = sm_count();
  long long chunk = ((long long)N + sms - 1) / sms;
  chunk = ((chunk + kActThreads - 1) / kActThreads) * kActThreads;
  const int blocks = (int)(((long long)N + chunk - 1) / chunk);
  cudaStream_t s = (cudaStream_t)stream;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
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
// HSA_PARTITION_STATIC_MAX_TOKENS tokens; every GPU that loads the library
// holds it until the process exits.

namespace {

constexpr size_t kStaticScratchBytes = sort_layout(HSA_PARTITION_STATIC_MAX_TOKENS).total;
static_assert(kStaticScratchBytes % 256 == 0, "scratch array size");

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
