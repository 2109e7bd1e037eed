// Active-query full-context attention (Sec. 2.3, step 3): the |A_i| active
// queries attend to all N rows of the layer's KV cache, O(|A_i| N) work.
//
// bf16 path: one CTA owns 256 active query rows (two 128-row Q tiles) of one
// head and streams every 128-key tile of that head's keys through shared
// memory.  The keys are the rows of up to two sources read in order: the KV
// cache, then (token reordering, Sec. 2.5) the fresh K/V of the baseline
// group, which is active at every iteration and so needs no cache.  Warp roles:
//   warp 0      TMA producer: K and V tiles of the head, 128-byte swizzled,
//               into a ring of shared-memory slots (rows >= N are zero-filled).
//   warp 1      tensor-core issuer (lane 0 issues, the warp walks the
//               schedule): S_t = Q_t K^T into TMEM and O_t += P_t V from TMEM
//               P and shared V, tcgen05.mma kind::f16.
//   warp 2      K/V watcher: waits for the K/V tiles to land, hands them to
//               the issuer at the P meetings, and gives ring slots back to
//               the producer.
//   warp 3      idle (it completes the first warpgroup).
//   warps 4-7   softmax of Q tile 0, warps 8-11 softmax of Q tile 1: each
//               thread owns one query row (its TMEM lane; a warp may only
//               reach the lane quarter warp%4), reads its S row,
//               keeps the running maximum and sum, writes P as bf16 back into
//               the S columns, and at the end normalises O and stores it.
//   all warps   load the 256 query rows once, by index, into swizzled smem.
// The two Q tiles ping-pong: while one softmax group works on its scores the
// tensor core runs the other tile's MMAs.  At D = 64 the TMEM also has room for
// a third S buffer, so each Q tile's next scores are computed while its softmax
// still works on the current ones.  The issuer waits only on hardware
// named barriers, two per key tile (P of a tile, with the K/V tiles the next
// MMAs read), where the other roles meet it; an mbarrier test on its path
// would idle the tensor core.  Units of odd waves walk their keys backwards
// (so they start on the tiles the previous wave of the head read last, still
// in L2), and the query and output rows, read and written once, are marked
// for early L2 eviction.  After the
// first key tile the probabilities are formed against the running reference
// maximum without computing the tile's maximum; only if a row sum would pass
// 2^32 is the tile redone with its exact maximum (and O rescaled in TMEM).
// The final division by the running sum makes the result exact whatever
// reference was used.
// Registers: the block launches at 168 per thread; the first warpgroup then
// gives registers back (setmaxnreg.dec to 96) and the two softmax warpgroups
// take them (setmaxnreg.inc to 200): 128*96 + 256*200 <= 384*168.
// Every mbarrier wait is bounded in time; on a timeout the kernel records
// HSA_ERR_TIMEOUT, stops loading K/V tiles and waiting for them, lets the MMA
// schedule run out over whatever the buffers hold, drains its own copies and
// MMAs, frees TMEM and returns.
//
// fp32 path: CUDA-core flash loop with K/V tiles in shared memory.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <cmath>

#include "hsa_internal.cuh"
#include "hsa_test.h"

namespace hsa {
namespace {

// ----------------------------------------------------------- PTX wrappers

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t *b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(b)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(b)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(b)) : "memory");
}

// Non-blocking test of phase `parity` (never suspends the thread).
__device__ __forceinline__ bool mbar_peek(uint64_t *b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(b)), "r"(parity)
      : "memory");
  return ok != 0;
}

// try_wait that lets the hardware suspend the thread for up to ~0.5 ms while
// the phase is incomplete, so waiting warps take no issue slots from the
// working ones.
__device__ __forceinline__ bool mbar_test_suspend(uint64_t *b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(b)), "r"(parity), "r"(500000u)
      : "memory");
  return ok != 0;
}

// About one second at the GB300 clock.
constexpr long long kWaitCycles = 2000000000LL;

// Bounded wait on phase `parity` of barrier b.  Gives up when the time runs
// out (records the timeout and raises the CTA's abort flag) or, if
// `honor_abort`, as soon as another role has raised the abort flag.  The
// first test is a non-blocking test_wait (a try_wait costs far more even on a
// completed phase); between tests the thread suspends in try_wait.
__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity, volatile int *abort_flag,
                                          unsigned *err, bool honor_abort = true) {
  if (mbar_peek(b, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_test_suspend(b, parity)) return true;
    if (honor_abort && *abort_flag) return false;
    if (clock64() - t0 > kWaitCycles) {
      set_error(err, kErrTimeout);
      *abort_flag = 1;
      return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_addr(dst)),
      "l"(map), "r"(smem_addr(bar)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor (tcgen05), 128-byte swizzle.  For a
// K-major operand only the stride between 8-row groups (sbo) matters; for an
// MN-major operand lbo is the stride between 64-element column chunks.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor of kind::f16 with bf16 A/B, fp32 accumulator.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, int b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)b_mn_major << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t id,
                                       uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(id), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t id,
                                       uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d),
      "r"(a_tmem), "l"(b), "r"(id), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *b) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_addr(b))
      : "memory");
}

// 32 consecutive TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}

// Packed fp32 pairs (sm_100 family): two lanes of work per instruction.
__device__ __forceinline__ uint64_t pack2(uint32_t lo, uint32_t hi) {
  return (uint64_t)lo | ((uint64_t)hi << 32);
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float lo_f(uint64_t v) { return __uint_as_float((uint32_t)v); }
__device__ __forceinline__ float hi_f(uint64_t v) { return __uint_as_float((uint32_t)(v >> 32)); }

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void named_barrier_sync(int id, int threads) {
  asm volatile("barrier.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}


__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// ------------------------------------------------------ tcgen05 kernel

constexpr int kBM = 128;         // query rows per Q tile (= TMEM lanes)
constexpr int kQT = 2;           // Q tiles per CTA
constexpr int kBN = 128;         // keys per K/V tile
constexpr int kTcThreads = 384;  // 12 warps = 3 warpgroups
constexpr int kLaunchRegs = 168;         // registers per thread at launch
constexpr int kRegsLow = 96;             // producer / MMA warpgroup
constexpr int kRegsHigh = 200;           // softmax warpgroups
static_assert(128 * kRegsLow + 256 * kRegsHigh <= kTcThreads * kLaunchRegs,
              "register split exceeds the launch allocation");
constexpr int kTmemCols = 512;
// Named barriers (hardware, not in shared memory): 1 = teardown of the whole
// CTA; kBarK0 = the first K tile has landed (the K/V watcher and the issuing
// warp meet once); kBarP0 + t = P of Q tile t is in TMEM, for key tile j (its
// 128 softmax threads, the issuing warp and the K/V watcher meet; at the
// meeting for P_0(j) the watcher has seen V_j and K_(j+1) land).  Every party
// syncs (a rendezvous, never a lone arrive) once per hand-off in the same
// order, so no party can run a whole round ahead and the barrier instances
// always pair up, also after a failed wait.
constexpr int kBarTeardown = 1;
constexpr int kBarP0 = 2;
constexpr int kBarK0 = 4;
constexpr int kMeetP = kBM + 64;   // threads at a P meeting

template <int D>
struct TcCfg {
  static constexpr int kTileBytes = kBM * D * 2;            // one Q, K or V tile
  static constexpr int kChunks = D / 64;                    // 128-byte column chunks
  static constexpr int kStages = D == 128 ? 5 : 8;          // K/V ring slots
  static constexpr int kSmem = (kQT + kStages) * kTileBytes + 1024;
  // D = 64: three S buffers in TMEM (384 columns) and O_t at 384 + 64t, so that
  // each Q tile's next S is computed while its softmax still works on the
  // current one.  D = 128: S_t in columns 128t, O_t at 256 + 128t.
  static constexpr bool kThreeS = D == 64;
  static constexpr int kOCol0 = kThreeS ? 384 : 256;        // O_t at kOCol0 + t*D
  static constexpr int kSBars = kThreeS ? 2 : 1;            // S barriers per Q tile
};

struct TcArgs {
  const __nv_bfloat16 *q;
  const int32_t *q_idx;
  __nv_bfloat16 *out;
  unsigned *err;
  int n_active, N, H, q_rows, n_kv_tiles;
  int rows1, rows2, tiles1;   // key sources: rows1 cache rows, then rows2 rows
  float scale_log2;
  int inject_stall;   // test hook (hsa_test.h): 1 = the first V tile is never loaded
  // Work split.  CTA b < n_whole owns unit b (head b / n_qblocks, query block
  // b % n_qblocks) over all key tiles.  Every later CTA owns one of `pieces`
  // key ranges of a tail unit and writes its unnormalised O, running maximum
  // and sum to ws_o / ws_ml for the combine kernel.
  int n_qblocks, n_whole, pieces;
  int wave;           // CTAs resident at once (one per SM): the length of a wave
  float *ws_o;        // [piece CTA][kQT*kBM rows][D] fp32
  float *ws_ml;       // [piece CTA][kQT*kBM rows][2] fp32: m (log2 units), l
};

// Key-tile range [j0, j1) and unit of CTA b.
struct CtaWork {
  int head, row0, j0, j1, piece;   // piece = -1 for a whole unit
};

__host__ __device__ inline CtaWork cta_work(int b, int n_qblocks, int n_whole, int pieces,
                                            int n_kv_tiles) {
  CtaWork w;
  int unit;
  if (b < n_whole) {
    unit = b;
    w.j0 = 0;
    w.j1 = n_kv_tiles;
    w.piece = -1;
  } else {
    const int pi = b - n_whole;
    unit = n_whole + pi / pieces;
    const int k = pi % pieces;
    w.j0 = (int)((long long)n_kv_tiles * k / pieces);
    w.j1 = (int)((long long)n_kv_tiles * (k + 1) / pieces);
    w.piece = pi;
  }
  w.head = unit / n_qblocks;
  w.row0 = (unit % n_qblocks) * (kBM * kQT);
  return w;
}

// P = 2^(s*scale*log2e - m) for this thread's 128 scores, as bf16 pairs
// written over the first 64 S columns (all scores are in registers, so P may
// overwrite S); returns the row sum of the fp32 values.
__device__ __forceinline__ float exp_store_tile(uint32_t tS, const uint32_t (&r)[128],
                                                float sl2, float m) {
  // x = s*scale*log2e - m for a pair of scores in one packed FMA; p = 2^x.
  const uint64_t scale2 = pack2(__float_as_uint(sl2), __float_as_uint(sl2));
  const uint64_t negm2 = pack2(__float_as_uint(-m), __float_as_uint(-m));
  uint64_t ps[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint32_t pk[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const uint64_t x = fma2(pack2(r[64 * h + 2 * i], r[64 * h + 2 * i + 1]), scale2, negm2);
      const float p0 = fast_exp2(lo_f(x));
      const float p1 = fast_exp2(hi_f(x));
      ps[i & 3] = add2(ps[i & 3], pack2(__float_as_uint(p0), __float_as_uint(p1)));
      pk[i] = pack_bf16(p0, p1);
    }
    tmem_st32(tS + 32 * h, pk);
  }
  const uint64_t s01 = add2(ps[0], ps[1]), s23 = add2(ps[2], ps[3]);
  const uint64_t st = add2(s01, s23);
  return lo_f(st) + hi_f(st);
}

// One 128-key tile of this thread's row.  softmax(s) V = sum 2^(c s - m) v /
// sum 2^(c s - m) holds for any reference m as long as nothing overflows, and
// m_run (a maximum of earlier tiles) never exceeds the row's true maximum, so
// after the first tile P is formed against m_run without looking at this
// tile's maximum (fast path).  If a row's sum then exceeds 2^32 (or is not
// finite) the warp redoes the tile on the exact path: the row maximum of the
// scores (still in registers) becomes the new reference, O (in TMEM) and the
// running sum take the factor 2^(m_old - m_new), and P is formed again.  O is
// rescaled only once o_idle() has returned true: the previous O += P V has
// then completed (false: a wait failed, O is left alone).  The first tile
// always takes the exact path.  kTail masks keys >= valid (the last, ragged
// tile); full tiles take no per-key test.
template <int D, bool kTail, typename OIdle>
__device__ __forceinline__ void softmax_tile(uint32_t tS, uint32_t tO, int valid, bool first,
                                             float sl2, float &m_run, float &l_run,
                                             OIdle &&o_idle) {
  // The second half of S is read while the first half is masked.
  uint32_t r[128];
  tmem_ld32(tS, *reinterpret_cast<uint32_t(*)[32]>(&r[0]));
  tmem_ld32(tS + 32, *reinterpret_cast<uint32_t(*)[32]>(&r[32]));
  tmem_wait_ld();
  tmem_ld32(tS + 64, *reinterpret_cast<uint32_t(*)[32]>(&r[64]));
  tmem_ld32(tS + 96, *reinterpret_cast<uint32_t(*)[32]>(&r[96]));
  if (kTail) {
#pragma unroll
    for (int i = 0; i < 64; ++i)
      if (i >= valid) r[i] = __float_as_uint(-INFINITY);
  }
  tmem_wait_ld();
  if (kTail) {
#pragma unroll
    for (int i = 64; i < 128; ++i)
      if (i >= valid) r[i] = __float_as_uint(-INFINITY);
  }
  if (!first) {
    const float rs = exp_store_tile(tS, r, sl2, m_run);
    const bool bad = !(rs <= 4294967296.0f);
    if (!__any_sync(0xffffffffu, bad)) {
      l_run += rs;
      return;
    }
    tmem_wait_st();   // the exact path rewrites the same P columns
  }
  // Exact path.  pm[p] = maximum of scores 16p .. 16p+15: seven
  // three-input steps cover 16p+1 .. 16p+14, the last step adds 16p+15.
  float pm[8];
#pragma unroll
  for (int p = 0; p < 8; ++p) {
    float m = __uint_as_float(r[16 * p]);
#pragma unroll
    for (int i = 1; i < 15; i += 2)
      m = max3f(m, __uint_as_float(r[16 * p + i]), __uint_as_float(r[16 * p + i + 1]));
    pm[p] = fmaxf(m, __uint_as_float(r[16 * p + 15]));
  }
  const float mx = fmaxf(max3f(pm[0], pm[1], pm[2]),
                         fmaxf(max3f(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7])));
  const float m_new = fmaxf(m_run, mx * sl2);
  const float alpha = (!first && m_new > m_run) ? fast_exp2(m_run - m_new) : 1.f;
  l_run = first ? 0.f : l_run * alpha;
  m_run = m_new;
  if (!first && __any_sync(0xffffffffu, alpha != 1.f) && o_idle()) {
#pragma unroll
    for (int c = 0; c < D / 16; ++c) {
      uint32_t o[16];
      tmem_ld16(tO + 16 * c, o);
      tmem_wait_ld();
#pragma unroll
      for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
      tmem_st16(tO + 16 * c, o);
    }
  }
  l_run += exp_store_tile(tS, r, sl2, m_run);
}

template <int D>
__global__ void __launch_bounds__(kTcThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
               const __grid_constant__ CUtensorMap tm_k2, const __grid_constant__ CUtensorMap tm_v2,
               const TcArgs a) {
  // Launched with programmatic dependent launch: wait for the kernels before
  // this one in the stream (the KV scatter writes the keys read below).  The
  // blocks of the last wave let the next kernel start launching onto the SMs
  // they free; no block of this grid is still waiting for an SM by then.
  pdl_wait();
  if (blockIdx.x + (unsigned)a.wave >= gridDim.x) pdl_trigger();
  using C = TcCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                            ~(uintptr_t)1023);
  uint8_t *sQ = sm;
  uint8_t *sKV = sm + kQT * C::kTileBytes;
  __shared__ __align__(8) uint64_t bar_full[C::kStages], bar_empty[C::kStages];
  __shared__ __align__(8) uint64_t bar_s[kQT * C::kSBars], bar_o;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const CtaWork wk = cta_work(blockIdx.x, a.n_qblocks, a.n_whole, a.pieces, a.n_kv_tiles);
  const int h = wk.head;
  const int row0 = wk.row0;
  const int j0 = wk.j0;
  const int nT = wk.j1 - wk.j0;        // key tiles of this CTA (local index j = 0..nT-1)
  // Key order of the unit.  Whole units of odd "waves" (blocks [k*sms,
  // (k+1)*sms) for odd k) walk the keys backwards, so they start on the key
  // tiles the previous wave's units of the same head read last, which are
  // still in L2.  The order of the keys does not change the result (up to
  // rounding): the softmax is accumulated online.
  const bool rev = wk.piece < 0 && ((blockIdx.x / a.wave) & 1);
  auto key_tile = [&](int j) { return rev ? wk.j1 - 1 - j : j0 + j; };

  // K or V tile L/2 of this unit's key range (L even: K, odd: V) into its
  // ring slot, completing on bar_full.  Issued by thread 0, the producer.
  auto load_kv = [&](int L) {
    const int slot = L % C::kStages;
    mbar_expect_tx(&bar_full[slot], C::kTileBytes);
    const int jg = key_tile(L >> 1);                // global key tile
    const bool second = jg >= a.tiles1;
    const CUtensorMap *map = second ? ((L & 1) ? &tm_v2 : &tm_k2) : ((L & 1) ? &tm_v : &tm_k);
    const int y = (second ? jg - a.tiles1 : jg) * kBN;
    uint8_t *dst = sKV + slot * C::kTileBytes;
#pragma unroll
    for (int c = 0; c < C::kChunks; ++c)
      tma_load_2d(dst + c * (kBN * 128), map, &bar_full[slot], h * D + c * 64, y);
  };
  const int withheld = a.inject_stall == 1 ? 1 : -1;   // test hook: V of tile 0 never loads
  const int n_pre = min(C::kStages, 2 * nT);          // loads issued before the Q tile
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_empty[s], 1);
    }
    for (int t = 0; t < kQT * C::kSBars; ++t) mbar_init(&bar_s[t], 1);
    mbar_init(&bar_o, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // The first ring's worth of K/V tiles load while the CTA loads its query
    // rows below.
    for (int L = 0; L < n_pre; ++L)
      if (L != withheld) load_kv(L);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(&tmem_base_sh)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }

  // ---- query rows, by index, into the two swizzled Q tiles (all threads)
  // Each thread first reads the indices of all its rows, then issues all its
  // 16-byte loads, then stores them: two dependent round trips to memory in
  // all rather than two per vector.
  {
    constexpr int kVecPerRow = D / 8;                        // 16-byte vectors per row
    constexpr int kVecs = kBM * kQT * kVecPerRow;
    constexpr int kPer = (kVecs + kTcThreads - 1) / kTcThreads;
    const size_t row_stride = (size_t)a.H * D;
    int src[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int i = threadIdx.x + u * kTcThreads;
      const int grow = row0 + i / kVecPerRow;
      src[u] = -1;
      if (i < kVecs && grow < a.n_active) src[u] = a.q_idx ? __ldg(a.q_idx + grow) : grow;
    }
    uint4 v[kPer];
    uint64_t pol;                       // the query rows are read once: evict first
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int i = threadIdx.x + u * kTcThreads;
      v[u] = make_uint4(0u, 0u, 0u, 0u);
      if (src[u] >= 0 && src[u] < a.q_rows) {
        const uint4 *p = reinterpret_cast<const uint4 *>(a.q + (size_t)src[u] * row_stride +
                                                         (size_t)h * D) + i % kVecPerRow;
        asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
                     : "=r"(v[u].x), "=r"(v[u].y), "=r"(v[u].z), "=r"(v[u].w)
                     : "l"(p), "l"(pol));
      }
      else if (i < kVecs && row0 + i / kVecPerRow < a.n_active && i % kVecPerRow == 0)
        set_error(a.err, kErrIndex);
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int i = threadIdx.x + u * kTcThreads;
      if (i < kVecs) {
        const int row = i / kVecPerRow, c = i % kVecPerRow;
        const int t = row / kBM, rr = row % kBM;
        uint8_t *dst = sQ + t * C::kTileBytes + (c >> 3) * (kBM * 128) + rr * 128 +
                       (((c & 7) ^ (rr & 7)) << 4);
        *reinterpret_cast<uint4 *>(dst) = v[u];
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = tmem_base_sh;

  // The warpgroups' code paths never rejoin below: each ends with its own
  // teardown on named barrier 1, so each path is compiled for its own
  // register budget.

  if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsLow));
    if (warp == 0) {
      // ------------------------------------------------ TMA producer
      if (lane == 0) {
        int issued = n_pre;
        for (int L = n_pre; L < 2 * nT; ++L) {
          const int slot = L % C::kStages, use = L / C::kStages;
          if (use > 0 && !mbar_wait(&bar_empty[slot], (use - 1) & 1, &abort_flag, a.err)) break;
          if (L == withheld) continue;
          load_kv(L);
          issued = L + 1;
        }
        // Drain: every issued copy has landed before the CTA may exit.  A
        // slot is only refilled once its previous tile was consumed, so the
        // copies in flight are among the last kStages issued.
        for (int L = issued > C::kStages ? issued - C::kStages : 0; L < issued; ++L)
          if (L != withheld)
            mbar_wait(&bar_full[L % C::kStages], (L / C::kStages) & 1, &abort_flag, a.err, false);
      }
      __syncwarp();
      } else if (warp == 1) {
      // ------------------------------------------------ MMA issuer
      // The whole warp walks the schedule so that it can take part in the
      // named-barrier hand-offs; lane 0 issues the MMAs and commits.  The
      // tensor pipe takes a new MMA only about when it starts it, so every
      // pause of the issuing thread between MMAs idles the tensor core.  An
      // mbarrier test on this path costs about a hundred clocks while an S
      // group's operand reads fill the shared-memory bandwidth; a named
      // barrier whose other parties have already arrived costs far less.
      // So the issuer waits on named barriers only, two per key tile:
      // kBarP0 + t, where the softmax of Q tile t has stored P and the K/V
      // watcher has seen the tiles the next MMAs read land (once, before the
      // loop, kBarK0 for the first K tile).  Every party meets it exactly once
      // per hand-off whatever happens, so each sync completes.  The issuer
      // reads no shared memory on this path either: a load waits behind the
      // MMAs' operand reads (a probe measured about 165 clocks of tensor time
      // per load of the abort flag), so after an abort it keeps issuing, over
      // whatever the ring and the TMEM hold, until the schedule ends; the
      // kernel then returns with the error recorded.
      const bool leader = lane == 0;
      constexpr uint32_t kIdS = idesc_bf16(kBM, kBN, 0);
      constexpr uint32_t kIdO = idesc_bf16(kBM, D, 1);
      const uint32_t q_base = smem_addr(sQ);
      const uint32_t kv_base = smem_addr(sKV);
      // Descriptors differ only in their start-address field (bits 0-13,
      // address >> 4), so each MMA adds a constant to a base descriptor.
      const uint64_t dq0 = sdesc(q_base, 16, 1024);
      const uint64_t dk0 = sdesc(kv_base, 16, 1024);
      const uint64_t dv0 = sdesc(kv_base, kBN * 128, 1024);
      constexpr uint32_t kTile16 = C::kTileBytes >> 4;
      // S_t = Q_t K^T: K = D in steps of 16 (32 bytes inside a 128-byte chunk).
      auto issue_s = [&](int t, int L) {
        const uint64_t dq = dq0 + t * kTile16;
        const uint64_t dk = dk0 + (L % C::kStages) * kTile16;
        const uint32_t ts = tmem + 128 * t;
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint32_t off = ((k >> 2) * (kBM * 128) + (k & 3) * 32) >> 4;
          mma_ss(ts, dq + off, dk + off, kIdS, k > 0);
        }
      };
      // O_t += P_t V: P in TMEM (bf16 pairs in the S_t columns), V MN-major.
      auto issue_o = [&](int t, int L, bool acc) {
        const uint64_t dv = dv0 + (L % C::kStages) * kTile16;
        const uint32_t to = tmem + C::kOCol0 + D * t, tp = tmem + 128 * t;
#pragma unroll
        for (int k = 0; k < kBN / 16; ++k)
          mma_ts(to, tp + 8 * k, dv + ((k * 2048) >> 4), kIdO, (acc || k > 0) ? 1u : 0u);
      };
      auto p_ready = [&](int t) {
        named_barrier_sync(kBarP0 + t, kMeetP);
        fence_after();
      };
      if constexpr (!C::kThreeS) {
        named_barrier_sync(kBarK0, 64);             // K_0 has landed
        fence_after();
        if (leader) {
          issue_s(0, 0);
          mma_commit(&bar_s[0]);
          issue_s(1, 0);
          mma_commit(&bar_s[1]);
        }
        for (int j = 0; j < nT; ++j) {
          const int Lv = 2 * j + 1, Lk = 2 * j + 2;
          const bool more = j + 1 < nT;
          p_ready(0);                               // P_0(j); V_j and K_(j+1) landed
          const bool go = leader;
          if (go) {
            issue_o(0, Lv, j > 0);
            if (more) {
              issue_s(0, Lk);
              mma_commit(&bar_s[0]);
            }
          }
          p_ready(1);
          if (go) {
            issue_o(1, Lv, j > 0);
            if (more) {
              issue_s(1, Lk);
              mma_commit(&bar_s[1]);
            }
          }
        }
      } else {
        // Three S buffers.  The s-th S MMA in issue order (S_t(j) is number
        // 2j + t) writes buffer s mod 3, so S_0(j+2) and S_1(j+1) reuse the
        // buffers whose P the O MMAs just issued have read (the tensor core
        // runs its MMAs in order).  Each Q tile's S is computed one or two key
        // tiles ahead of its softmax.  S_t(j) completes on bar_s[2t + j%2];
        // alternating two barriers per Q tile means no waiter can be overtaken
        // by two completions of the barrier it waits on.
        auto issue_s3 = [&](int t, int j) {
          const uint64_t dq = dq0 + t * kTile16;
          const uint64_t dk = dk0 + ((2 * j) % C::kStages) * kTile16;
          const uint32_t ts = tmem + 128 * ((2 * j + t) % 3);
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint32_t off = ((k >> 2) * (kBM * 128) + (k & 3) * 32) >> 4;
            mma_ss(ts, dq + off, dk + off, kIdS, k > 0);
          }
          mma_commit(&bar_s[2 * t + (j & 1)]);
        };
        auto issue_o3 = [&](int t, int j) {
          const uint64_t dv = dv0 + ((2 * j + 1) % C::kStages) * kTile16;
          const uint32_t to = tmem + C::kOCol0 + D * t, tp = tmem + 128 * ((2 * j + t) % 3);
#pragma unroll
          for (int k = 0; k < kBN / 16; ++k)
            mma_ts(to, tp + 8 * k, dv + ((k * 2048) >> 4), kIdO, (j > 0 || k > 0) ? 1u : 0u);
        };
        named_barrier_sync(kBarK0, 64);             // K_0 (and K_1) have landed
        fence_after();
        if (leader) {
          issue_s3(0, 0);
          issue_s3(1, 0);
          if (nT > 1) issue_s3(0, 1);
        }
        for (int j = 0; j < nT; ++j) {
          p_ready(0);                               // P_0(j); V_j and K_(j+1) landed
          const bool go = leader;
          if (go) {
            issue_o3(0, j);
            if (j + 1 < nT) issue_s3(1, j + 1);
          }
          p_ready(1);                               // P_1(j); K_(j+2) landed
          if (go) {
            issue_o3(1, j);
            if (j + 2 < nT)
              issue_s3(0, j + 2);
            else if (j + 2 == nT)
              mma_commit(&bar_s[(j + 2) & 1]);      // O_1(j) done, for the last tile's rescale
          }
        }
      }
      if (leader) {
        // Completes once every MMA issued above has finished (also on
        // abort), so TMEM is quiet before it is freed.
        mma_commit(&bar_o);
        mbar_wait(&bar_o, 0, &abort_flag, a.err, false);
      }
      __syncwarp();
    } else if (warp == 2) {
      // ------------------------------------------------ K/V watcher
      // Waits (bounded) for the K/V tiles to land and hands them to the
      // issuer at the P meetings: V_j and K_(j+1) before P_0(j) (K_0 alone,
      // before the loop).  It also gives ring slots back to the producer, so
      // the issuer commits nothing for them: once S_1 of key tile j has
      // completed (the tensor core runs its MMAs in order), K_j and V_(j-1)
      // have been read by every MMA that uses them.  It waits for that between
      // the meetings for P_0(j) and P_1(j); S_1 of key tile j+1 is issued only
      // after the meeting for P_1(j), so the phase it waits for is never
      // overtaken.  It meets the issuer at every meeting even after a failed
      // wait, so the issuer never waits forever, and after a failure it gives
      // nothing back, so no slot is refilled while a copy into it may still be
      // in flight.
      bool live = true;
      auto landed = [&](int L) {
        if (live)
          live = __all_sync(0xffffffffu, mbar_wait(&bar_full[L % C::kStages],
                                                   (L / C::kStages) & 1, &abort_flag, a.err));
      };
      auto give_back = [&](int L) {
        if (lane == 0) mbar_arrive(&bar_empty[L % C::kStages]);
      };
      if constexpr (!C::kThreeS) {
        landed(0);
        named_barrier_sync(kBarK0, 64);
        for (int j = 0; j < nT; ++j) {
          landed(2 * j + 1);                       // V_j
          if (j + 1 < nT) landed(2 * j + 2);       // K_(j+1)
          named_barrier_sync(kBarP0, kMeetP);
          if (live) {
            live = __all_sync(0xffffffffu, mbar_wait(&bar_s[1], j & 1, &abort_flag, a.err));
            if (live) {
              give_back(2 * j);                    // K_j
              if (j > 0) give_back(2 * j - 1);     // V_(j-1)
            }
          }
          named_barrier_sync(kBarP0 + 1, kMeetP);
        }
      } else {
        // Three S buffers: K_(j+2) is needed at the meeting for P_1(j) (the
        // issuer then issues S_0(j+2)).  S_0(j+1) is issued after O_1(j-1), so
        // once it has completed K_j and V_(j-1) have been read by every MMA
        // that uses them; it waits for that between the meetings for P_0(j) and
        // P_1(j).  The next completion of the same barrier, S_0(j+3), is issued
        // only after the meeting for P_1(j+1).
        landed(0);                                 // K_0
        if (nT > 1) landed(2);                     // K_1
        named_barrier_sync(kBarK0, 64);
        for (int j = 0; j < nT; ++j) {
          landed(2 * j + 1);                       // V_j
          named_barrier_sync(kBarP0, kMeetP);
          if (live && j + 1 < nT) {
            live = __all_sync(0xffffffffu, mbar_wait(&bar_s[(j + 1) & 1], ((j + 1) >> 1) & 1,
                                                     &abort_flag, a.err));
            if (live) {
              give_back(2 * j);                    // K_j
              if (j > 0) give_back(2 * j - 1);     // V_(j-1)
            }
          }
          if (j + 2 < nT) landed(2 * j + 4);       // K_(j+2)
          named_barrier_sync(kBarP0 + 1, kMeetP);
        }
      }
    }
    fence_before();
    named_barrier_sync(kBarTeardown, kTcThreads);
    if (warp == 1) {
      fence_after();
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                   "r"(kTmemCols)
                   : "memory");
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsHigh));
    // ------------------------------------------------ softmax / epilogue
    const int t = (warp - 4) >> 2;
    const int wq = warp & 3;                       // TMEM lane quarter of this warp
    const int r = wq * 32 + lane;                  // row within the Q tile
    const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
    const uint32_t tS = tmem + lane_off + 128 * t;
    const uint32_t tO = tmem + lane_off + C::kOCol0 + D * t;
    const float sl2 = a.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    // `ok` stays warp-uniform (the tile code votes across the warp).  After
    // a failed wait the warp does no more work but still meets the issuer for
    // every P, so the issuing warp's named-barrier syncs all complete.
    // Meeting (rather than arriving) costs nothing: S_t(j+1) is issued only
    // after the issuer has passed this meeting for P_t(j).
    bool ok = true;
    for (int j = 0; j < nT; ++j) {
      if constexpr (!C::kThreeS) {
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bar_s[t], j & 1, &abort_flag, a.err));
      } else {
        if (ok)
          ok = __all_sync(0xffffffffu, mbar_wait(&bar_s[2 * t + (j & 1)], (j >> 1) & 1,
                                                 &abort_flag, a.err));
      }
      if (ok) {
        fence_after();
        const int jg = key_tile(j);                // keys of this tile that exist
        const int valid = jg < a.tiles1 ? a.rows1 - jg * kBN : a.rows2 - (jg - a.tiles1) * kBN;
        // three S buffers (D = 64): S_t(j) is the (2j + t)-th S MMA
        const uint32_t tSj = C::kThreeS ? tmem + lane_off + 128 * ((2 * j + t) % 3) : tS;
        // O_t(j-1) has completed once an MMA issued after it has.  With two
        // S buffers that is S_t(j), complete already.  With three, S_t(j) is
        // issued before O_t(j-1): wait for S_1(j) (Q tile 0) or S_0(j+1) (Q
        // tile 1; at the last key tile the issuer commits that barrier with
        // no MMA).  Neither barrier can complete again before this warp's
        // next meeting.  Needed only on the exact path's rescale, so rare.
        auto o_idle = [&]() -> bool {
          if constexpr (!C::kThreeS) return true;
          uint64_t *b = t == 0 ? &bar_s[2 + (j & 1)] : &bar_s[(j + 1) & 1];
          const uint32_t par = t == 0 ? (j >> 1) & 1 : ((j + 1) >> 1) & 1;
          const bool idle = __all_sync(0xffffffffu, mbar_wait(b, par, &abort_flag, a.err));
          fence_after();
          return idle;
        };
        if (valid >= kBN)
          softmax_tile<D, false>(tSj, tO, valid, j == 0, sl2, m_run, l_run, o_idle);
        else
          softmax_tile<D, true>(tSj, tO, valid, j == 0, sl2, m_run, l_run, o_idle);
        tmem_wait_st();
      }
      fence_before();
      named_barrier_sync(kBarP0 + t, kMeetP);
    }
    if (ok && wk.piece >= 0 && mbar_wait(&bar_o, 0, &abort_flag, a.err)) {
      // Piece of a split unit: unnormalised O, maximum and sum, for the combine.
      fence_after();
      const int prow = t * kBM + r;
      float *po = a.ws_o + ((size_t)wk.piece * (kQT * kBM) + prow) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + 32 * c, o);
        tmem_wait_ld();
        float4 *d4 = reinterpret_cast<float4 *>(po + 32 * c);
#pragma unroll
        for (int v = 0; v < 8; ++v)
          d4[v] = make_float4(__uint_as_float(o[4 * v]), __uint_as_float(o[4 * v + 1]),
                              __uint_as_float(o[4 * v + 2]), __uint_as_float(o[4 * v + 3]));
      }
      reinterpret_cast<float2 *>(a.ws_ml)[(size_t)wk.piece * (kQT * kBM) + prow] =
          make_float2(m_run, l_run);
    } else if (ok && mbar_wait(&bar_o, 0, &abort_flag, a.err)) {
      fence_after();
      const int grow = row0 + t * kBM + r;
      const float inv = 1.f / l_run;
      __nv_bfloat16 *dst = a.out + ((size_t)grow * a.H + h) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + 32 * c, o);
        tmem_wait_ld();
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i)
          pk[i] = pack_bf16(__uint_as_float(o[2 * i]) * inv, __uint_as_float(o[2 * i + 1]) * inv);
        if (grow < a.n_active) {
          uint64_t pol;                 // the output rows are written once: evict first
          asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
#pragma unroll
          for (int v = 0; v < 4; ++v)
            asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1,%2,%3,%4}, %5;" ::"l"(
                             dst + 32 * c + 8 * v),
                         "r"(pk[4 * v]), "r"(pk[4 * v + 1]), "r"(pk[4 * v + 2]),
                         "r"(pk[4 * v + 3]), "l"(pol)
                         : "memory");
        }
      }
    }
    fence_before();
    named_barrier_sync(kBarTeardown, kTcThreads);
  }
}

// ------------------------------------------------------ split-unit combine
//
// One warp per (tail unit, row): merge the unit's key-range pieces,
// O = sum_p 2^(m_p - M) O_p / sum_p 2^(m_p - M) l_p with M = max_p m_p, and
// store the bf16 row.  Lanes stride over D, so every access is coalesced.
template <int D>
__global__ void __launch_bounds__(256)
attn_combine_kernel(const float *__restrict__ ws_o, const float *__restrict__ ws_ml, int n_tail,
                    int n_whole, int pieces, int n_qblocks, int n_active, int H,
                    __nv_bfloat16 *__restrict__ out) {
  pdl_wait();
  pdl_trigger();
  constexpr int kRows = kQT * kBM;
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  const int u = wid / kRows, row = wid % kRows;
  if (u >= n_tail) return;
  const int unit = n_whole + u;
  const int head = unit / n_qblocks;
  const int grow = (unit % n_qblocks) * kRows + row;
  if (grow >= n_active) return;
  const float2 *ml = reinterpret_cast<const float2 *>(ws_ml);
  float M = -INFINITY;
  for (int p = 0; p < pieces; ++p) M = fmaxf(M, ml[((size_t)u * pieces + p) * kRows + row].x);
  float L = 0.f, acc[D / 32];
#pragma unroll
  for (int i = 0; i < D / 32; ++i) acc[i] = 0.f;
  for (int p = 0; p < pieces; ++p) {
    const size_t pr = ((size_t)u * pieces + p) * kRows + row;
    const float2 v = ml[pr];
    const float w = exp2f(v.x - M);
    L = fmaf(w, v.y, L);
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc[i] = fmaf(w, ws_o[pr * D + lane + 32 * i], acc[i]);
  }
  const float inv = 1.f / L;
  __nv_bfloat16 *dst = out + ((size_t)grow * H + head) * D;
#pragma unroll
  for (int i = 0; i < D / 32; ++i) dst[lane + 32 * i] = __float2bfloat16_rn(acc[i] * inv);
}

// ------------------------------------------------------ fp32 CUDA-core kernel

constexpr int kF32Threads = 128;
constexpr int kF32Keys = 32;
constexpr int kF32Dims = 8;      // dimensions per thread

// TPQ = D/8 threads cooperate on one query (8 dimensions each, so that small
// layers still give the GPU enough threads); thread slice s owns dimensions
// s, s+TPQ, s+2*TPQ, ... so that the slices of one query hit distinct banks.
template <int D>
__global__ void __launch_bounds__(kF32Threads)
attn_f32_kernel(const float *__restrict__ q, const int32_t *__restrict__ q_idx,
                const float *__restrict__ kc, const float *__restrict__ vc, int rows1,
                const float *__restrict__ kb, const float *__restrict__ vb,
                float *__restrict__ out, int n_active, int N, int H, int q_rows, float scale,
                unsigned *err) {
  constexpr int TPQ = D / kF32Dims;
  constexpr int QPB = kF32Threads / TPQ;
  __shared__ float sK[kF32Keys][D];
  __shared__ float sV[kF32Keys][D];
  const int h = blockIdx.y;
  const int ql = threadIdx.x / TPQ, sl = threadIdx.x % TPQ;
  const int j = blockIdx.x * QPB + ql;
  const bool active = j < n_active;
  float qv[kF32Dims], o[kF32Dims];
  bool row_ok = false;
  if (active) {
    const int src = q_idx ? q_idx[j] : j;
    row_ok = src >= 0 && src < q_rows;
    if (!row_ok && sl == 0) set_error(err, kErrIndex);
#pragma unroll
    for (int i = 0; i < kF32Dims; ++i)
      qv[i] = row_ok ? q[((size_t)src * H + h) * D + sl + TPQ * i] : 0.f;
  } else {
#pragma unroll
    for (int i = 0; i < kF32Dims; ++i) qv[i] = 0.f;
  }
#pragma unroll
  for (int i = 0; i < kF32Dims; ++i) o[i] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int n0 = 0; n0 < N; n0 += kF32Keys) {
    __syncthreads();
    for (int e = threadIdx.x; e < kF32Keys * D / 4; e += kF32Threads) {
      const int kk = e / (D / 4), d4 = e % (D / 4);
      float4 kv = make_float4(0.f, 0.f, 0.f, 0.f), vv = kv;
      const int key = n0 + kk;
      if (key < N) {
        const bool first = key < rows1;
        const size_t off = ((size_t)(first ? key : key - rows1) * H + h) * D;
        kv = reinterpret_cast<const float4 *>((first ? kc : kb) + off)[d4];
        vv = reinterpret_cast<const float4 *>((first ? vc : vb) + off)[d4];
      }
      reinterpret_cast<float4 *>(&sK[kk][0])[d4] = kv;
      reinterpret_cast<float4 *>(&sV[kk][0])[d4] = vv;
    }
    __syncthreads();
    float sc[kF32Keys];
    float tmax = -INFINITY;
#pragma unroll
    for (int kk = 0; kk < kF32Keys; ++kk) {
      float dot = 0.f;
#pragma unroll
      for (int i = 0; i < kF32Dims; ++i) dot = fmaf(qv[i], sK[kk][sl + TPQ * i], dot);
#pragma unroll
      for (int o2 = 1; o2 < TPQ; o2 <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o2);
      sc[kk] = (n0 + kk < N) ? dot * scale : -INFINITY;
      tmax = fmaxf(tmax, sc[kk]);
    }
    const float m_new = fmaxf(m, tmax);
    const float corr = expf(m - m_new);
    l *= corr;
#pragma unroll
    for (int i = 0; i < kF32Dims; ++i) o[i] *= corr;
#pragma unroll
    for (int kk = 0; kk < kF32Keys; ++kk) {
      const float p = expf(sc[kk] - m_new);
      l += p;
#pragma unroll
      for (int i = 0; i < kF32Dims; ++i) o[i] = fmaf(p, sV[kk][sl + TPQ * i], o[i]);
    }
    m = m_new;
  }
  if (active) {
    const float inv = 1.f / l;
#pragma unroll
    for (int i = 0; i < kF32Dims; ++i) out[((size_t)j * H + h) * D + sl + TPQ * i] = o[i] * inv;
  }
}

// -------------------------------------------------------------- host side

std::atomic<int> g_inject_stall{0};

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::atomic<PFN_cuTensorMapEncodeTiled_v12000> fn{nullptr};
  PFN_cuTensorMapEncodeTiled_v12000 f = fn.load();
  if (!f) {
    cudaDriverEntryPointQueryResult q;
    void *p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    f = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    fn.store(f);
  }
  return f;
}

// 2-D map over a [N, H*D] bf16 cache: boxes of 64 columns x 128 rows,
// 128-byte swizzle, rows past N read as zero.
bool make_kv_map(CUtensorMap *map, const void *base, int N, int H, int D) {
  auto enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)H * D, (cuuint64_t)N};
  const cuuint64_t strides[1] = {(cuuint64_t)H * D * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)kBN};
  const cuuint32_t estride[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
             box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Bytes of split-unit workspace for head dimension D: at most two pieces per
// SM, kQT*kBM rows each, D fp32 of O plus (m, l).
size_t split_workspace_bytes(int D) {
  return 2 * (size_t)sm_count() * (kQT * kBM) * ((size_t)D * 4 + 8) + 512;
}

// Pieces per tail unit.  The rem units of the last wave, cut into P key
// ranges each, occupy ceil(rem*P / sms) waves of 1/P unit: minimise that,
// plus 0.005 unit per piece for its extra prologue, partial write and merge,
// with at most two waves of pieces and at least one key tile per piece.
int tail_pieces(int rem, int sms, int n_kv_tiles) {
  if (rem <= 0) return 1;
  int best = 1;
  double best_cost = 1.0 + 0.005;
  const int pmax = std::min(n_kv_tiles, (2 * sms) / rem);
  for (int p = 2; p <= pmax; ++p) {
    const double cost = (double)((rem * p + sms - 1) / sms) / p + 0.005 * p;
    if (cost < best_cost - 1e-12) {
      best_cost = cost;
      best = p;
    }
  }
  return best;
}

template <int D>
int launch_tc(const void *q, const int32_t *q_idx, int n_active, const void *k_cache,
              const void *v_cache, int rows1, const void *k_base, const void *v_base, int rows2,
              int H, float scale, void *out, void *ws, size_t ws_bytes, cudaStream_t stream,
              unsigned *err) {
  const int N = rows1 + rows2;
  using C = TcCfg<D>;
  static std::atomic<int> configured[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return HSA_ERR_CUDA;
  if (!configured[dev].load()) {
    // The register hand-over inside the kernel assumes exactly kLaunchRegs
    // registers per thread at launch; any other count could leave the
    // softmax warps waiting for registers, so refuse to launch.
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, attn_tc_kernel<D>) != cudaSuccess) return HSA_ERR_CUDA;
    if (fa.numRegs != kLaunchRegs || fa.maxThreadsPerBlock < kTcThreads) return HSA_ERR_UNSUPPORTED;
    if (cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmem) != cudaSuccess)
      return HSA_ERR_CUDA;
    configured[dev].store(1);
  }
  CUtensorMap mk, mv, mk2, mv2;
  if (rows1 > 0 && (!make_kv_map(&mk, k_cache, rows1, H, D) ||
                    !make_kv_map(&mv, v_cache, rows1, H, D)))
    return HSA_ERR_CUDA;
  if (rows2 > 0 && (!make_kv_map(&mk2, k_base, rows2, H, D) ||
                    !make_kv_map(&mv2, v_base, rows2, H, D)))
    return HSA_ERR_CUDA;
  if (rows1 == 0) mk = mk2, mv = mv2;   // unused source: any valid map
  if (rows2 == 0) mk2 = mk, mv2 = mv;
  TcArgs a;
  a.q = static_cast<const __nv_bfloat16 *>(q);
  a.q_idx = q_idx;
  a.out = static_cast<__nv_bfloat16 *>(out);
  a.err = err;
  a.n_active = n_active;
  a.N = N;
  a.H = H;
  a.q_rows = q_idx ? N : n_active;
  a.rows1 = rows1;
  a.rows2 = rows2;
  a.tiles1 = (rows1 + kBN - 1) / kBN;
  a.n_kv_tiles = a.tiles1 + (rows2 + kBN - 1) / kBN;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.inject_stall = g_inject_stall.load(std::memory_order_relaxed);
  // Work plan: one CTA per SM at a time, so U units take ceil(U / sms) waves.
  // With a workspace, the rem = U mod sms units of the last wave are split
  // along the keys into `pieces` ranges (tail_pieces) that shorten that wave,
  // then combined.
  a.n_qblocks = (n_active + kQT * kBM - 1) / (kQT * kBM);
  const long long units = (long long)a.n_qblocks * H;
  if (units > 0x7fffffffLL) return HSA_ERR_UNSUPPORTED;
  const int sms = sm_count();
  a.wave = sms;
  const int rem = (int)(units % sms);
  int pieces = 1;
  if (ws && rem > 0) {
    pieces = tail_pieces(rem, sms, a.n_kv_tiles);
    const size_t need = (size_t)rem * pieces * (kQT * kBM) * ((size_t)D * 4 + 8);
    if (pieces < 2 || need > ws_bytes || (reinterpret_cast<uintptr_t>(ws) & 15)) pieces = 1;
  }
  a.pieces = pieces;
  a.n_whole = pieces > 1 ? (int)(units - rem) : (int)units;
  a.ws_o = pieces > 1 ? static_cast<float *>(ws) : nullptr;
  a.ws_ml = pieces > 1 ? a.ws_o + (size_t)rem * pieces * (kQT * kBM) * D : nullptr;
  const long long grid = (long long)a.n_whole + (pieces > 1 ? (long long)rem * pieces : 0);
  count_launches(1);
  launch_pdl(attn_tc_kernel<D>, dim3((unsigned)grid), dim3(kTcThreads), C::kSmem, stream, mk, mv,
             mk2, mv2, a);
  if (cudaGetLastError() != cudaSuccess) return HSA_ERR_CUDA;
  if (pieces > 1) {
    const long long warps = (long long)rem * (kQT * kBM);
    count_launches(1);
    launch_pdl(attn_combine_kernel<D>, dim3((unsigned)((warps * 32 + 255) / 256)), dim3(256), 0,
               stream, (const float *)a.ws_o, (const float *)a.ws_ml, (int)rem, a.n_whole,
               pieces, a.n_qblocks, n_active, H, a.out);
  }
  return launch_status();
}

template <int D>
int launch_f32(const void *q, const int32_t *q_idx, int n_active, const void *k_cache,
               const void *v_cache, int rows1, const void *k_base, const void *v_base, int rows2,
               int H, float scale, void *out, cudaStream_t stream, unsigned *err) {
  constexpr int QPB = kF32Threads / (D / kF32Dims);
  const int N = rows1 + rows2;
  const dim3 grid((n_active + QPB - 1) / QPB, H);
  count_launches(1);
  attn_f32_kernel<D><<<grid, kF32Threads, 0, stream>>>(
      static_cast<const float *>(q), q_idx, static_cast<const float *>(k_cache),
      static_cast<const float *>(v_cache), rows1, static_cast<const float *>(k_base),
      static_cast<const float *>(v_base), static_cast<float *>(out), n_active, N, H,
      q_idx ? N : n_active, scale, err);
  return launch_status();
}

}  // namespace
}  // namespace hsa

using namespace hsa;

extern "C" size_t hsa_active_attention_workspace_bytes(int n_active, int N, int H, int D,
                                                      hsa_dtype dtype) {
  if (dtype != HSA_BF16 || (D != 64 && D != 128) || n_active <= 0 || N <= 0 || H <= 0) return 0;
  return split_workspace_bytes(D);
}

namespace {

int attention_two_sources(const void *q, const int32_t *q_idx, int n_active, const void *k_cache,
                          const void *v_cache, int rows1, const void *k_base,
                          const void *v_base, int rows2, int H, int D, float scale, void *out,
                          hsa_dtype dtype, void *workspace, size_t workspace_bytes,
                          hsa_stream_t stream) {
  const long long N = (long long)rows1 + rows2;
  if (n_active < 0 || rows1 < 0 || rows2 < 0 || N < 1 || N > 0x7fffffffLL || H < 1)
    return HSA_ERR_INVALID_ARG;
  if (dtype != HSA_BF16 && dtype != HSA_F32) return HSA_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return HSA_ERR_UNSUPPORTED;
  if ((long long)H * D > (1LL << 24)) return HSA_ERR_UNSUPPORTED;
  if (!q_idx && n_active > N) return HSA_ERR_INVALID_ARG;
  if (n_active == 0) return HSA_OK;
  if (!q || !out || (rows1 > 0 && (!k_cache || !v_cache)) || (rows2 > 0 && (!k_base || !v_base)))
    return HSA_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || (rows1 > 0 && (!aligned16(k_cache) || !aligned16(v_cache))) ||
      (rows2 > 0 && (!aligned16(k_base) || !aligned16(v_base))))
    return HSA_ERR_INVALID_ARG;
  if (!(scale > 0.f) || !std::isfinite(scale)) scale = 1.f / std::sqrt((float)D);
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  if (H > 65535) return HSA_ERR_UNSUPPORTED;
  if (dtype == HSA_BF16)
    return D == 128 ? launch_tc<128>(q, q_idx, n_active, k_cache, v_cache, rows1, k_base, v_base,
                                     rows2, H, scale, out, workspace, workspace_bytes, s, err)
                    : launch_tc<64>(q, q_idx, n_active, k_cache, v_cache, rows1, k_base, v_base,
                                    rows2, H, scale, out, workspace, workspace_bytes, s, err);
  return D == 128 ? launch_f32<128>(q, q_idx, n_active, k_cache, v_cache, rows1, k_base, v_base,
                                    rows2, H, scale, out, s, err)
                  : launch_f32<64>(q, q_idx, n_active, k_cache, v_cache, rows1, k_base, v_base,
                                   rows2, H, scale, out, s, err);
}

}  // namespace

extern "C" int hsa_active_attention(const void *q, const int32_t *q_idx, int n_active,
                                    const void *k_cache, const void *v_cache, int N, int H,
                                    int D, float scale, void *out, hsa_dtype dtype,
                                    void *workspace, size_t workspace_bytes,
                                    hsa_stream_t stream) {
  if (N < 1) return HSA_ERR_INVALID_ARG;
  return attention_two_sources(q, q_idx, n_active, k_cache, v_cache, N, nullptr, nullptr, 0, H,
                               D, scale, out, dtype, workspace, workspace_bytes, stream);
}

extern "C" int hsa_active_attention_prefix(const void *q, const int32_t *q_idx, int n_active,
                                           const void *k_cache, const void *v_cache, int M,
                                           const void *k_base, const void *v_base, int B, int H,
                                           int D, float scale, void *out, hsa_dtype dtype,
                                           void *workspace, size_t workspace_bytes,
                                           hsa_stream_t stream) {
  return attention_two_sources(q, q_idx, n_active, k_cache, v_cache, M, k_base, v_base, B, H, D,
                               scale, out, dtype, workspace, workspace_bytes, stream);
}

extern "C" int hsa_test_inject_attention_stall(int mode) {
  if (mode != 0 && mode != 1) return HSA_ERR_INVALID_ARG;
  return g_inject_stall.exchange(mode);
}
