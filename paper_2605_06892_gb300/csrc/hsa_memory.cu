// Memory-bound steps of the HSA iteration: gather of the active rows
// (Sec. 2.3, step 1), KV-cache synchronisation scatter (Sec. 2.3, step 2) and
// the cached Euler update (Sec. 2.4, Eq. 6).
//
// All three move whole token rows.  A row is split into 16-byte vectors and a
// group of L lanes (L a power of two <= 32) of one warp cooperates on a row, so
// a warp covers 32/L rows at once and every access is a coalesced 128-bit load
// or store.  Each lane keeps several vectors in flight before storing.
// The row index is read once per row by its lane group; indices are checked
// against the row count and a bad one skips its row and sets the error word.
#include <cuda_bf16.h>

#include <atomic>
#include <cmath>

#include "hsa_internal.cuh"

namespace hsa {
namespace {

constexpr int kThreads = 256;
// 16-byte vectors each lane keeps in flight (measured on GB300 with an L2-
// flushed size sweep: the gather reaches its best rate at 4, the scatter,
// whose loads are contiguous, at 8; Euler holds two vectors per step).
constexpr int kGatherUnroll = 4;
constexpr int kScatterUnroll = 8;
constexpr int kEulerUnroll = 2;  // float4 positions per thread per pass (large N)

__device__ __forceinline__ uint4 ld_stream(const uint4 *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// Row loop shared by gather and scatter: rows are handed out to lane groups
// in a grid-stride loop; `map(j, s, d)` sets the source and destination row
// pointers of row j, or returns false to skip the row.
template <int kUnroll, class RowMap>
__device__ __forceinline__ void copy_rows(long long n_rows, int vecs, int lpr_log2,
                                          RowMap map) {
  const int L = 1 << lpr_log2;
  const int lane = threadIdx.x & 31;
  const int sub = lane >> lpr_log2;                  // row slot within the warp
  const int sl = lane & (L - 1);                     // lane within the row group
  const int rows_per_warp = 32 >> lpr_log2;
  const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
  for (long long j = warp * rows_per_warp + sub; j < n_rows; j += nwarps * rows_per_warp) {
    const uint4 *s;
    uint4 *d;
    if (!map(j, s, d)) continue;
    for (int v0 = sl; v0 < vecs; v0 += kUnroll * L) {
      uint4 buf[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int v = v0 + u * L;
        if (v < vecs) buf[u] = ld_stream(s + v);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int v = v0 + u * L;
        if (v < vecs) d[v] = buf[u];
      }
    }
  }
}

__global__ void __launch_bounds__(kThreads)
gather_rows_kernel(const uint4 *__restrict__ src, uint4 *__restrict__ dst,
              const int32_t *__restrict__ idx, int n_active, int N, int vecs,
              int lpr_log2, unsigned *err) {
  pdl_wait();
  pdl_trigger();
  copy_rows<kGatherUnroll>(n_active, vecs, lpr_log2, [&](long long j, const uint4 *&s, uint4 *&d) {
    const int r = __ldg(idx + j);
    if (r < 0 || r >= N) {
      set_error(err, kErrIndex);
      return false;
    }
    s = src + (long long)r * vecs;
    d = dst + j * vecs;
    return true;
  });
}

// Rows 0..n_active-1 are K rows, n_active..2*n_active-1 the V rows, so a warp
// moves K and V rows of different tokens with the same code.
__global__ void __launch_bounds__(kThreads)
kv_scatter_kernel(uint4 *__restrict__ kc, uint4 *__restrict__ vc,
               const uint4 *__restrict__ kf, const uint4 *__restrict__ vf,
               const int32_t *__restrict__ idx, int n_active, int N, int vecs,
               int lpr_log2, unsigned *err) {
  pdl_wait();
  pdl_trigger();
  copy_rows<kScatterUnroll>(2LL * n_active, vecs, lpr_log2, [&](long long jj, const uint4 *&s, uint4 *&d) {
    const bool is_v = jj >= n_active;
    const long long j = is_v ? jj - n_active : jj;
    const int r = __ldg(idx + j);
    if (r < 0 || r >= N) {
      if (!is_v) set_error(err, kErrIndex);
      return false;
    }
    s = (is_v ? vf : kf) + j * vecs;
    d = (is_v ? vc : kc) + (long long)r * vecs;
    return true;
  });
}

// x[n] = fma(vhat[n], dsigma, x[n]) with vhat[n] refreshed from
// v_fresh[pos[n]] when pos[n] >= 0.  Element-wise over the N*C/4 float4
// vectors: each thread takes kU vectors a grid-stride apart.  The pos entries
// of a pass are loaded one pass ahead (software pipelining), so a pass issues
// its x loads and its velocity loads (v_fresh rows by pos, or the cache)
// at once: 2*kU independent loads in flight per thread whatever C is.  The
// grid is the number of blocks resident at once (a single wave).  Measured on
// GB300 with an L2-flushed size sweep: kU = 2 with the pos loads one pass
// ahead reaches 0.85-1.0 of the HBM copy rate, kU = 4 (more registers, fewer
// resident threads) 0.68-0.85.
// vec_shift = log2(C/4) when C/4 is a power of two, else -1 (division).
// Small N uses one vector per thread (kU = 1) so that every SM has work.
template <int kU>
__device__ __forceinline__ void load_pos_pass(const int32_t *__restrict__ pos, long long base,
                                              long long stride, long long total, int vecs,
                                              int vec_shift, int n_fresh_rows, unsigned *err,
                                              int (&p)[kU]) {
#pragma unroll
  for (int u = 0; u < kU; ++u) {
    const long long e = base + u * stride;
    p[u] = -1;
    if (pos && e < total) {
      const long long row = vec_shift >= 0 ? (e >> vec_shift) : e / vecs;
      p[u] = __ldg(pos + row);
      if (p[u] >= n_fresh_rows || p[u] < -1) {   // only -1 means "no fresh row"
        set_error(err, kErrIndex);
        p[u] = -1;
      }
    }
  }
}

template <int kU>
__global__ void __launch_bounds__(kThreads)
cached_euler_kernel(float4 *__restrict__ x, float4 *__restrict__ vhat,
                    const float4 *__restrict__ v_fresh, const int32_t *__restrict__ pos,
                    long long total, int vecs, int vec_shift, float dsigma, int n_fresh_rows,
                    unsigned *err) {
  pdl_wait();
  pdl_trigger();
  const long long stride = (long long)gridDim.x * blockDim.x;
  long long base = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  int pn[kU];
  load_pos_pass<kU>(pos, base, stride, total, vecs, vec_shift, n_fresh_rows, err, pn);
  for (; base < total; base += stride * kU) {
    int p[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) p[u] = pn[u];
    load_pos_pass<kU>(pos, base + stride * kU, stride, total, vecs, vec_shift, n_fresh_rows,
                      err, pn);
    float4 vb[kU], xb[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const long long e = base + u * stride;
      if (e < total) {
        const long long row = vec_shift >= 0 ? (e >> vec_shift) : e / vecs;
        const long long c = e - row * vecs;
        xb[u] = x[e];
        vb[u] = p[u] >= 0 ? __ldg(v_fresh + (long long)p[u] * vecs + c) : vhat[e];
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const long long e = base + u * stride;
      if (e < total) {
        if (p[u] >= 0) vhat[e] = vb[u];
        float4 o;
        o.x = __fmaf_rn(vb[u].x, dsigma, xb[u].x);
        o.y = __fmaf_rn(vb[u].y, dsigma, xb[u].y);
        o.z = __fmaf_rn(vb[u].z, dsigma, xb[u].z);
        o.w = __fmaf_rn(vb[u].w, dsigma, xb[u].w);
        x[e] = o;
      }
    }
  }
}

// The cached Euler step fused with the velocity statistic (below), element-
// wise like cached_euler_kernel, for C/4 a power of two <= 32: the C/4 lanes
// of a token are consecutive lanes of one warp (passes start at a multiple of
// 32), so the token's two L1 norms are reduced with log2(C/4) shuffles and the
// token's first lane updates stat.  Every lane of a warp runs the same passes
// (the shuffles span the warp).
template <int kU>
__global__ void __launch_bounds__(kThreads)
euler_l1rel_elem_kernel(float4 *__restrict__ x, float4 *__restrict__ vhat,
                        const float4 *__restrict__ v_fresh, const int32_t *__restrict__ pos,
                        long long total, int vecs, int vec_shift, float dsigma,
                        int n_fresh_rows, float *__restrict__ stat, float weight, unsigned *err) {
  const long long stride = (long long)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  long long base = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  int pn[kU];
  load_pos_pass<kU>(pos, base, stride, total, vecs, vec_shift, n_fresh_rows, err, pn);
  for (; base - lane < total; base += stride * kU) {
    int p[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) p[u] = pn[u];
    load_pos_pass<kU>(pos, base + stride * kU, stride, total, vecs, vec_shift, n_fresh_rows,
                      err, pn);
    float4 vo[kU], vn[kU], xb[kU];
    float st[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const long long e = base + u * stride;
      st[u] = 0.f;
      if (e < total) {
        const long long row = e >> vec_shift;
        const long long c = e - row * vecs;
        xb[u] = x[e];
        vo[u] = vhat[e];
        vn[u] = p[u] >= 0 ? __ldg(v_fresh + (long long)p[u] * vecs + c) : vo[u];
        if (p[u] >= 0 && (lane & (vecs - 1)) == 0) st[u] = stat[row];   // with the data
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const long long e = base + u * stride;
      float num = 0.f, den = 0.f;
      if (e < total) {
        if (p[u] >= 0) {
          num = fabsf(vn[u].x - vo[u].x) + fabsf(vn[u].y - vo[u].y) + fabsf(vn[u].z - vo[u].z) +
                fabsf(vn[u].w - vo[u].w);
          den = fabsf(vn[u].x) + fabsf(vn[u].y) + fabsf(vn[u].z) + fabsf(vn[u].w);
          vhat[e] = vn[u];
        }
        float4 o;
        o.x = __fmaf_rn(vn[u].x, dsigma, xb[u].x);
        o.y = __fmaf_rn(vn[u].y, dsigma, xb[u].y);
        o.z = __fmaf_rn(vn[u].z, dsigma, xb[u].z);
        o.w = __fmaf_rn(vn[u].w, dsigma, xb[u].w);
        x[e] = o;
      }
      for (int o = 1; o < vecs; o <<= 1) {
        num += __shfl_xor_sync(0xffffffffu, num, o);
        den += __shfl_xor_sync(0xffffffffu, den, o);
      }
      if (e < total && p[u] >= 0 && (lane & (vecs - 1)) == 0) {
        const long long row = e >> vec_shift;
        const float r = den > 0.f ? num / den : (num > 0.f ? 3.402823466e38f : 0.f);
        stat[row] = fmaf(weight, r, st[u]);
      }
    }
  }
}

// Cached Euler step fused with the velocity statistic of the dynamic token
// selection (App. B, Eq. 7): for a refreshed token (pos[n] >= 0) the old cache
// row is v_{i-1}[n] and the fresh row v_i[n]; the kernel adds
// weight * ||v_i - v_{i-1}||_1 / ||v_i||_1 to stat[n] (a zero denominator
// counts 0 with a zero numerator, FLT_MAX otherwise), then refreshes the cache
// and advances x exactly as cached_euler_kernel does.  This layout (for C/4
// not a power of two, or above 32): a group of L lanes owns a token; the two
// L1 norms are reduced across the group with shuffles.
constexpr int kL1relRows = 2;   // tokens per lane group per pass

__global__ void __launch_bounds__(kThreads, 4)
euler_l1rel_kernel(float4 *__restrict__ x, float4 *__restrict__ vhat,
                   const float4 *__restrict__ v_fresh, const int32_t *__restrict__ pos,
                   int N, int vecs, int lpr_log2, float dsigma, int n_fresh_rows,
                   float *__restrict__ stat, float weight, unsigned *err) {
  const int L = 1 << lpr_log2;
  const int lane = threadIdx.x & 31;
  const int sub = lane >> lpr_log2;
  const int sl = lane & (L - 1);
  const int rows_per_warp = 32 >> lpr_log2;
  const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
  const long long step = nwarps * rows_per_warp;            // between a group's tokens
  // All lanes of a warp run the same number of passes (the shuffles below
  // span the warp): the bound is the token count rounded up to whole passes.
  const long long span = step * kL1relRows;
  const long long rows_pad = ((long long)N + span - 1) / span * span;
  for (long long n0 = warp * rows_per_warp; n0 < rows_pad; n0 += span) {
    long long n[kL1relRows];
    int p[kL1relRows];
#pragma unroll
    for (int k = 0; k < kL1relRows; ++k) {
      n[k] = n0 + k * step + sub;
      p[k] = (n[k] < N) ? __ldg(pos + n[k]) : -1;
      if (p[k] >= n_fresh_rows || p[k] < -1) {
        set_error(err, kErrIndex);
        p[k] = -1;
      }
    }
    float num[kL1relRows], den[kL1relRows];
#pragma unroll
    for (int k = 0; k < kL1relRows; ++k) num[k] = den[k] = 0.f;
    for (int v = sl; v < vecs; v += L) {
      float4 vo[kL1relRows], vn[kL1relRows], xv[kL1relRows];
#pragma unroll
      for (int k = 0; k < kL1relRows; ++k) {
        if (n[k] < N) {
          vo[k] = vhat[n[k] * vecs + v];
          vn[k] = p[k] >= 0 ? __ldg(v_fresh + (long long)p[k] * vecs + v) : vo[k];
          xv[k] = x[n[k] * vecs + v];
        }
      }
#pragma unroll
      for (int k = 0; k < kL1relRows; ++k) {
        if (n[k] < N) {
          if (p[k] >= 0) {
            num[k] += fabsf(vn[k].x - vo[k].x) + fabsf(vn[k].y - vo[k].y) +
                      fabsf(vn[k].z - vo[k].z) + fabsf(vn[k].w - vo[k].w);
            den[k] += fabsf(vn[k].x) + fabsf(vn[k].y) + fabsf(vn[k].z) + fabsf(vn[k].w);
            vhat[n[k] * vecs + v] = vn[k];
          }
          float4 o;
          o.x = __fmaf_rn(vn[k].x, dsigma, xv[k].x);
          o.y = __fmaf_rn(vn[k].y, dsigma, xv[k].y);
          o.z = __fmaf_rn(vn[k].z, dsigma, xv[k].z);
          o.w = __fmaf_rn(vn[k].w, dsigma, xv[k].w);
          x[n[k] * vecs + v] = o;
        }
      }
    }
#pragma unroll
    for (int k = 0; k < kL1relRows; ++k) {
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        if (o < L) {
          num[k] += __shfl_xor_sync(0xffffffffu, num[k], o);
          den[k] += __shfl_xor_sync(0xffffffffu, den[k], o);
        }
      }
      if (n[k] < N && p[k] >= 0 && sl == 0) {
        const float r = den[k] > 0.f ? num[k] / den[k] : (num[k] > 0.f ? 3.402823466e38f : 0.f);
        stat[n[k]] = fmaf(weight, r, stat[n[k]]);
      }
    }
  }
}

// Rotary position embedding of the active rows (Sec. 2.3: the positional
// frequencies are subsampled to A_i): row j of a token tensor is rotated by
// the (cos, sin) table row of its token idx[j].  One 16-byte vector holds 8
// bf16 values = 4 rotation pairs; pair (x0, x1) becomes
// (fma(x0, c, -(x1 s)), fma(x0, s, x1 c)) in fp32, rounded to bf16.
__device__ __forceinline__ uint4 rope8(uint4 v, const float4 *tab) {
  uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float4 cs2 = __ldg(tab + (k >> 1));          // (c, s) of two pairs
    const float c = (k & 1) ? cs2.z : cs2.x, s = (k & 1) ? cs2.w : cs2.y;
    const float x0 = __uint_as_float(w[k] << 16), x1 = __uint_as_float(w[k] & 0xffff0000u);
    const float y0 = __fmaf_rn(x0, c, -(x1 * s));
    const float y1 = __fmaf_rn(x0, s, x1 * c);
    const __nv_bfloat162 r = __floats2bfloat162_rn(y0, y1);
    w[k] = *reinterpret_cast<const uint32_t *>(&r);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// In-place rotation of rows j < n of x [n, H*D] (bf16): a lane group owns a
// row; vector c covers head 8c / D and pairs ((8c) % D)/2 .. +3.
__global__ void __launch_bounds__(kThreads)
rope_rows_kernel(uint4 *__restrict__ x, const int32_t *__restrict__ idx, int n, int vecs, int D,
                 const float4 *__restrict__ table, int N, int lpr_log2, unsigned *err) {
  const int L = 1 << lpr_log2;
  const int lane = threadIdx.x & 31;
  const int sub = lane >> lpr_log2, sl = lane & (L - 1);
  const int rows_per_warp = 32 >> lpr_log2;
  const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
  const int pairs = D / 2;
  for (long long j = warp * rows_per_warp + sub; j < n; j += nwarps * rows_per_warp) {
    const int t = __ldg(idx + j);
    if (t < 0 || t >= N) {
      set_error(err, kErrIndex);
      continue;
    }
    const float4 *trow = table + (size_t)t * (pairs / 2);
    uint4 *row = x + j * vecs;
    for (int v = sl; v < vecs; v += L) {
      const int pair0 = ((v * 8) % D) / 2;
      row[v] = rope8(row[v], trow + pair0 / 2);
    }
  }
}

// KV-cache synchronisation with K rotated on the way in: rows 0..n-1 are K
// rows (rotated by the table row of token idx[j]), rows n..2n-1 the V rows
// (copied).
__global__ void __launch_bounds__(kThreads)
kv_scatter_rope_kernel(uint4 *__restrict__ kc, uint4 *__restrict__ vc,
                       const uint4 *__restrict__ kf, const uint4 *__restrict__ vf,
                       const int32_t *__restrict__ idx, int n_active, int N, int vecs, int D,
                       const float4 *__restrict__ table, int lpr_log2, unsigned *err) {
  const int L = 1 << lpr_log2;
  const int lane = threadIdx.x & 31;
  const int sub = lane >> lpr_log2, sl = lane & (L - 1);
  const int rows_per_warp = 32 >> lpr_log2;
  const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
  const int pairs = D / 2;
  for (long long jj = warp * rows_per_warp + sub; jj < 2LL * n_active;
       jj += nwarps * rows_per_warp) {
    const bool is_v = jj >= n_active;
    const long long j = is_v ? jj - n_active : jj;
    const int r = __ldg(idx + j);
    if (r < 0 || r >= N) {
      if (!is_v) set_error(err, kErrIndex);
      continue;
    }
    const uint4 *s = (is_v ? vf : kf) + j * vecs;
    uint4 *d = (is_v ? vc : kc) + (long long)r * vecs;
    const float4 *trow = table + (size_t)r * (pairs / 2);
    for (int v0 = sl; v0 < vecs; v0 += kScatterUnroll * L) {
      uint4 buf[kScatterUnroll];
#pragma unroll
      for (int u = 0; u < kScatterUnroll; ++u) {
        const int v = v0 + u * L;
        if (v < vecs) buf[u] = ld_stream(s + v);
      }
#pragma unroll
      for (int u = 0; u < kScatterUnroll; ++u) {
        const int v = v0 + u * L;
        if (v < vecs) d[v] = is_v ? buf[u] : rope8(buf[u], trow + (((v * 8) % D) / 2) / 2);
      }
    }
  }
}

// Index check (opt-in, for debugging a caller's index arrays): every entry of
// idx must lie in [0, N) and no value may appear twice.  Sec. 2.2 makes the
// groups disjoint, so A_i never repeats a token; a repeated id would make the
// KV scatter race.  One bit per token in a caller workspace, cleared first
// (bitmap_clear_kernel), then set with atomicOr: an entry that finds its bit
// already set is a repeat.
__global__ void __launch_bounds__(kThreads)
bitmap_clear_kernel(uint4 *__restrict__ bits, long long n_vec) {
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long v = blockIdx.x * (long long)blockDim.x + threadIdx.x; v < n_vec; v += stride)
    bits[v] = make_uint4(0u, 0u, 0u, 0u);
}

__global__ void __launch_bounds__(kThreads)
check_indices_kernel(const int32_t *__restrict__ idx, long long n, int N,
                     unsigned *__restrict__ bits, unsigned *err) {
  const long long stride = (long long)gridDim.x * blockDim.x;
  bool bad = false;
  for (long long j = blockIdx.x * (long long)blockDim.x + threadIdx.x; j < n; j += stride) {
    const int t = __ldg(idx + j);
    if (t < 0 || t >= N) {
      bad = true;
      continue;
    }
    const unsigned bit = 1u << (t & 31);
    if (atomicOr(bits + (t >> 5), bit) & bit) bad = true;
  }
  if (bad) set_error(err, kErrIndex);
}

// Grid for n_rows rows handled by lane groups of size L: up to 8 blocks of
// 256 threads per SM (a full SM), no more than the rows need; blocks beyond
// what is resident wait their turn.
int grid_for(long long n_rows, int L) {
  const long long rows_per_block = (long long)(kThreads / 32) * (32 / L);
  long long blocks = (n_rows + rows_per_block - 1) / rows_per_block;
  const long long cap = (long long)sm_count() * (2048 / kThreads);
  if (blocks > cap) blocks = cap;
  return (int)(blocks < 1 ? 1 : blocks);
}

// Blocks of kernel K (kThreads threads) resident on the whole device at once,
// resolved once per device: a grid-stride kernel launched with this many
// blocks runs in a single wave.
template <auto K>
long long resident_blocks() {
  static std::atomic<int> per_sm[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return sm_count();
  int nb = per_sm[dev].load(std::memory_order_relaxed);
  if (nb <= 0) {
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, K, kThreads, 0) != cudaSuccess ||
        nb < 1)
      nb = 1;
    per_sm[dev].store(nb, std::memory_order_relaxed);
  }
  return (long long)nb * sm_count();
}

int log2i(int L) {
  int s = 0;
  while ((1 << s) < L) ++s;
  return s;
}

}  // namespace
}  // namespace hsa

using namespace hsa;

extern "C" int hsa_gather_active(const void *src, size_t row_bytes, int N,
                                 const int32_t *idx, int n_active, void *dst,
                                 hsa_stream_t stream) {
  if (N < 0 || n_active < 0 || row_bytes == 0 || (row_bytes & 15)) return HSA_ERR_INVALID_ARG;
  if (n_active == 0) return HSA_OK;
  if (!src || !dst || !idx || !aligned16(src) || !aligned16(dst)) return HSA_ERR_INVALID_ARG;
  const long long vecs = (long long)(row_bytes / 16);
  if (vecs > (1LL << 30)) return HSA_ERR_UNSUPPORTED;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const int L = lanes_per_row(vecs);
  count_launches(1);
  launch_pdl(gather_rows_kernel, dim3(grid_for(n_active, L)), dim3(kThreads), 0,
             (cudaStream_t)stream, (const uint4 *)src, (uint4 *)dst, idx, n_active, N, (int)vecs,
             log2i(L), err);
  return launch_status();
}

extern "C" int hsa_kv_sync_scatter(void *k_cache, void *v_cache, const void *k_fresh,
                                   const void *v_fresh, const int32_t *idx, int n_active,
                                   int N, int H, int D, hsa_dtype dtype,
                                   hsa_stream_t stream) {
  if (N < 0 || n_active < 0 || H < 1 || D < 1) return HSA_ERR_INVALID_ARG;
  if (dtype != HSA_BF16 && dtype != HSA_F32) return HSA_ERR_INVALID_ARG;
  const long long row_bytes = (long long)H * D * (dtype == HSA_BF16 ? 2 : 4);
  if (row_bytes & 15) return HSA_ERR_UNSUPPORTED;
  if (n_active == 0) return HSA_OK;
  if (!k_cache || !v_cache || !k_fresh || !v_fresh || !idx) return HSA_ERR_INVALID_ARG;
  if (!aligned16(k_cache) || !aligned16(v_cache) || !aligned16(k_fresh) || !aligned16(v_fresh))
    return HSA_ERR_INVALID_ARG;
  const long long vecs = row_bytes / 16;
  if (vecs > (1LL << 30)) return HSA_ERR_UNSUPPORTED;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const int L = lanes_per_row(vecs);
  count_launches(1);
  launch_pdl(kv_scatter_kernel, dim3(grid_for(2LL * n_active, L)), dim3(kThreads), 0,
             (cudaStream_t)stream, (uint4 *)k_cache, (uint4 *)v_cache, (const uint4 *)k_fresh,
             (const uint4 *)v_fresh, idx, n_active, N, (int)vecs, log2i(L), err);
  return launch_status();
}

extern "C" int hsa_cached_euler(float *x, float *v_cache, const float *v_fresh,
                                const int32_t *pos, int n_fresh, int N, int C, float dsigma,
                                hsa_stream_t stream) {
  if (N < 0 || C < 4 || (C & 3) || n_fresh < 0) return HSA_ERR_INVALID_ARG;
  if ((pos == nullptr) != (v_fresh == nullptr)) return HSA_ERR_INVALID_ARG;
  if (N == 0) return HSA_OK;
  if (!x || !v_cache || !aligned16(x) || !aligned16(v_cache)) return HSA_ERR_INVALID_ARG;
  if (v_fresh && !aligned16(v_fresh)) return HSA_ERR_INVALID_ARG;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const int vecs = C / 4;
  const long long total = (long long)N * vecs;
  int vec_shift = -1;
  for (int sh = 0; sh < 31; ++sh)
    if ((1 << sh) == vecs) vec_shift = sh;
  const long long resident = (long long)sm_count() * 2048;     // threads
  const int per = total >= (long long)kEulerUnroll * resident ? kEulerUnroll : 1;
  long long blocks = (total + (long long)kThreads * per - 1) / ((long long)kThreads * per);
  const long long cap = per == kEulerUnroll ? resident_blocks<cached_euler_kernel<kEulerUnroll>>()
                                            : resident_blocks<cached_euler_kernel<1>>();
  if (blocks > cap) blocks = cap;
  count_launches(1);
  if (per == kEulerUnroll)
    launch_pdl(cached_euler_kernel<kEulerUnroll>, dim3((unsigned)blocks), dim3(kThreads), 0,
               (cudaStream_t)stream, (float4 *)x, (float4 *)v_cache, (const float4 *)v_fresh,
               pos, total, vecs, vec_shift, dsigma, pos ? n_fresh : 0, err);
  else
    launch_pdl(cached_euler_kernel<1>, dim3((unsigned)blocks), dim3(kThreads), 0,
               (cudaStream_t)stream, (float4 *)x, (float4 *)v_cache, (const float4 *)v_fresh,
               pos, total, vecs, vec_shift, dsigma, pos ? n_fresh : 0, err);
  return launch_status();
}

extern "C" int hsa_cached_euler_l1rel(float *x, float *v_cache, const float *v_fresh,
                                      const int32_t *pos, int n_fresh, int N, int C,
                                      float dsigma, float *stat, float weight,
                                      hsa_stream_t stream) {
  if (N < 0 || C < 4 || (C & 3) || n_fresh < 0) return HSA_ERR_INVALID_ARG;
  if (!pos || !v_fresh || !stat) return HSA_ERR_INVALID_ARG;
  if (N == 0) return HSA_OK;
  if (!x || !v_cache || !aligned16(x) || !aligned16(v_cache) || !aligned16(v_fresh))
    return HSA_ERR_INVALID_ARG;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const int vecs = C / 4;
  int vec_shift = -1;
  for (int sh = 0; sh <= 5; ++sh)
    if ((1 << sh) == vecs) vec_shift = sh;
  if (vec_shift >= 0) {
    // element-wise: C/4 a power of two, at most 32 (a token within one warp)
    const long long total = (long long)N * vecs;
    const long long resident = (long long)sm_count() * 2048;     // threads
    const int per = total >= (long long)kEulerUnroll * resident ? kEulerUnroll : 1;
    long long blocks = (total + (long long)kThreads * per - 1) / ((long long)kThreads * per);
    const long long cap = per == kEulerUnroll
                              ? resident_blocks<euler_l1rel_elem_kernel<kEulerUnroll>>()
                              : resident_blocks<euler_l1rel_elem_kernel<1>>();
    if (blocks > cap) blocks = cap;
    count_launches(1);
    if (per == kEulerUnroll)
      euler_l1rel_elem_kernel<kEulerUnroll><<<(int)blocks, kThreads, 0, (cudaStream_t)stream>>>(
          (float4 *)x, (float4 *)v_cache, (const float4 *)v_fresh, pos, total, vecs, vec_shift,
          dsigma, n_fresh, stat, weight, err);
    else
      euler_l1rel_elem_kernel<1><<<(int)blocks, kThreads, 0, (cudaStream_t)stream>>>(
          (float4 *)x, (float4 *)v_cache, (const float4 *)v_fresh, pos, total, vecs, vec_shift,
          dsigma, n_fresh, stat, weight, err);
    return launch_status();
  }
  const int L = lanes_per_row(vecs);
  count_launches(1);
  euler_l1rel_kernel<<<grid_for(((long long)N + kL1relRows - 1) / kL1relRows, L), kThreads, 0,
                       (cudaStream_t)stream>>>(
      (float4 *)x, (float4 *)v_cache, (const float4 *)v_fresh, pos, N, vecs, log2i(L), dsigma,
      n_fresh, stat, weight, err);
  return launch_status();
}

extern "C" int hsa_rope_table(int F, int Hh, int Ww, int D, double theta, float *table) {
  if (F < 1 || Hh < 1 || Ww < 1 || D < 8 || (D & 7) || !(theta > 1.0) || !table)
    return HSA_ERR_INVALID_ARG;
  const int P = D / 2, ph = D / 6, pt = P - 2 * ph;
  for (int f = 0; f < F; ++f)
    for (int h = 0; h < Hh; ++h)
      for (int w = 0; w < Ww; ++w) {
        const size_t n = ((size_t)f * Hh + h) * Ww + w;
        for (int i = 0; i < P; ++i) {
          const bool tb = i < pt, hb = !tb && i < pt + ph;
          const int bi = tb ? i : (hb ? i - pt : i - pt - ph);
          const int bp = tb ? pt : ph;
          const int pos = tb ? f : (hb ? h : w);
          const double ang = (double)pos * std::pow(theta, -(double)bi / (double)bp);
          table[(n * P + i) * 2] = (float)std::cos(ang);
          table[(n * P + i) * 2 + 1] = (float)std::sin(ang);
        }
      }
  return HSA_OK;
}

extern "C" int hsa_rope_rows(void *x, const int32_t *idx, int n, int H, int D,
                             const float *table, int N, hsa_stream_t stream) {
  if (n < 0 || H < 1 || D < 8 || (D & 7) || N < 1) return HSA_ERR_INVALID_ARG;
  if (n == 0) return HSA_OK;
  if (!x || !idx || !table || !aligned16(x) || !aligned16(table)) return HSA_ERR_INVALID_ARG;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const long long vecs = (long long)H * D / 8;
  if (vecs > (1LL << 30)) return HSA_ERR_UNSUPPORTED;
  const int L = lanes_per_row(vecs);
  count_launches(1);
  rope_rows_kernel<<<grid_for(n, L), kThreads, 0, (cudaStream_t)stream>>>(
      (uint4 *)x, idx, n, (int)vecs, D, (const float4 *)table, N, log2i(L), err);
  return launch_status();
}

extern "C" int hsa_kv_sync_scatter_rope(void *k_cache, void *v_cache, const void *k_fresh,
                                        const void *v_fresh, const int32_t *idx, int n_active,
                                        int N, int H, int D, const float *table,
                                        hsa_stream_t stream) {
  if (N < 0 || n_active < 0 || H < 1 || D < 8 || (D & 7)) return HSA_ERR_INVALID_ARG;
  if (n_active == 0) return HSA_OK;
  if (!k_cache || !v_cache || !k_fresh || !v_fresh || !idx || !table) return HSA_ERR_INVALID_ARG;
  if (!aligned16(k_cache) || !aligned16(v_cache) || !aligned16(k_fresh) || !aligned16(v_fresh) ||
      !aligned16(table))
    return HSA_ERR_INVALID_ARG;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const long long vecs = (long long)H * D / 8;
  if (vecs > (1LL << 30)) return HSA_ERR_UNSUPPORTED;
  const int L = lanes_per_row(vecs);
  count_launches(1);
  kv_scatter_rope_kernel<<<grid_for(2LL * n_active, L), kThreads, 0, (cudaStream_t)stream>>>(
      (uint4 *)k_cache, (uint4 *)v_cache, (const uint4 *)k_fresh, (const uint4 *)v_fresh, idx,
      n_active, N, (int)vecs, D, (const float4 *)table, log2i(L), err);
  return launch_status();
}

extern "C" size_t hsa_check_indices_workspace_bytes(int N) {
  if (N <= 0) return 0;
  return (((size_t)N + 31) / 32 * 4 + 255) / 256 * 256;   // one bit per token, whole uint4s
}

extern "C" int hsa_check_indices(const int32_t *idx, int n, int N, void *workspace,
                                 size_t workspace_bytes, hsa_stream_t stream) {
  if (n < 0 || N < 0) return HSA_ERR_INVALID_ARG;
  if (n == 0) return HSA_OK;
  if (!idx) return HSA_ERR_INVALID_ARG;
  const size_t need = hsa_check_indices_workspace_bytes(N);
  if (N > 0 && (!workspace || workspace_bytes < need ||
                (reinterpret_cast<uintptr_t>(workspace) & 255)))
    return HSA_ERR_WORKSPACE;
  unsigned *err = device_error_word();
  if (!err) return HSA_ERR_CUDA;
  const long long cap = (long long)sm_count() * (2048 / kThreads);
  const long long n_vec = (long long)(need / 16);
  long long b0 = (n_vec + kThreads - 1) / kThreads, b1 = (n + kThreads - 1) / kThreads;
  b0 = b0 < 1 ? 1 : (b0 > cap ? cap : b0);
  b1 = b1 > cap ? cap : b1;
  cudaStream_t s = (cudaStream_t)stream;
  if (n_vec > 0) {
    count_launches(1);
    bitmap_clear_kernel<<<(int)b0, kThreads, 0, s>>>(static_cast<uint4 *>(workspace), n_vec);
  }
  count_launches(1);
  check_indices_kernel<<<(int)b1, kThreads, 0, s>>>(idx, n, N, static_cast<unsigned *>(workspace),
                                                    err);
  return launch_status();
}
