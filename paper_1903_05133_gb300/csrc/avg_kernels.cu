// Local and global averages of Algorithm 1 (Sec. 3.1) over a learner-indexed
// fp32 matrix w[P, ld]: in-memory segmented / full means over the learner axis.
//
// Each thread owns one 16-byte column slice (4 consecutive parameters) and walks
// the n rows of its cluster (or of all P learners): loads are 128-bit and a warp
// reads 512 contiguous bytes per row, so every row access is fully coalesced.
// The sum over rows follows the canonical adjacent-pair tree (v[i] += v[i+h] for
// h = 1, 2, 4, ..., unpaired elements carried up), evaluated as a streaming binary
// counter: pushing value i combines it with the pending partials of the same
// size, exactly like incrementing a binary number, so only log2(n)+1 partials
// live in registers.  Then one IEEE division by n and a broadcast write-back.
// The arithmetic is __fadd_rn / __fdiv_rn only (no FMA, no flush to zero), so the
// result is bit-identical to the CPU definition of the same tree.
#include <cstdint>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace ha {
namespace {

__device__ __forceinline__ float vadd(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ float4 vadd(float4 a, float4 b) {
  return make_float4(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y), __fadd_rn(a.z, b.z),
                     __fadd_rn(a.w, b.w));
}
__device__ __forceinline__ float vdiv(float a, float n) { return __fdiv_rn(a, n); }
__device__ __forceinline__ float4 vdiv(float4 a, float n) {
  return make_float4(__fdiv_rn(a.x, n), __fdiv_rn(a.y, n), __fdiv_rn(a.z, n),
                     __fdiv_rn(a.w, n));
}

// Sum of the 2^LOG consecutive rows starting at p (row stride ld_v in vectors).
template <int LOG, class V>
__device__ __forceinline__ V tree_pow2(const V* __restrict__ p, int64_t ld_v) {
  constexpr int N = 1 << LOG;
  V stack[LOG + 1];
#pragma unroll
  for (int i = 0; i < N; ++i) {
    V x = p[static_cast<int64_t>(i) * ld_v];
    int l = 0;
#pragma unroll
    for (; l < LOG; ++l) {
      if (((i >> l) & 1) == 0) break;
      x = vadd(stack[l], x);
    }
    stack[l] = x;
  }
  return stack[LOG];
}

template <class V>
__device__ __forceinline__ void store_rows(V* p, int64_t ld_v, int n, V m) {
#pragma unroll 8
  for (int i = 0; i < n; ++i) p[static_cast<int64_t>(i) * ld_v] = m;
}

// Group means, n = 2^LOG rows per group; grid.y = group index.
template <int LOG>
__global__ void __launch_bounds__(256) k_mean_pow2(float4* __restrict__ w, int64_t ld_v,
                                                   int64_t cols_v) {
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c >= cols_v) return;
  float4* p = w + static_cast<int64_t>(blockIdx.y) * (int64_t(1) << LOG) * ld_v + c;
  const float4 m = vdiv(tree_pow2<LOG>(p, ld_v), static_cast<float>(1 << LOG));
  store_rows(p, ld_v, 1 << LOG, m);
}

// The same group sums divided by div, written once per group, to row blockIdx.y of
// out (row stride out_ld_v): compact cluster means, the rows of w only read.  div is
// the group size, or, when the rows of w are themselves sums of the first tree levels
// (group sums of Q learners), the cluster size.
template <int LOG>
__global__ void __launch_bounds__(256) k_mean_pow2_to(const float4* __restrict__ w, int64_t ld_v,
                                                      int64_t cols_v, float div,
                                                      float4* __restrict__ out, int64_t out_ld_v) {
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c >= cols_v) return;
  const float4* p = w + static_cast<int64_t>(blockIdx.y) * (int64_t(1) << LOG) * ld_v + c;
  out[static_cast<int64_t>(blockIdx.y) * out_ld_v + c] = vdiv(tree_pow2<LOG>(p, ld_v), div);
}

// Fused last local average + global average: G = 2^LOGG clusters of S = 2^LOGS.
// The global tree runs over the P values the local average would have written
// (S copies of each cluster mean, in learner order), so the result is the literal
// two-pass result: the S equal copies of a cluster form one complete sub-tree of
// the global tree, whose value is the cluster mean added to itself LOGS times.
// Each cluster's sum is the tree over its 2^(LOGS - LOGQ) rows of src (row stride
// src_ld_v): the learner rows themselves (LOGQ = 0, src = w), or sums of Q = 2^LOGQ
// learners each that hold the first LOGQ levels of the cluster's tree.  The result
// is written to all P rows of w (src may be rows of w: a thread reads its column of
// every source row before it writes).
template <int LOGQ, int LOGS, int LOGG>
__global__ void __launch_bounds__(256) k_local_global_pow2(const float4* src, int64_t src_ld_v,
                                                           float4* w, int64_t ld_v, int64_t cols_v) {
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c >= cols_v) return;
  constexpr int S = 1 << LOGS, G = 1 << LOGG, N = 1 << (LOGS - LOGQ);
  const float4* q = src + c;
  float4 stack[LOGG + 1];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float4 x = vdiv(tree_pow2<LOGS - LOGQ>(q + static_cast<int64_t>(g) * N * src_ld_v, src_ld_v),
                    static_cast<float>(S));
#pragma unroll
    for (int l = 0; l < LOGS; ++l) x = vadd(x, x);
    int l = 0;
#pragma unroll
    for (; l < LOGG; ++l) {
      if (((g >> l) & 1) == 0) break;
      x = vadd(stack[l], x);
    }
    stack[l] = x;
  }
  const float4 m = vdiv(stack[LOGG], static_cast<float>(S * G));
  store_rows(w + c, ld_v, S * G, m);
}

// The same two kernels with each column's rows split between two threads (threadIdx.y),
// for short rows (D small against the GPU): twice the threads, each walking half the
// rows.  The tree over 2^LOG rows is the tree over each half joined by one addition
// (first half + second half), so the result has the same bits.  blockDim = (128, 2).
template <int LOG>
__global__ void __launch_bounds__(256) k_mean_pow2_split(float4* w, int64_t ld_v, int64_t cols_v) {
  __shared__ float4 part[128];
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * 128 + threadIdx.x;
  const bool valid = c < cols_v;
  constexpr int H = 1 << (LOG - 1);
  float4* p = w + static_cast<int64_t>(blockIdx.y) * (int64_t(1) << LOG) * ld_v + c +
              static_cast<int64_t>(threadIdx.y) * H * ld_v;
  float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
  if (valid) x = tree_pow2<LOG - 1>(p, ld_v);
  if (threadIdx.y == 1) part[threadIdx.x] = x;
  __syncthreads();
  if (threadIdx.y == 0) part[threadIdx.x] = vdiv(vadd(x, part[threadIdx.x]), static_cast<float>(1 << LOG));
  __syncthreads();
  if (valid) store_rows(p, ld_v, H, part[threadIdx.x]);
}

// (threadIdx.y = which half of the G clusters; the first G / 2 clusters' S copies form a
// complete sub-tree of the global tree.)
template <int LOGQ, int LOGS, int LOGG>
__global__ void __launch_bounds__(256) k_local_global_pow2_split(const float4* src, int64_t src_ld_v,
                                                                 float4* w, int64_t ld_v,
                                                                 int64_t cols_v) {
  __shared__ float4 part[128];
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * 128 + threadIdx.x;
  const bool valid = c < cols_v;
  constexpr int S = 1 << LOGS, G2 = 1 << (LOGG - 1), N = 1 << (LOGS - LOGQ);
  const int g0 = static_cast<int>(threadIdx.y) * G2;
  float4 half = make_float4(0.f, 0.f, 0.f, 0.f);
  if (valid) {
    const float4* q = src + c;
    float4 stack[LOGG];
#pragma unroll
    for (int g = 0; g < G2; ++g) {
      float4 x = vdiv(tree_pow2<LOGS - LOGQ>(q + static_cast<int64_t>(g0 + g) * N * src_ld_v, src_ld_v),
                      static_cast<float>(S));
#pragma unroll
      for (int l = 0; l < LOGS; ++l) x = vadd(x, x);
      int l = 0;
#pragma unroll
      for (; l < LOGG - 1; ++l) {
        if (((g >> l) & 1) == 0) break;
        x = vadd(stack[l], x);
      }
      stack[l] = x;
    }
    half = stack[LOGG - 1];
  }
  if (threadIdx.y == 1) part[threadIdx.x] = half;
  __syncthreads();
  if (threadIdx.y == 0)
    part[threadIdx.x] = vdiv(vadd(half, part[threadIdx.x]), static_cast<float>(S * (2 * G2)));
  __syncthreads();
  if (valid) store_rows(w + c + static_cast<int64_t>(g0) * S * ld_v, ld_v, G2 * S, part[threadIdx.x]);
}

// Generic path: any n (also non-powers of two) and scalar columns.  The binary
// counter lives in a small local array; after n pushes its pending partials are
// the set bits of n, folded from the smallest upward.
template <class V>
__device__ V tree_any(const V* __restrict__ p, int64_t ld_v, int n) {
  V stack[32];
  for (int i = 0; i < n; ++i) {
    V x = p[static_cast<int64_t>(i) * ld_v];
    int l = 0;
    while ((i >> l) & 1) {
      x = vadd(stack[l], x);
      ++l;
    }
    stack[l] = x;
  }
  V acc{};
  bool have = false;
  for (int l = 0; l < 32; ++l) {
    if ((n >> l) & 1) {
      acc = have ? vadd(stack[l], acc) : stack[l];
      have = true;
    }
  }
  return acc;
}

template <class V>
__global__ void __launch_bounds__(256) k_mean_any(V* __restrict__ w, int64_t ld_v,
                                                  int64_t cols_v, int n) {
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c >= cols_v) return;
  V* p = w + static_cast<int64_t>(blockIdx.y) * n * ld_v + c;
  const V m = vdiv(tree_any(p, ld_v, n), static_cast<float>(n));
  store_rows(p, ld_v, n, m);
}

template <class V>
__global__ void __launch_bounds__(256) k_mean_any_to(const V* __restrict__ w, int64_t ld_v,
                                                     int64_t cols_v, int n, float div,
                                                     V* __restrict__ out, int64_t out_ld_v) {
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c >= cols_v) return;
  const V* p = w + static_cast<int64_t>(blockIdx.y) * n * ld_v + c;
  out[static_cast<int64_t>(blockIdx.y) * out_ld_v + c] = vdiv(tree_any(p, ld_v, n), div);
}

// (src, src_ld_v, n: as in k_local_global_pow2, n = S / Q source rows per cluster.)
template <class V>
__global__ void __launch_bounds__(256) k_local_global_any(const V* src, int64_t src_ld_v, int n,
                                                          V* w, int64_t ld_v, int64_t cols_v, int S,
                                                          int G) {
  grid_dep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c >= cols_v) return;
  V* p = w + c;
  const V* q = src + c;
  V stack[32];
  int64_t i = 0;   // index of the next pushed value of the global sequence
  for (int g = 0; g < G; ++g) {
    const V m = vdiv(tree_any(q + static_cast<int64_t>(g) * n * src_ld_v, src_ld_v, n),
                     static_cast<float>(S));
    for (int r = 0; r < S; ++r, ++i) {
      V x = m;
      int l = 0;
      while ((i >> l) & 1) {
        x = vadd(stack[l], x);
        ++l;
      }
      stack[l] = x;
    }
  }
  const int total = S * G;
  V acc{};
  bool have = false;
  for (int l = 0; l < 32; ++l) {
    if ((total >> l) & 1) {
      acc = have ? vadd(stack[l], acc) : stack[l];
      have = true;
    }
  }
  store_rows(p, ld_v, total, vdiv(acc, static_cast<float>(total)));
}

constexpr int kThreads = 256;

int ilog2_exact(int64_t n) {
  if (n < 1 || (n & (n - 1)) != 0) return -1;
  int l = 0;
  while ((int64_t(1) << l) < n) ++l;
  return l;
}

// Fewer columns than about two waves of one-thread-per-column CTAs: split each column's
// rows between two threads.
constexpr int64_t kSplitCols = 2 * 152 * 8 * 256;
bool split_rows(int64_t cols_v, int64_t groups) { return cols_v * groups <= kSplitCols; }

template <int LOG>
void launch_mean_pow2(float4* w, int64_t ld_v, int64_t cols_v, int64_t groups,
                      cudaStream_t s) {
  if (split_rows(cols_v, groups)) {
    dim3 grid(static_cast<unsigned>((cols_v + 127) / 128), static_cast<unsigned>(groups));
    launch_pdl(k_mean_pow2_split<LOG>, grid, dim3(128, 2), 0, s, false, 1, w, ld_v, cols_v);
    return;
  }
  dim3 grid(static_cast<unsigned>((cols_v + kThreads - 1) / kThreads),
            static_cast<unsigned>(groups));
  launch_pdl(k_mean_pow2<LOG>, grid, dim3(kThreads), 0, s, false, 1, w, ld_v, cols_v);
}

// (The _to launches: rows of w with stride ld_v, rows of out with stride out_ld_v.)
template <int LOG>
void launch_mean_pow2_to(const float4* w, int64_t ld_v, int64_t cols_v, int64_t groups, float div,
                         float4* out, int64_t out_ld_v, cudaStream_t s) {
  dim3 grid(static_cast<unsigned>((cols_v + kThreads - 1) / kThreads),
            static_cast<unsigned>(groups));
  launch_pdl(k_mean_pow2_to<LOG>, grid, dim3(kThreads), 0, s, false, 1, w, ld_v, cols_v, div, out,
             out_ld_v);
}

bool mean_pow2_to_dispatch(int log, const float4* w, int64_t ld_v, int64_t cols_v, int64_t groups,
                           float div, float4* out, int64_t out_ld_v, cudaStream_t s) {
  switch (log) {
    case 0: launch_mean_pow2_to<0>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 1: launch_mean_pow2_to<1>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 2: launch_mean_pow2_to<2>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 3: launch_mean_pow2_to<3>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 4: launch_mean_pow2_to<4>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 5: launch_mean_pow2_to<5>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 6: launch_mean_pow2_to<6>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    case 7: launch_mean_pow2_to<7>(w, ld_v, cols_v, groups, div, out, out_ld_v, s); return true;
    default: return false;
  }
}

template <class V>
void launch_mean_any_to(const V* w, int64_t ld_v, int64_t cols_v, int n, int64_t groups, float div,
                        V* out, int64_t out_ld_v, cudaStream_t s) {
  dim3 grid(static_cast<unsigned>((cols_v + kThreads - 1) / kThreads),
            static_cast<unsigned>(groups));
  launch_pdl(k_mean_any_to<V>, grid, dim3(kThreads), 0, s, false, 1, w, ld_v, cols_v, n, div, out,
             out_ld_v);
}

bool mean_pow2_dispatch(int log, float4* w, int64_t ld_v, int64_t cols_v, int64_t groups,
                        cudaStream_t s) {
  switch (log) {
    case 1: launch_mean_pow2<1>(w, ld_v, cols_v, groups, s); return true;
    case 2: launch_mean_pow2<2>(w, ld_v, cols_v, groups, s); return true;
    case 3: launch_mean_pow2<3>(w, ld_v, cols_v, groups, s); return true;
    case 4: launch_mean_pow2<4>(w, ld_v, cols_v, groups, s); return true;
    case 5: launch_mean_pow2<5>(w, ld_v, cols_v, groups, s); return true;
    case 6: launch_mean_pow2<6>(w, ld_v, cols_v, groups, s); return true;
    case 7: launch_mean_pow2<7>(w, ld_v, cols_v, groups, s); return true;
    default: return false;
  }
}

template <int LOGQ, int LOGS, int LOGG>
void launch_lg(const float4* src, int64_t src_ld_v, float4* w, int64_t ld_v, int64_t cols_v,
               cudaStream_t s) {
  if constexpr (LOGG >= 1) {
    if (split_rows(cols_v, 1)) {
      dim3 grid(static_cast<unsigned>((cols_v + 127) / 128));
      launch_pdl(k_local_global_pow2_split<LOGQ, LOGS, LOGG>, grid, dim3(128, 2), 0, s, false, 1, src,
                 src_ld_v, w, ld_v, cols_v);
      return;
    }
  }
  dim3 grid(static_cast<unsigned>((cols_v + kThreads - 1) / kThreads));
  launch_pdl(k_local_global_pow2<LOGQ, LOGS, LOGG>, grid, dim3(kThreads), 0, s, false, 1, src,
             src_ld_v, w, ld_v, cols_v);
}

template <int LOGQ, int LOGS>
bool lg_dispatch_g(int logg, const float4* src, int64_t src_ld_v, float4* w, int64_t ld_v,
                   int64_t cols_v, cudaStream_t s) {
  if constexpr (LOGQ <= LOGS) {
#define HA_LG(G_) \
    if constexpr (LOGS + G_ <= 7) \
      if (logg == G_) { launch_lg<LOGQ, LOGS, G_>(src, src_ld_v, w, ld_v, cols_v, s); return true; }
    HA_LG(0) HA_LG(1) HA_LG(2) HA_LG(3) HA_LG(4) HA_LG(5) HA_LG(6)
#undef HA_LG
  }
  return false;
}

template <int LOGQ>
bool lg_dispatch_s(int logs, int logg, const float4* src, int64_t src_ld_v, float4* w,
                   int64_t ld_v, int64_t cols_v, cudaStream_t s) {
  switch (logs) {
    case 1: return lg_dispatch_g<LOGQ, 1>(logg, src, src_ld_v, w, ld_v, cols_v, s);
    case 2: return lg_dispatch_g<LOGQ, 2>(logg, src, src_ld_v, w, ld_v, cols_v, s);
    case 3: return lg_dispatch_g<LOGQ, 3>(logg, src, src_ld_v, w, ld_v, cols_v, s);
    case 4: return lg_dispatch_g<LOGQ, 4>(logg, src, src_ld_v, w, ld_v, cols_v, s);
    case 5: return lg_dispatch_g<LOGQ, 5>(logg, src, src_ld_v, w, ld_v, cols_v, s);
    default: return false;
  }
}

bool lg_dispatch(int logq, int logs, int logg, const float4* src, int64_t src_ld_v, float4* w,
                 int64_t ld_v, int64_t cols_v, cudaStream_t s) {
  switch (logq) {
    case 0: return lg_dispatch_s<0>(logs, logg, src, src_ld_v, w, ld_v, cols_v, s);
    case 1: return lg_dispatch_s<1>(logs, logg, src, src_ld_v, w, ld_v, cols_v, s);
    case 2: return lg_dispatch_s<2>(logs, logg, src, src_ld_v, w, ld_v, cols_v, s);
    default: return false;
  }
}

template <class V>
void launch_mean_any(V* w, int64_t ld_v, int64_t cols_v, int n, int64_t groups,
                     cudaStream_t s) {
  dim3 grid(static_cast<unsigned>((cols_v + kThreads - 1) / kThreads),
            static_cast<unsigned>(groups));
  launch_pdl(k_mean_any<V>, grid, dim3(kThreads), 0, s, false, 1, w, ld_v, cols_v, n);
}

template <class V>
void launch_lg_any(const V* src, int64_t src_ld_v, int n, V* w, int64_t ld_v, int64_t cols_v, int S,
                   int G, cudaStream_t s) {
  dim3 grid(static_cast<unsigned>((cols_v + kThreads - 1) / kThreads));
  launch_pdl(k_local_global_any<V>, grid, dim3(kThreads), 0, s, false, 1, src, src_ld_v, n, w, ld_v,
             cols_v, S, G);
}

}  // namespace

// Vector path for the 16-byte aligned bulk, scalar generic path for the tail.
static bool vec_ok(const float* w, int64_t ld) {
  return (reinterpret_cast<uintptr_t>(w) % 16 == 0) && (ld % 4 == 0);
}

cudaError_t launch_group_mean(float* w, int64_t P, int64_t n, int64_t D, int64_t ld,
                              cudaStream_t s) {
  if (D == 0 || n == 1) return cudaSuccess;   // a mean of one row is that row
  const int64_t groups = P / n;
  int64_t head = 0;
  if (vec_ok(w, ld) && D >= 4) {
    head = D & ~int64_t(3);
    float4* w4 = reinterpret_cast<float4*>(w);
    const int log = ilog2_exact(n);
    if (!(log >= 1 && mean_pow2_dispatch(log, w4, ld / 4, head / 4, groups, s)))
      launch_mean_any<float4>(w4, ld / 4, head / 4, static_cast<int>(n), groups, s);
  }
  if (head < D) launch_mean_any<float>(w + head, ld, D - head, static_cast<int>(n), groups, s);
  return cudaGetLastError();
}

cudaError_t launch_group_mean_to(const float* w, int64_t P, int64_t n, int64_t D, int64_t ld,
                                 float* out, cudaStream_t s) {
  return launch_group_sum_mean_to(w, P, n, D, ld, static_cast<float>(n), out, ld, s);
}

cudaError_t launch_group_sum_mean_to(const float* w, int64_t rows, int64_t n, int64_t D, int64_t ld,
                                     float div, float* out, int64_t out_ld, cudaStream_t s) {
  if (D == 0) return cudaSuccess;
  const int64_t groups = rows / n;
  int64_t head = 0;
  if (vec_ok(w, ld) && vec_ok(out, out_ld) && D >= 4) {
    head = D & ~int64_t(3);
    const float4* w4 = reinterpret_cast<const float4*>(w);
    float4* o4 = reinterpret_cast<float4*>(out);
    const int log = ilog2_exact(n);
    if (!(log >= 0 && mean_pow2_to_dispatch(log, w4, ld / 4, head / 4, groups, div, o4, out_ld / 4, s)))
      launch_mean_any_to<float4>(w4, ld / 4, head / 4, static_cast<int>(n), groups, div, o4,
                                 out_ld / 4, s);
  }
  if (head < D)
    launch_mean_any_to<float>(w + head, ld, D - head, static_cast<int>(n), groups, div, out + head,
                              out_ld, s);
  return cudaGetLastError();
}

cudaError_t launch_local_global_mean(float* w, int64_t P, int64_t S, int64_t D, int64_t ld,
                                     cudaStream_t s) {
  if (D == 0) return cudaSuccess;
  // S = 1: the local average is the identity, so the pair is one global mean.
  // (S = P is NOT shortcut: the literal second pass re-averages P equal copies.)
  if (S == 1) return launch_group_mean(w, P, P, D, ld, s);
  return launch_local_global_from_groups(w, ld, 1, w, P, S, D, ld, s);
}

cudaError_t launch_local_global_from_groups(const float* src, int64_t src_ld, int64_t Q, float* w,
                                            int64_t P, int64_t S, int64_t D, int64_t ld,
                                            cudaStream_t s) {
  if (D == 0) return cudaSuccess;
  const int64_t G = P / S, n = S / Q;
  int64_t head = 0;
  if (vec_ok(w, ld) && vec_ok(src, src_ld) && D >= 4) {
    head = D & ~int64_t(3);
    float4* w4 = reinterpret_cast<float4*>(w);
    const float4* s4 = reinterpret_cast<const float4*>(src);
    const int logq = ilog2_exact(Q), logs = ilog2_exact(S), logg = ilog2_exact(G);
    if (!(logq >= 0 && logs >= 1 && logg >= 0 &&
          lg_dispatch(logq, logs, logg, s4, src_ld / 4, w4, ld / 4, head / 4, s)))
      launch_lg_any<float4>(s4, src_ld / 4, static_cast<int>(n), w4, ld / 4, head / 4,
                            static_cast<int>(S), static_cast<int>(G), s);
  }
  if (head < D)
    launch_lg_any<float>(src + head, src_ld, static_cast<int>(n), w + head, ld, D - head,
                         static_cast<int>(S), static_cast<int>(G), s);
  return cudaGetLastError();
}

}  // namespace ha
