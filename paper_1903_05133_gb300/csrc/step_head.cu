// Last layer of the learner step when it is small (at most 16 classes), on CUDA
// cores (Algorithm 1 inner loop, Sec. 3.1).  The layer holds only C x d_{L-1}
// weights, far too few to feed a tensor-core tile; bf16 operands, fp32
// accumulation in a fixed order.  Two kernels:
//   k_head_fwd  one CTA per learner.  Z[b][c] = sum_k H[b][k] W_q[c][k] + b_L[c]
//               (warps own samples, lanes split k, butterfly sum), the CE gradient
//               g[b][c] = (softmax(Z[b])_c - [c == y_b]) / B into a scratch buffer
//               (fp32 and bf16-rounded), b_L -= lr * sum_b g, and the loss.
//   k_head_bwd  one CTA per (128-feature slice, learner), one thread per feature k:
//               with W before its update, dW[c][k] = sum_b g_q[b][c] H[b][k],
//               dH[b][k] = sum_c g_q[b][c] W_q[c][k], dZ_{L-1}[b][k] = dH [H > 0]
//               (bf16 and transposed copies, fp32 sum into b_{L-1}[k]), then
//               W[c][k] -= lr * dW[c][k].
// (_q = rounded to bf16).  The class count is a template parameter so no work is
// issued for absent classes.  For a one-layer model the input rows are read from X.
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"

namespace ha {
namespace {

constexpr int kFwdThreads = 512;
constexpr int kFwdWarps = kFwdThreads / 32;
constexpr int kKC = 512;                      // input features staged per chunk
constexpr int kRowsPerWarp = 4;               // B <= 64 = kFwdWarps * kRowsPerWarp
constexpr int kHeadMaxC = 16;
constexpr int kBwdCols = 128;                 // features per backward CTA

__device__ __forceinline__ float bf16r(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}

__device__ __forceinline__ const __nv_bfloat16* head_row(const HeadArgs& a, int j, int b) {
  if (a.x_rows) return a.H + (static_cast<int64_t>(j) * a.N + (a.t * a.B + b) % a.N) * a.in;
  return a.H + (static_cast<int64_t>(j) * a.Bn + b) * a.pitch_in;
}

// C: compile-time class count (0 = runtime count up to kHeadMaxC).
template <int CT>
__global__ void __launch_bounds__(kFwdThreads, 1) k_head_fwd(const HeadArgs a) {
  constexpr int CM = CT > 0 ? CT : kHeadMaxC;
  extern __shared__ __align__(16) uint8_t smem[];
  const int C = CT > 0 ? CT : a.C, B = a.B, in = a.in;
  __nv_bfloat16* wq = reinterpret_cast<__nv_bfloat16*>(smem);                       // [C][in]
  __nv_bfloat16* hs = wq + static_cast<size_t>(C) * in;                              // [64][kKC]
  float* rl = reinterpret_cast<float*>(hs + 64 * kKC);                               // [B]
  float* gsum = rl + 64;                                                             // [64][CM]
  float* bls = gsum + 64 * CM;                                                       // [CM]
  int* ys = reinterpret_cast<int*>(bls + CM);                                        // [64]
  const int j = blockIdx.x, t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const float* W = a.W + static_cast<int64_t>(j) * a.ld;
  float* bL = a.bias + static_cast<int64_t>(j) * a.ld;
  if (t < B) ys[t] = a.y[static_cast<int64_t>(j) * a.N + (a.t * B + t) % a.N];
  if (t < C) bls[t] = bL[t];

  for (int e = t * 4; e < C * in; e += kFwdThreads * 4) {
    const float4 v = *reinterpret_cast<const float4*>(W + e);
    reinterpret_cast<__nv_bfloat162*>(wq + e)[0] = __floats2bfloat162_rn(v.x, v.y);
    reinterpret_cast<__nv_bfloat162*>(wq + e)[1] = __floats2bfloat162_rn(v.z, v.w);
  }
  float acc[kRowsPerWarp][CM];
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r)
#pragma unroll
    for (int c = 0; c < CM; ++c) acc[r][c] = 0.f;
  for (int k0 = 0; k0 < in; k0 += kKC) {
    const int kc = min(kKC, in - k0);
    const int vpr = kc / 8;
    if (k0 > 0) __syncthreads();
    for (int idx = t; idx < B * vpr; idx += kFwdThreads) {
      const int b = idx / vpr, v = idx - b * vpr;
      *reinterpret_cast<uint4*>(hs + b * kKC + v * 8) =
          *reinterpret_cast<const uint4*>(head_row(a, j, b) + k0 + v * 8);
    }
    __syncthreads();
    for (int kk = 2 * lane; kk < kc; kk += 64) {
      float2 hv[kRowsPerWarp];
#pragma unroll
      for (int r = 0; r < kRowsPerWarp; ++r) {
        const int b = warp + r * kFwdWarps;
        hv[r] = b < B ? __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(hs + b * kKC + kk))
                      : make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int c = 0; c < CM; ++c) {
        if (CT > 0 || c < C) {
          const float2 wv =
              __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(wq + c * in + k0 + kk));
#pragma unroll
          for (int r = 0; r < kRowsPerWarp; ++r)
            acc[r][c] = fmaf(hv[r].y, wv.y, fmaf(hv[r].x, wv.x, acc[r][c]));
        }
      }
    }
  }
  const float fB = static_cast<float>(B);
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    const int b = warp + r * kFwdWarps;
    if (b >= B) continue;                       // warp-uniform
#pragma unroll
    for (int c = 0; c < CM; ++c) {
      if (CT > 0 || c < C) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc[r][c] += __shfl_xor_sync(0xffffffffu, acc[r][c], off);
      }
    }
    float z = -INFINITY;
#pragma unroll
    for (int c = 0; c < CM; ++c)
      if (c == lane && (CT > 0 || c < C)) z = __fadd_rn(acc[r][c], bls[c]);
    float m = z;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    const float e = lane < C ? expf(z - m) : 0.f;
    float s = e;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    const int yb = ys[b];
    const float zy = __shfl_sync(0xffffffffu, z, yb & 31);
    if (lane < C) {
      const float p = __fdiv_rn(e, s);
      const float g = __fdiv_rn(__fsub_rn(p, lane == yb ? 1.f : 0.f), fB);
      gsum[b * CM + lane] = g;
      a.gq[(static_cast<int64_t>(j) * a.Bn + b) * kHeadMaxC + lane] = bf16r(g);
    }
    if (lane == 0) rl[b] = logf(s) + m - zy;
  }
  __syncthreads();
  if (t < C) {
    float db = 0.f;
    for (int b = 0; b < B; ++b) db = __fadd_rn(db, gsum[b * CM + t]);
    bL[t] = __fsub_rn(bls[t], __fmul_rn(a.lr, db));
  }
  if (t == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += rl[b];
    a.loss[j] = l / B;
  }
}

template <int CT>
__global__ void __launch_bounds__(kBwdCols) k_head_bwd(const HeadArgs a) {
  constexpr int CM = CT > 0 ? CT : kHeadMaxC;
  __shared__ float gq[64 * kHeadMaxC];
  const int C = CT > 0 ? CT : a.C, B = a.B, in = a.in;
  const int j = blockIdx.y, t = threadIdx.x, k = blockIdx.x * kBwdCols + t;
  for (int e = t; e < B * kHeadMaxC; e += kBwdCols)
    gq[e] = a.gq[static_cast<int64_t>(j) * a.Bn * kHeadMaxC + e];
  __syncthreads();
  if (k >= in) return;
  float* W = a.W + static_cast<int64_t>(j) * a.ld;
  float w32[CM], wk[CM], dw[CM];
#pragma unroll
  for (int c = 0; c < CM; ++c) {
    w32[c] = (CT > 0 || c < C) ? W[c * in + k] : 0.f;
    wk[c] = bf16r(w32[c]);
    dw[c] = 0.f;
  }
  float db = 0.f;
  for (int b0 = 0; b0 < a.Bn; b0 += 8) {
    float h[8];
#pragma unroll
    for (int q = 0; q < 8; ++q)
      h[q] = b0 + q < B ? __bfloat162float(head_row(a, j, b0 + q)[k]) : 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int b = b0 + q;
      if (b < B) {
        float dh = 0.f;
#pragma unroll
        for (int c = 0; c < CM; ++c) {
          if (CT > 0 || c < C) {
            const float g = gq[b * kHeadMaxC + c];
            dw[c] = fmaf(g, h[q], dw[c]);
            dh = fmaf(g, wk[c], dh);
          }
        }
        if (a.has_dx) {
          const float dz = h[q] > 0.f ? dh : 0.f;
          db = __fadd_rn(db, dz);
          a.dz_prev[(static_cast<int64_t>(j) * a.Bn + b) * a.pitch_in + k] = __float2bfloat16_rn(dz);
        }
      }
    }
  }
#pragma unroll
  for (int c = 0; c < CM; ++c)
    if (CT > 0 || c < C) W[c * in + k] = __fsub_rn(w32[c], __fmul_rn(a.lr, dw[c]));
  if (a.has_dx) {
    float* bp = a.bias_prev + static_cast<int64_t>(j) * a.ld + k;
    *bp = __fsub_rn(*bp, __fmul_rn(a.lr, db));
  }
}

int fwd_smem_bytes(int C, int in) {
  return C * in * 2 + 64 * kKC * 2 + 64 * 4 + 64 * kHeadMaxC * 4 + kHeadMaxC * 4 + 64 * 4;
}

template <int CT>
cudaError_t launch_pair(const HeadArgs& a, int P, cudaStream_t s) {
  k_head_fwd<CT><<<P, kFwdThreads, fwd_smem_bytes(a.C, a.in), s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  dim3 grid((a.in + kBwdCols - 1) / kBwdCols, P);
  k_head_bwd<CT><<<grid, kBwdCols, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

int head_scratch_floats(int P, int Bn) { return P * Bn * kHeadMaxC; }

bool head_supported(int C, int in, int B) {
  return C <= kHeadMaxC && in % 64 == 0 && B <= 64 && fwd_smem_bytes(C, in) <= 200 * 1024;
}

cudaError_t head_configure() {
  cudaError_t e = cudaFuncSetAttribute(k_head_fwd<10>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       200 * 1024);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_head_fwd<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
}

cudaError_t launch_head(const HeadArgs& a, int P, cudaStream_t s) {
  return a.C == 10 ? launch_pair<10>(a, P, s) : launch_pair<0>(a, P, s);
}

}  // namespace ha
