// Last layer of the learner step when it is small (at most 16 classes), on CUDA
// cores (Algorithm 1 inner loop, Sec. 3.1).  The layer holds only C x d_{L-1}
// weights, far too few to feed a tensor-core tile; bf16 operands, fp32
// accumulation in a fixed order.  One kernel, one thread-block cluster of S CTAs
// per learner, CTA s owning the input features [s*F, (s+1)*F):
//   1. partial logits over its features: Zp_s[b][c] = sum_k H[b][k] W_q[c][k]
//      (k ascending);
//   2. after a cluster barrier every CTA reads all S partials through distributed
//      shared memory and adds them in slice order: Z = sum_s Zp_s + b_L, then the
//      softmax cross-entropy gradient g[b][c] = (softmax(Z[b])_c - [c == y_b]) / B
//      (recomputed identically in every CTA); the first CTA updates b_L -= lr sum_b g
//      and writes the loss;
//   3. one thread per feature k of its slice: with W before its update,
//      dW[c][k] = sum_b g_q[b][c] H[b][k], dH[b][k] = sum_c g_q[b][c] W_q[c][k],
//      dZ_{L-1}[b][k] = dH [H > 0] (bf16, fp32 sum into b_{L-1}[k]), then
//      W[c][k] -= lr * dW[c][k].
// (_q = rounded to bf16).  The class count is a template parameter so no work is
// issued for absent classes.  For a one-layer model the input rows are read from X.
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace ha {
namespace {

constexpr int kHeadThreads = 128;
constexpr int kHeadMaxC = 16;
constexpr int kHeadClusterMax = 8;
constexpr int kHeadPad = 8;                   // bf16 row padding (spreads banks)

__device__ __forceinline__ float bf16r(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}

__device__ __forceinline__ const __nv_bfloat16* head_row(const HeadArgs& a, int j, int b) {
  if (a.x_rows) return a.H + (static_cast<int64_t>(j) * a.N + (a.t * a.B + b) % a.N) * a.in;
  return a.H + (static_cast<int64_t>(j) * a.Bn + b) * a.pitch_in;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}
// The float at the same shared-memory offset in CTA `rank` of this cluster.
__device__ __forceinline__ float ld_cluster(const float* p, int rank) {
  const uint32_t la = static_cast<uint32_t>(__cvta_generic_to_shared(p));
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(la), "r"(rank));
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(ra) : "memory");
  return v;
}

// Features per CTA: a multiple of 64, at least 128, and at most 8 CTAs per learner.
__host__ __device__ inline int head_slice(int in) {
  const int f = ((in + kHeadClusterMax - 1) / kHeadClusterMax + 63) / 64 * 64;
  return f < 128 ? 128 : f;
}
__host__ __device__ inline int head_smem_bytes(int in, int Bn) {
  return (Bn + kHeadMaxC) * (head_slice(in) + kHeadPad) * 2 + 3 * 64 * kHeadMaxC * 4 + 64 * 4;
}

template <int CT>
__global__ void __launch_bounds__(kHeadThreads) k_head(const HeadArgs a) {
  constexpr int CM = CT > 0 ? CT : kHeadMaxC;
  extern __shared__ __align__(16) uint8_t smem[];
  grid_dep_wait();
  const int C = CT > 0 ? CT : a.C, B = a.B, in = a.in;
  const int S = gridDim.x, s = blockIdx.x, j = blockIdx.y, t = threadIdx.x;
  const int F = head_slice(in), FP = F + kHeadPad;
  const int k0 = s * F, kc = min(F, in - k0);          // kc > 0, a multiple of 64
  __nv_bfloat16* hs = reinterpret_cast<__nv_bfloat16*>(smem);   // [Bn][FP]  H slice
  __nv_bfloat16* wq = hs + a.Bn * FP;                           // [16][FP]  W_q slice
  float* zp = reinterpret_cast<float*>(wq + kHeadMaxC * FP);    // [64][16]  partial logits
  float* zz = zp + 64 * kHeadMaxC;                              // [64][16]  logits
  float* gs = zz + 64 * kHeadMaxC;                              // [64][16]  CE gradient
  float* rl = gs + 64 * kHeadMaxC;                              // [64]      per-sample loss
  float* W = a.W + static_cast<int64_t>(j) * a.ld;
  float* bL = a.bias + static_cast<int64_t>(j) * a.ld;

  // ---- 1. stage the slice and form the partial logits
  const int vpr = kc / 8;                                       // 16-byte vectors per H row
  for (int idx = t; idx < B * vpr; idx += kHeadThreads) {
    const int b = idx / vpr, v = idx - b * vpr;
    *reinterpret_cast<uint4*>(hs + b * FP + v * 8) =
        *reinterpret_cast<const uint4*>(head_row(a, j, b) + k0 + v * 8);
  }
  const int wpr = kc / 4;                                       // float4s per W row
  for (int idx = t; idx < C * wpr; idx += kHeadThreads) {
    const int c = idx / wpr, v = idx - c * wpr;
    const float4 w = *reinterpret_cast<const float4*>(W + static_cast<int64_t>(c) * in + k0 + v * 4);
    __nv_bfloat162* d = reinterpret_cast<__nv_bfloat162*>(wq + c * FP + v * 4);
    d[0] = __floats2bfloat162_rn(w.x, w.y);
    d[1] = __floats2bfloat162_rn(w.z, w.w);
  }
  __syncthreads();
  for (int pr = t; pr < B * C; pr += kHeadThreads) {
    const int b = pr / C, c = pr - b * C;
    const __nv_bfloat162* hp = reinterpret_cast<const __nv_bfloat162*>(hs + b * FP);
    const __nv_bfloat162* wp = reinterpret_cast<const __nv_bfloat162*>(wq + c * FP);
    float acc = 0.f;
    for (int k = 0; k < kc / 2; ++k) {
      const float2 h = __bfloat1622float2(hp[k]), w = __bfloat1622float2(wp[k]);
      acc = fmaf(h.y, w.y, fmaf(h.x, w.x, acc));
    }
    zp[b * kHeadMaxC + c] = acc;
  }
  cluster_sync();

  // ---- 2. full logits (partials added in slice order), bias read before its update
  for (int pr = t; pr < B * C; pr += kHeadThreads) {
    const int b = pr / C, c = pr - b * C;
    float z = 0.f;
    for (int r = 0; r < S; ++r) z = __fadd_rn(z, ld_cluster(zp + b * kHeadMaxC + c, r));
    zz[b * kHeadMaxC + c] = __fadd_rn(z, bL[c]);
  }
  cluster_sync();   // every CTA is done with the partials and with b_L
  if (t < B) {
    const float* z = zz + t * kHeadMaxC;
    const int yb = a.y[static_cast<int64_t>(j) * a.N + (a.t * B + t) % a.N];
    float m = -INFINITY;
#pragma unroll
    for (int c = 0; c < CM; ++c)
      if (CT > 0 || c < C) m = fmaxf(m, z[c]);
    float e[CM], sum = 0.f;
#pragma unroll
    for (int c = 0; c < CM; ++c) {
      e[c] = (CT > 0 || c < C) ? expf(z[c] - m) : 0.f;
      sum += e[c];
    }
    const float fB = static_cast<float>(B);
#pragma unroll
    for (int c = 0; c < CM; ++c)
      if (CT > 0 || c < C)
        gs[t * kHeadMaxC + c] = __fdiv_rn(__fsub_rn(__fdiv_rn(e[c], sum), c == yb ? 1.f : 0.f), fB);
    rl[t] = logf(sum) + m - z[yb];
  }
  __syncthreads();
  if (s == 0) {
    if (t < C) {
      float db = 0.f;
      for (int b = 0; b < B; ++b) db = __fadd_rn(db, gs[b * kHeadMaxC + t]);
      bL[t] = __fsub_rn(bL[t], __fmul_rn(a.lr, db));
    } else if (t == 32) {
      float l = 0.f;
      for (int b = 0; b < B; ++b) l += rl[b];
      a.loss[j] = l / B;
    }
  }

  // ---- 3. backward of the slice, one thread per feature
  for (int kk = t; kk < kc; kk += kHeadThreads) {
    const int k = k0 + kk;
    float w32[CM], wk[CM], dw[CM];
#pragma unroll
    for (int c = 0; c < CM; ++c) {
      w32[c] = (CT > 0 || c < C) ? W[static_cast<int64_t>(c) * in + k] : 0.f;
      wk[c] = bf16r(w32[c]);
      dw[c] = 0.f;
    }
    float db = 0.f;
    for (int b = 0; b < B; ++b) {
      const float h = __bfloat162float(hs[b * FP + kk]);
      float dh = 0.f;
#pragma unroll
      for (int c = 0; c < CM; ++c) {
        if (CT > 0 || c < C) {
          const float g = bf16r(gs[b * kHeadMaxC + c]);
          dw[c] = fmaf(g, h, dw[c]);
          dh = fmaf(g, wk[c], dh);
        }
      }
      if (a.has_dx) {
        const float dz = h > 0.f ? dh : 0.f;
        db = __fadd_rn(db, dz);
        a.dz_prev[(static_cast<int64_t>(j) * a.Bn + b) * a.pitch_in + k] = __float2bfloat16_rn(dz);
      }
    }
#pragma unroll
    for (int c = 0; c < CM; ++c)
      if (CT > 0 || c < C) W[static_cast<int64_t>(c) * in + k] = __fsub_rn(w32[c], __fmul_rn(a.lr, dw[c]));
    if (a.has_dx) {
      float* bp = a.bias_prev + static_cast<int64_t>(j) * a.ld + k;
      *bp = __fsub_rn(*bp, __fmul_rn(a.lr, db));
    }
  }
}

template <int CT>
cudaError_t launch_cluster(const HeadArgs& a, int P, cudaStream_t s) {
  const int S = (a.in + head_slice(a.in) - 1) / head_slice(a.in);
  return launch_pdl(k_head<CT>, dim3(S, P), dim3(kHeadThreads), head_smem_bytes(a.in, a.Bn), s,
                    false, S, a);
}

}  // namespace

bool head_supported(int C, int in, int B) {
  return C <= kHeadMaxC && in % 64 == 0 && B <= 64 && head_smem_bytes(in, 64) <= 200 * 1024;
}

cudaError_t head_configure() {
  cudaError_t e = cudaFuncSetAttribute(k_head<10>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       200 * 1024);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_head<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
}

cudaError_t launch_head(const HeadArgs& a, int P, cudaStream_t s) {
  return a.C == 10 ? launch_cluster<10>(a, P, s) : launch_cluster<0>(a, P, s);
}

}  // namespace ha
