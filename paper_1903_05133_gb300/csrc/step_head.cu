// Last layer of the learner step when it is small (at most 16 classes): forward,
// softmax cross-entropy, and backward of that layer in one kernel, one CTA per
// learner (Algorithm 1 inner loop, Sec. 3.1).  The layer holds only C x d_{L-1}
// weights, far too few to feed a tensor-core tile, and running it as three
// launches costs more in latency than in work; here it is CUDA-core FMAs on
// bf16 operands with fp32 accumulation in a fixed order:
//   phase 1  Z[b][c] = sum_k H[b][k] W_q[c][k] + b_L[c]   (each warp owns a few
//            samples; lanes split k, butterfly sum), then the CE gradient
//            g[b][c] = (softmax(Z[b])_c - [c == y_b]) / B and the loss
//   phase 2  b_L[c] -= lr * sum_b g[b][c]
//   phase 3  per input feature k (thread per k): with W before its update,
//            dW[c][k] = sum_b g_q[b][c] H[b][k], dH[b][k] = sum_c g_q[b][c] W_q[c][k],
//            dZ_{L-1}[b][k] = dH [H > 0] (bf16 and transposed copies, fp32 sum into
//            b_{L-1}[k]), then W[c][k] -= lr * dW[c][k]
// (_q = rounded to bf16).  The activations are staged in shared memory chunk by
// chunk with 16-byte loads.  For a one-layer model the input rows are read from X.
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"

namespace ha {
namespace {

constexpr int kHeadThreads = 512;
constexpr int kHeadWarps = kHeadThreads / 32;
constexpr int kKC = 512;                      // input features staged per chunk
constexpr int kRowsPerWarp = 4;               // B <= 64 = kHeadWarps * kRowsPerWarp
constexpr int kHeadMaxC = 16;                 // classes held in registers per sample

__device__ __forceinline__ float bf16r(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}

template <int CMAX>
__global__ void __launch_bounds__(kHeadThreads, 1) k_head(const HeadArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int C = a.C, B = a.B, in = a.in;
  __nv_bfloat16* wq = reinterpret_cast<__nv_bfloat16*>(smem);                       // [C][in]
  __nv_bfloat16* hs = wq + static_cast<size_t>(C) * in;                              // [64][kKC]
  float* gs = reinterpret_cast<float*>(hs + 64 * kKC);                               // [B][C]
  float* gq = gs + 64 * CMAX;                                                        // [B][C]
  float* rl = gq + 64 * CMAX;                                                        // [B]
  const int j = blockIdx.x, t = threadIdx.x, warp = t >> 5, lane = t & 31;
  float* W = a.W + static_cast<int64_t>(j) * a.ld;
  float* bL = a.bias + static_cast<int64_t>(j) * a.ld;

  // bf16 copy of W_L for the forward and for dX (the weights before the update)
  for (int e = t * 4; e < C * in; e += kHeadThreads * 4) {
    const float4 v = *reinterpret_cast<const float4*>(W + e);
    reinterpret_cast<__nv_bfloat162*>(wq + e)[0] = __floats2bfloat162_rn(v.x, v.y);
    reinterpret_cast<__nv_bfloat162*>(wq + e)[1] = __floats2bfloat162_rn(v.z, v.w);
  }
  auto row = [&](int b) -> const __nv_bfloat16* {
    if (a.x_rows) return a.H + (static_cast<int64_t>(j) * a.N + (a.t * B + b) % a.N) * in;
    return a.H + (static_cast<int64_t>(j) * a.Bn + b) * a.pitch_in;
  };
  // Stage rows 0..B-1, features [k0, k0 + kKC) into hs with 16-byte loads.
  auto stage = [&](int k0) {
    const int kc = min(kKC, in - k0);
    const int vec_per_row = kc / 8;
    for (int idx = t; idx < B * vec_per_row; idx += kHeadThreads) {
      const int b = idx / vec_per_row, v = idx - b * vec_per_row;
      *reinterpret_cast<uint4*>(hs + b * kKC + v * 8) =
          *reinterpret_cast<const uint4*>(row(b) + k0 + v * 8);
    }
  };

  // ---- phase 1: logits.  Warp w owns samples w, w + 16, ...; each lane sums its
  // k pairs for all of them, then a butterfly per (sample, class).
  float acc[kRowsPerWarp][CMAX];
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r)
#pragma unroll
    for (int c = 0; c < CMAX; ++c) acc[r][c] = 0.f;
  for (int k0 = 0; k0 < in; k0 += kKC) {
    __syncthreads();
    stage(k0);
    __syncthreads();
    const int kc = min(kKC, in - k0);
    for (int kk = 2 * lane; kk < kc; kk += 64) {
      float2 hv[kRowsPerWarp];
#pragma unroll
      for (int r = 0; r < kRowsPerWarp; ++r) {
        const int b = warp + r * kHeadWarps;
        hv[r] = b < B ? __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(hs + b * kKC + kk))
                      : make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int c = 0; c < CMAX; ++c) {
        if (c < C) {
          const float2 wv =
              __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(wq + c * in + k0 + kk));
#pragma unroll
          for (int r = 0; r < kRowsPerWarp; ++r)
            acc[r][c] = fmaf(hv[r].y, wv.y, fmaf(hv[r].x, wv.x, acc[r][c]));
        }
      }
    }
  }
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    const int b = warp + r * kHeadWarps;
#pragma unroll
    for (int c = 0; c < CMAX; ++c) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) acc[r][c] += __shfl_xor_sync(0xffffffffu, acc[r][c], off);
    }
    if (b >= B) continue;
    // CE gradient of sample b: lane c holds class c
    float z = -INFINITY;
#pragma unroll
    for (int c = 0; c < CMAX; ++c)
      if (c == lane && c < C) z = __fadd_rn(acc[r][c], bL[c]);
    float m = z;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    const float e = lane < C ? expf(z - m) : 0.f;
    float s = e;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    const int yb = a.y[static_cast<int64_t>(j) * a.N + (a.t * B + b) % a.N];
    const float zy = __shfl_sync(0xffffffffu, z, yb & 31);
    if (lane < C) {
      const float p = __fdiv_rn(e, s);
      const float g = __fdiv_rn(__fsub_rn(p, lane == yb ? 1.f : 0.f), static_cast<float>(B));
      gs[b * C + lane] = g;
      gq[b * C + lane] = bf16r(g);
    }
    if (lane == 0) rl[b] = logf(s) + m - zy;
  }
  __syncthreads();

  // ---- phase 2: last bias and the loss
  if (t < C) {
    float db = 0.f;
    for (int b = 0; b < B; ++b) db = __fadd_rn(db, gs[b * C + t]);
    bL[t] = __fsub_rn(bL[t], __fmul_rn(a.lr, db));
  }
  if (t == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += rl[b];
    a.loss[j] = l / B;
  }

  // ---- phase 3: per input feature k, dW and dX with the old weights, then the update
  for (int k0 = 0; k0 < in; k0 += kKC) {
    __syncthreads();
    stage(k0);
    __syncthreads();
    const int kc = min(kKC, in - k0);
    for (int kk = t; kk < kc; kk += kHeadThreads) {
      const int k = k0 + kk;
      float wk[CMAX], dw[CMAX];
#pragma unroll
      for (int c = 0; c < CMAX; ++c) {
        wk[c] = c < C ? __bfloat162float(wq[c * in + k]) : 0.f;
        dw[c] = 0.f;
      }
      float db = 0.f;
      for (int b0 = 0; b0 < a.Bn; b0 += 8) {
        uint32_t pk[4];
#pragma unroll
        for (int q = 0; q < 8; q += 2) {
          float dz2[2];
#pragma unroll
          for (int e2 = 0; e2 < 2; ++e2) {
            const int b = b0 + q + e2;
            float dz = 0.f;
            if (b < B) {
              const float h = __bfloat162float(hs[b * kKC + kk]);
              float dh = 0.f;
#pragma unroll
              for (int c = 0; c < CMAX; ++c) {
                if (c < C) {
                  const float g = gq[b * C + c];
                  dw[c] = fmaf(g, h, dw[c]);
                  dh = fmaf(g, wk[c], dh);
                }
              }
              if (a.has_dx) {
                dz = h > 0.f ? dh : 0.f;
                db = __fadd_rn(db, dz);
                a.dz_prev[(static_cast<int64_t>(j) * a.Bn + b) * a.pitch_in + k] = __float2bfloat16_rn(dz);
              }
            }
            dz2[e2] = dz;
          }
          const __nv_bfloat162 pr = __floats2bfloat162_rn(dz2[0], dz2[1]);
          pk[q / 2] = *reinterpret_cast<const uint32_t*>(&pr);
        }
        if (a.has_dx)
          *reinterpret_cast<uint4*>(a.dzt_prev + (static_cast<int64_t>(j) * in + k) * a.Kp + b0) =
              make_uint4(pk[0], pk[1], pk[2], pk[3]);
      }
#pragma unroll
      for (int c = 0; c < CMAX; ++c)
        if (c < C) W[c * in + k] = __fsub_rn(W[c * in + k], __fmul_rn(a.lr, dw[c]));
      if (a.has_dx) {
        float* bp = a.bias_prev + static_cast<int64_t>(j) * a.ld + k;
        *bp = __fsub_rn(*bp, __fmul_rn(a.lr, db));
      }
    }
  }
}

}  // namespace

int head_smem_bytes(int C, int in, int B) {
  (void)B;
  return C * in * 2 + 64 * kKC * 2 + 2 * 64 * kHeadMaxC * 4 + 64 * 4 + 16;
}

bool head_supported(int C, int in, int B) {
  return C <= kHeadMaxC && in % 64 == 0 && B <= 64 && head_smem_bytes(C, in, B) <= 220 * 1024;
}

cudaError_t head_configure() {
  return cudaFuncSetAttribute(k_head<kHeadMaxC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              220 * 1024);
}

cudaError_t launch_head(const HeadArgs& a, int P, cudaStream_t s) {
  k_head<kHeadMaxC><<<P, kHeadThreads, head_smem_bytes(a.C, a.in, a.B), s>>>(a);
  return cudaGetLastError();
}

}  // namespace ha
