// The small last layer (at most 16 classes) of the learner step, on warp-level bf16
// MMAs (Algorithm 1 inner loop, Sec. 3.1).  head_body runs one learner (or one
// feature slice of it, the CTAs of a cluster sharing the learner) on 256 threads:
//   1. Zp = H W_q^T over the features [k0, k0 + F) (classes padded to 16);
//   2. Z = sum of the slices' Zp (clustered: read through distributed shared memory
//      and added in slice order) + b_L, then the softmax cross-entropy gradient
//      g[b][c] = (softmax(Z[b])_c - [c == y_b]) / B; slice 0 updates b_L and the loss;
//   3. for its features, with W before its update: dW = g_q^T H, dH = g_q W_q,
//      dZ_{L-1} = dH [H > 0] (bf16), b_{L-1} -= lr sum_b dZ_{L-1}, W -= lr dW (fp32).
// (_q = rounded to bf16.)  For a one-layer model the input rows are read from X.
#pragma once
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace ha {
namespace head {

constexpr int kHeadThreads = 256;
constexpr int kHeadMaxC = 16;
constexpr int kHeadClusterMax = 8;
constexpr int kHeadClusterPref = 4;           // CTAs per learner when 8 per learner would not fit in one wave
constexpr int kHeadPad = 8;                   // bf16 row padding: ldmatrix rows hit distinct banks
constexpr int kGA = kHeadMaxC + 8;            // g_q   [b][c] row stride (bf16)
constexpr int kGT = 64 + 8;                   // g_q^T [c][b] row stride (bf16)

__device__ __forceinline__ const __nv_bfloat16* head_row(const HeadArgs& a, int j, int b) {
  if (a.x_rows) return a.H + (static_cast<int64_t>(j) * a.N + (a.row0 + b) % a.N) * a.in;
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

// ---- warp-level MMA helpers (m16n8k16, bf16 inputs, fp32 accumulators)
__device__ __forceinline__ void ldsm_x4(const void* p, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void ldsm_x2(const void* p, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void ldsm_x2_t(const void* p, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Row of the 16x16 A tile whose address lane l supplies to ldsm_x4, and its column
// offset (0 or 8): the four 8x8 matrices are (rows 0-7 | 8-15) x (cols 0-7 | 8-15).
__device__ __forceinline__ int a_row(int l) { return ((l >> 3) & 1) * 8 + (l & 7); }
__device__ __forceinline__ int a_col(int l) { return (l >> 4) * 8; }




// Shared memory needed by head_body for slices of F features.
__host__ __device__ inline int head_body_smem(int F, int Bn) {
  return (Bn + kHeadMaxC) * (F + kHeadPad) * 2 + 3 * 64 * kHeadMaxC * 4 + 64 * 4 + 64 * 4 +
         kHeadMaxC * 4 + 64 * kGA * 2 + kHeadMaxC * kGT * 2;
}

// Slice s (F features wide) of learner j on threads t = 0..255, the S slices being
// the CTAs of a cluster; sync() is a barrier over the 256 threads.
template <int CT, class Sync>
__device__ __forceinline__ void head_body(const HeadArgs& a, uint8_t* smem, int j, int s, int S,
                                          int F, int t, Sync sync) {
  const int C = CT > 0 ? CT : a.C, B = a.B, Bn = a.Bn, in = a.in;
  const int warp = t >> 5, lane = t & 31;
  const int FP = F + kHeadPad;
  const int k0 = s * F, kc = min(F, in - k0);          // kc > 0, a multiple of 64
  __nv_bfloat16* hs = reinterpret_cast<__nv_bfloat16*>(smem);   // [Bn][FP]  H slice
  __nv_bfloat16* wq = hs + Bn * FP;                             // [16][FP]  W_q slice
  float* zp = reinterpret_cast<float*>(wq + kHeadMaxC * FP);    // [64][16]  partial logits
  float* zz = zp + 64 * kHeadMaxC;                              // [64][16]  logits
  float* gs = zz + 64 * kHeadMaxC;                              // [64][16]  CE gradient (fp32)
  float* rl = gs + 64 * kHeadMaxC;                              // [64]      per-sample loss
  float* bls = rl + 64;                                         // [16]      b_L before update
  int* ys = reinterpret_cast<int*>(bls + kHeadMaxC);            // [64]      labels
  __nv_bfloat16* gqa = reinterpret_cast<__nv_bfloat16*>(ys + 64);           // [64][kGA]  g_q
  __nv_bfloat16* gqt = gqa + 64 * kGA;                                      // [16][kGT]  g_q^T
  float* W = a.W + static_cast<int64_t>(j) * a.ld;                 // written
  float* bL = a.bias + static_cast<int64_t>(j) * a.ld;
  const int64_t src_row = static_cast<int64_t>(j / a.src_div) * a.ld; // read
  const float* Wr = a.W_src + src_row;

  // ---- 1. stage the slice (padding rows zero) and the labels, form the partial logits
  const int vpr = kc / 8;                                       // 16-byte vectors per H row
  for (int idx = t; idx < Bn * vpr; idx += kHeadThreads) {
    const int b = idx / vpr, v = idx - b * vpr;
    uint4 x = make_uint4(0, 0, 0, 0);
    if (b < B) x = *reinterpret_cast<const uint4*>(head_row(a, j, b) + k0 + v * 8);
    *reinterpret_cast<uint4*>(hs + b * FP + v * 8) = x;
  }
  const int wpr = kc / 4;                                       // float4s per W row
  for (int idx = t; idx < kHeadMaxC * wpr; idx += kHeadThreads) {
    const int c = idx / wpr, v = idx - c * wpr;
    float4 w = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c < C) w = *reinterpret_cast<const float4*>(Wr + static_cast<int64_t>(c) * in + k0 + v * 4);
    __nv_bfloat162* d = reinterpret_cast<__nv_bfloat162*>(wq + c * FP + v * 4);
    d[0] = __floats2bfloat162_rn(w.x, w.y);
    d[1] = __floats2bfloat162_rn(w.z, w.w);
  }
  if (t < kHeadMaxC) bls[t] = t < C ? a.bias_src[src_row + t] : 0.f;
  if (t >= 64 && t < 64 + B) ys[t - 64] = a.y[static_cast<int64_t>(j) * a.N + (a.row0 + t - 64) % a.N];
  sync();
  for (int tile = warp; tile < (Bn / 16) * 2; tile += kHeadThreads / 32) {
    const int mt = tile >> 1, nt = tile & 1;                    // 16 samples x 8 classes
    float d[4] = {0.f, 0.f, 0.f, 0.f};
    for (int k = 0; k < kc; k += 16) {
      uint32_t af[4], b0, b1;
      ldsm_x4(hs + (mt * 16 + a_row(lane)) * FP + k + a_col(lane), af);
      ldsm_x2(wq + (nt * 8 + (lane & 7)) * FP + k + ((lane >> 3) & 1) * 8, b0, b1);
      mma16816(d, af, b0, b1);
    }
    const int r = mt * 16 + (lane >> 2), cc = nt * 8 + (lane & 3) * 2;
    zp[r * kHeadMaxC + cc] = d[0];
    zp[r * kHeadMaxC + cc + 1] = d[1];
    zp[(r + 8) * kHeadMaxC + cc] = d[2];
    zp[(r + 8) * kHeadMaxC + cc + 1] = d[3];
  }

  // ---- 2. full logits (partials added in slice order), softmax cross-entropy
  cluster_sync();
  for (int pr = t; pr < B * C; pr += kHeadThreads) {
    const int b = pr / C, c = pr - b * C;
    float v[kHeadClusterMax];
#pragma unroll
    for (int r = 0; r < kHeadClusterMax; ++r)
      v[r] = r < S ? ld_cluster(zp + b * kHeadMaxC + c, r) : 0.f;
    float z = 0.f;
#pragma unroll
    for (int r = 0; r < kHeadClusterMax; ++r)
      if (r < S) z = __fadd_rn(z, v[r]);
    zz[b * kHeadMaxC + c] = __fadd_rn(z, bls[c]);
  }
  cluster_sync();   // every CTA is done with the partials
  // Softmax cross-entropy: 16 lanes per sample (one per class slot), max and sum of
  // exponentials by butterflies over the sample's lanes.
  for (int b0 = 0; b0 < Bn; b0 += kHeadThreads / kHeadMaxC) {
    const int b = b0 + (t >> 4), c = t & (kHeadMaxC - 1);
    const bool live = b < B && c < C;
    const float z = live ? zz[b * kHeadMaxC + c] : -INFINITY;
    float m = z;
#pragma unroll
    for (int off = 1; off < kHeadMaxC; off <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    const float e = live ? expf(z - m) : 0.f;
    float sum = e;
#pragma unroll
    for (int off = 1; off < kHeadMaxC; off <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    float g = 0.f;
    if (live) {
      const int yb = ys[b];
      g = __fdiv_rn(__fsub_rn(__fdiv_rn(e, sum), c == yb ? 1.f : 0.f), static_cast<float>(B));
      if (c == yb) rl[b] = logf(sum) + m - z;
    }
    if (b < Bn) {
      gs[b * kHeadMaxC + c] = g;
      const __nv_bfloat16 q = __float2bfloat16_rn(g);
      gqa[b * kGA + c] = q;
      gqt[c * kGT + b] = q;
    }
  }
  sync();
  if (s == 0) {
    if (t < C) {
      float db = 0.f;
      for (int b = 0; b < B; ++b) db = __fadd_rn(db, gs[b * kHeadMaxC + t]);
      bL[t] = __fsub_rn(bls[t], __fmul_rn(a.lr, db));
    } else if (t == 32) {
      float l = 0.f;
      for (int b = 0; b < B; ++b) l += rl[b];
      a.loss[j] = l / B;
    }
  }

  // ---- 3. backward of the slice: one 8-feature column block per warp at a time.
  // The fp32 values this lane updates are loaded first; the MMAs hide their latency.
  auto load_upd = [&](int nt, float2 (&w32)[2], float2& bp32) {
    const int f = nt * 8 + (lane & 3) * 2;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = (lane >> 2) + 8 * h;
      w32[h] = c < C ? *reinterpret_cast<const float2*>(Wr + static_cast<int64_t>(c) * in + k0 + f)
                     : make_float2(0.f, 0.f);
    }
    bp32 = (a.has_dx && lane < 4)
               ? *reinterpret_cast<const float2*>(a.bias_prev_src + src_row + k0 + f)
               : make_float2(0.f, 0.f);
  };
  float2 nw32[2], nbp32;
  if (warp < kc / 8) load_upd(warp, nw32, nbp32);
  for (int nt = warp; nt < kc / 8; nt += kHeadThreads / 32) {
    const int f = nt * 8 + (lane & 3) * 2;                      // this lane's two features
    float2 w32[2] = {nw32[0], nw32[1]}, bp32 = nbp32;
    if (nt + kHeadThreads / 32 < kc / 8) load_upd(nt + kHeadThreads / 32, nw32, nbp32);  // next block
    // dW^T block: rows c (16), cols f; K = samples
    float dw[4] = {0.f, 0.f, 0.f, 0.f};
    for (int kb = 0; kb < Bn; kb += 16) {
      uint32_t af[4], b0, b1;
      ldsm_x4(gqt + a_row(lane) * kGT + kb + a_col(lane), af);
      ldsm_x2_t(hs + (kb + (lane & 15)) * FP + nt * 8, b0, b1);
      mma16816(dw, af, b0, b1);
    }
    // dH block: rows b, cols f; K = classes (16)
    float db0 = 0.f, db1 = 0.f;
    uint32_t wb0, wb1;
    ldsm_x2_t(wq + (lane & 15) * FP + nt * 8, wb0, wb1);
    for (int mt = 0; mt < Bn / 16; ++mt) {
      uint32_t af[4];
      ldsm_x4(gqa + (mt * 16 + a_row(lane)) * kGA + a_col(lane), af);
      float dh[4] = {0.f, 0.f, 0.f, 0.f};
      mma16816(dh, af, wb0, wb1);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int b = mt * 16 + (lane >> 2) + 8 * h;
        const __nv_bfloat162 hv = *reinterpret_cast<const __nv_bfloat162*>(hs + b * FP + f);
        const float z0 = __bfloat162float(hv.x) > 0.f ? dh[2 * h] : 0.f;
        const float z1 = __bfloat162float(hv.y) > 0.f ? dh[2 * h + 1] : 0.f;
        if (a.has_dx && b < B) {
          db0 = __fadd_rn(db0, z0);
          db1 = __fadd_rn(db1, z1);
          *reinterpret_cast<__nv_bfloat162*>(
              a.dz_prev + (static_cast<int64_t>(j) * Bn + b) * a.pitch_in + k0 + f) =
              __floats2bfloat162_rn(z0, z1);
        }
      }
    }
    if (a.has_dx) {
      // b_{L-1} for the two features: sum over the 8 row groups (fixed butterfly)
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        db0 = __fadd_rn(db0, __shfl_xor_sync(0xffffffffu, db0, off));
        db1 = __fadd_rn(db1, __shfl_xor_sync(0xffffffffu, db1, off));
      }
      if (lane < 4)
        *reinterpret_cast<float2*>(a.bias_prev + static_cast<int64_t>(j) * a.ld + k0 + f) =
            make_float2(__fsub_rn(bp32.x, __fmul_rn(a.lr, db0)),
                        __fsub_rn(bp32.y, __fmul_rn(a.lr, db1)));
    }
    // W -= lr dW for the valid classes
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = (lane >> 2) + 8 * h;
      if (c < C)
        *reinterpret_cast<float2*>(W + static_cast<int64_t>(c) * in + k0 + f) =
            make_float2(__fsub_rn(w32[h].x, __fmul_rn(a.lr, dw[2 * h])),
                        __fsub_rn(w32[h].y, __fmul_rn(a.lr, dw[2 * h + 1])));
    }
  }
}

}  // namespace head
}  // namespace ha
