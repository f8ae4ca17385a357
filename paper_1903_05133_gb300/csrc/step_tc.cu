// bf16 learner step on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// One local SGD step of Algorithm 1 (Sec. 3.1) for every learner of a ReLU MLP:
// forward Z_l = H_{l-1} W_l^T + b_l, softmax cross-entropy gradient, backward
// dH_{l-1} = dZ_l W_l (with W_l before its update) and W_l -= lr * dZ_l^T H_{l-1}.
// The fp32 master weights W_l [P][out][in] are streamed from HBM by TMA and
// rounded to bf16 in shared memory by the CTA itself; MMAs accumulate in fp32 in
// tensor memory.  All operands use the K-major 128-byte-swizzle layout.
//
// Because the per-learner batch B (<= 64) is far below the MMA's M, every GEMM
// is issued "swap-AB": the weight tile supplies M = 128 rows and the batch is
// the N extent.
//
// Forward kernel  (grid: out tiles of 128 x P learners)
//   warp 4: TMA producer - fp32 W tile [128 x 64] + bf16 H tile [Bn x 64] per stage
//   warps 0-3: round W to bf16 into the swizzled A tile; then the epilogue
//              (bias, ReLU, bf16 H and H^T of the next layer, or fp32 logits)
//   warp 5: TMEM allocation + single-thread MMA issue, Z^T[128 x Bn] += W H^T
// Backward kernel (grid: in tiles of 128 x P learners), one pass over W_l:
//   per out-chunk of 64 rows: TMA loads fp32 W [64 x 128], dZ [Bn x 64],
//   dZ^T [64 x 64]; warps 0-3 write W^T (bf16) for the dX MMA; MMA warp issues
//     dH^T[128 x Bn] += W^T(chunk) dZ^T(chunk)          (accumulated over chunks)
//     dW^T[128 x 64]  = H^T[128 x B] dZ(chunk)           (double-buffered in TMEM)
//   warps 0-3 then update the fp32 chunk in shared memory (w - lr * dw, separate
//   rounded multiply and subtract) and TMA-store it back: W is read once and
//   written once per step.  Finally dZ_{l-1} = dH * [H_{l-1} > 0] and the bias
//   b_{l-1} -= lr * sum_b dZ_{l-1}.
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace ha {
namespace {

constexpr int kStages = 3;
constexpr int kThreads = 192;          // warps 0-3 convert/epilogue, 4 TMA, 5 MMA
constexpr int kConv = 128;

// ------------------------------------------------------------------ forward
// Persistent stream-K forward.  The work of one layer is a list of units
// u = (tile, chunk): tile = (learner j, 128 output features), chunk = 64 input
// features.  CTA g of G owns the contiguous units [g*U/G, (g+1)*U/G), so every SM
// streams the same number of chunks and the TMA ring runs straight across tile
// boundaries.  A tile whose chunks are spread over several CTAs is finished by
// the contributor that arrives last: it sums the published partial accumulators
// in CTA order (deterministic) and runs the epilogue.
// Warps 0-7 convert the fp32 weight tiles to bf16 and own the accumulator rows:
// warp w serves TMEM lanes 32*(w%4).., and the two warps on the same lanes split
// the batch columns in interleaved 16-column blocks (group w/4 takes blocks
// 2m + w/4).  Warp 8 issues TMA, warp 9 the MMAs.
// Shared memory: two TMA rings, the fp32 weight tiles (released by the converter
// warps as soon as they have read them, so conversion and MMA latency stay out of
// the weight stream) and the bf16 batch tiles (released by the MMA); a
// double-buffered bf16 A tile the converter warps fill for the MMA; and (fused
// cross-entropy only) a staging area for the epilogue.  The MMA of chunk i waits
// for batch tile i, which is reloaded only after the MMA nh chunks earlier, so the
// batch ring takes all the shared memory left (its tiles are Bn x 128 bytes).
constexpr int kFwdConv = 256;
constexpr int kFwdThreads = kFwdConv + 64;
constexpr int kFwdWRingMax = 5, kFwdHRingMax = 8;
constexpr int kFwdWf32 = 128 * 64 * 4;                 // 32 KB fp32 W tile
constexpr int kFwdWbf = 128 * 64 * 2;                  // 16 KB bf16 A tile (x2)
constexpr int kFwdSmemMax = 227 * 1024;
constexpr int kXentSmem = (2 * 128 * 65 + 4 * 64) * 4; // logits, gradients, statistics
// The tensor core's fp32 accumulation loses precision roughly in proportion to the
// number of MMAs chained into one accumulator, so the accumulator is promoted:
// every kSegChunks chunks (16 MMAs) the partial sum is folded into fp32 registers
// with IEEE adds, in chunk order, while the MMAs continue in the other TMEM buffer.
constexpr int kSegChunks = 4;
constexpr uint32_t kFwdTmemCols = 128;   // two accumulator buffers of 64 columns
constexpr int kFwdHidden = 0, kFwdXent = 2;   // TcFwdArgs::mode (1 = logits)

// Layout: W ring | A tiles | epilogue staging (mode 2) | batch ring | barriers.
__host__ __device__ constexpr int fwd_wring(int mode) { return mode == 2 ? 3 : 5; }
__host__ __device__ constexpr int fwd_h_off(int mode) {
  return fwd_wring(mode) * kFwdWf32 + 2 * kFwdWbf + (mode == 2 ? kXentSmem : 0);
}
__host__ __device__ constexpr int fwd_hring(int mode, int Bn) {
  return (kFwdSmemMax - 1024 - 512 - fwd_h_off(mode)) / (Bn * 128) < kFwdHRingMax
             ? (kFwdSmemMax - 1024 - 512 - fwd_h_off(mode)) / (Bn * 128)
             : kFwdHRingMax;
}
__host__ __device__ constexpr int fwd_bar_off(int mode, int Bn) {
  return fwd_h_off(mode) + fwd_hring(mode, Bn) * Bn * 128;
}
__host__ __device__ constexpr int fwd_smem(int mode, int Bn) { return fwd_bar_off(mode, Bn) + 512 + 1024; }
static_assert(fwd_hring(2, 64) >= 3 && fwd_hring(0, 64) >= 4 && fwd_smem(2, 64) <= kFwdSmemMax &&
                  fwd_smem(0, 64) <= kFwdSmemMax && fwd_smem(0, 16) <= kFwdSmemMax,
              "forward shared-memory plan");

// Bounded wait whose outcome is made uniform across the warp, so that a warp never
// reaches a .sync.aligned tcgen05 instruction with only some of its lanes.
__device__ __forceinline__ bool wait_warp(uint64_t* bar, uint32_t parity, int* err) {
  const bool r = mbar_wait(bar, parity, err);
  return __all_sync(0xffffffffu, r);
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  return reinterpret_cast<uint8_t*>((a + 1023) & ~uintptr_t(1023));
}

// A barrier of the converter threads on an mbarrier, bounded like every other
// wait.  `phase` counts this thread's uses.
struct GroupSync {
  uint64_t* bar;
  uint32_t phase;
  int* err;
  __device__ __forceinline__ bool operator()() {
    mbar_arrive(bar);
    const bool ok = mbar_wait(bar, phase & 1, err);
    ++phase;
    return ok;
  }
};

// Epilogue of the last layer when every class fits in one 128-row tile: the
// softmax cross-entropy gradient straight from the accumulator (no logits
// round trip).  Row r = class, group gr holds the column blocks 2m + gr of it
// (blocks of 16 samples) in acc[16m ..].  Work is then spread over all converter
// threads: column statistics, all class x sample gradients, per-class bias sums
// in sample order.
__device__ __forceinline__ void xent_epilogue(const TcFwdArgs& a, int j, int t, int r, int gr,
                                              const float* acc, float* sm, GroupSync& gsync) {
  constexpr int ZP = 65;
  float* zs = sm;                  // [128][ZP] logits, class-major
  float* gs = sm + 128 * ZP;       // [128][ZP] gradients
  float* stat = gs + 128 * ZP;     // max[64], sum[64], label[64], loss[64]
  const int C = a.out, B = a.B;
  if (r < C) {
#pragma unroll
    for (int m = 0; m < 2; ++m) {
      const int cb = (2 * m + gr) * 16;
      if (cb < a.Bn) {
#pragma unroll
        for (int q = 0; q < 16; ++q) zs[r * ZP + cb + q] = acc[16 * m + q];
      }
    }
  }
  gsync();
  if (t < B) {
    float m = -INFINITY;
    for (int c = 0; c < C; ++c) m = fmaxf(m, zs[c * ZP + t]);
    float s = 0.f;
    for (int c = 0; c < C; ++c) s += expf(zs[c * ZP + t] - m);
    const int yb = a.y[static_cast<int64_t>(j) * a.N + (a.t * B + t) % a.N];
    stat[t] = m;
    stat[64 + t] = s;
    stat[128 + t] = __int_as_float(yb);
    stat[192 + t] = logf(s) + m - zs[yb * ZP + t];
  }
  gsync();
  const float fB = static_cast<float>(B);
  for (int e = t; e < C * B; e += kFwdConv) {
    const int c = e / B, b = e - c * B;
    const float p = __fdiv_rn(expf(zs[c * ZP + b] - stat[b]), stat[64 + b]);
    const float g = __fdiv_rn(__fsub_rn(p, __float_as_int(stat[128 + b]) == c ? 1.f : 0.f), fB);
    gs[c * ZP + b] = g;
    a.dz_out[(static_cast<int64_t>(j) * a.Bn + b) * a.pitch_out + c] = __float2bfloat16_rn(g);
  }
  gsync();
  if (t == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += stat[192 + b];
    a.loss[j] = l / B;
  }
  if (t < C) {
    float db = 0.f;
    for (int b0 = 0; b0 < a.Bn; b0 += 8) {
      uint32_t pk[4];
#pragma unroll
      for (int q = 0; q < 8; q += 2) {
        const int b = b0 + q;
        const float g0 = b < B ? gs[t * ZP + b] : 0.f;
        const float g1 = b + 1 < B ? gs[t * ZP + b + 1] : 0.f;
        if (b < B) db = __fadd_rn(db, g0);
        if (b + 1 < B) db = __fadd_rn(db, g1);
        pk[q / 2] = pack_bf16x2(g0, g1);
      }
      *reinterpret_cast<uint4*>(a.dzt_out + (static_cast<int64_t>(j) * C + t) * a.Kp + b0) =
          make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
    float* bp = const_cast<float*>(a.bias) + static_cast<int64_t>(j) * a.ld + t;
    *bp = __fsub_rn(*bp, __fmul_rn(a.lr, db));
  }
  gsync();   // the staging area is reused by the next tile
}

// First unit of CTA g when U units are split over G CTAs (G <= U).
__device__ __forceinline__ int unit_begin(int g, int U, int G) {
  return static_cast<int>(static_cast<int64_t>(g) * U / G);
}
// The CTA that owns unit u.
__device__ __forceinline__ int cta_of(int u, int U, int G) {
  int g = static_cast<int>(static_cast<int64_t>(u) * G / U);
  while (g + 1 < G && unit_begin(g + 1, U, G) <= u) ++g;
  while (g > 0 && unit_begin(g, U, G) > u) --g;
  return g;
}

__global__ void __launch_bounds__(kFwdThreads, 1)
    k_tc_forward(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_h,
                 const TcFwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x, G = gridDim.x;
  const int nk = (a.in + 63) / 64;
  const int U = a.n_tiles * nk;
  const int u0 = unit_begin(g, U, G), u1 = unit_begin(g + 1, U, G);
  const int n_local = u1 - u0;
  const int nw = fwd_wring(a.mode), nh = fwd_hring(a.mode, a.Bn);
  const int hbytes = a.Bn * 128;
  const int h_row0 = a.x_direct ? a.x_row0 : 0;           // batch rows inside the H (or X) map
  const int tile0 = u0 / nk, c0 = u0 - tile0 * nk;         // first unit's tile and chunk
  uint8_t* wbf_base = smem + nw * kFwdWf32;
  uint8_t* xent_sm = wbf_base + 2 * kFwdWbf;
  uint8_t* h_base = smem + fwd_h_off(a.mode);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + fwd_bar_off(a.mode, a.Bn));
  uint64_t* wempty = wfull + kFwdWRingMax;  // weight tile read by every converter warp
  uint64_t* hfull = wempty + kFwdWRingMax;
  uint64_t* hempty = hfull + kFwdHRingMax;  // batch tile consumed by the MMA
  uint64_t* conv = hempty + kFwdHRingMax;   // [2] A tile written
  uint64_t* wfree = conv + 2;              // [2] A tile consumed by the MMA
  uint64_t* accf = wfree + 2;              // [2] accumulator segment complete
  uint64_t* accr = accf + 2;               // [2] accumulator segment drained
  uint64_t* gbar = accr + 2;               // converter-group barrier
  uint64_t* done = gbar + 1;
  uint64_t* pready = done + 1;             // this CTA's split-tile partial is written
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pready + 1);
  auto wf = [&](int s) { return smem + s * kFwdWf32; };
  auto hb = [&](int s) { return h_base + s * hbytes; };
  auto wb = [&](int b) { return wbf_base + b * kFwdWbf; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFwdWRingMax; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], kFwdConv / 32);   // one arrival per converter warp
    }
    for (int s = 0; s < kFwdHRingMax; ++s) {
      mbar_init(&hfull[s], 1);
      mbar_init(&hempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&conv[b], kFwdConv / 32);
      mbar_init(&wfree[b], 1);
      mbar_init(&accf[b], 1);
      mbar_init(&accr[b], kFwdConv);
    }
    mbar_init(gbar, kFwdConv);
    mbar_init(done, 1);
    mbar_init(pready, kFwdConv / 32);
    fence_barrier_init();
  }
  if (warp == 9) {
    tmem_alloc(tmem_slot, kFwdTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 8) {
    // Lane 0 streams the weight tiles, lane 1 the batch tiles: each ring runs as
    // far ahead as its own consumer allows.
    if (lane < 2) {
      const bool wside = lane == 0;
      const int n = wside ? nw : nh;
      uint64_t* fullb = wside ? wfull : hfull;
      uint64_t* emptyb = wside ? wempty : hempty;
      if (wside) tma_prefetch_desc(&tm_w);
      else tma_prefetch_desc(&tm_h);
      int issued = 0, tau = tile0, c = c0;
      for (int i = 0; i < n_local; ++i) {
        const int j = tau / a.o_tiles, ot = tau - j * a.o_tiles;
        const int s = i % n;
        if (i >= n && !mbar_wait(&emptyb[s], ((i / n) - 1) & 1, a.err)) break;
        if (wside) {
          mbar_arrive_expect_tx(&fullb[s], kFwdWf32);
          tma_load_3d(wf(s), &tm_w, &fullb[s], c * 64, ot * 128, j);
        } else {
          mbar_arrive_expect_tx(&fullb[s], a.Bn * 128);
          tma_load_3d(hb(s), &tm_h, &fullb[s], c * 64, h_row0, j);
        }
        issued = i + 1;
        if (++c == nk) { c = 0; ++tau; }
      }
      // Every load issued must have landed before the CTA may exit.
      for (int i = issued - n > 0 ? issued - n : 0; i < issued; ++i)
        mbar_wait(&fullb[i % n], (i / n) & 1, a.err);
    } else if (lane == 2 && c0 != 0 && n_local > 0) {
      // The first tile began in an earlier CTA, which finishes it: once the
      // converter warps have written this CTA's partial, publish it (release
      // order makes the partial visible before the count).
      if (mbar_wait(pready, 0, a.err)) red_release_add(a.counters + tile0, 1);
    }
  } else if (warp == 9) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(128, a.Bn);
      int q = -1, c = c0, p = 0;        // accumulator segment index, chunk, position in run
      for (int i = 0; i < n_local; ++i) {
        const bool tlast = i == n_local - 1 || c == nk - 1;
        const bool first = p % kSegChunks == 0, last = tlast || p % kSegChunks == kSegChunks - 1;
        const int sh = i % nh, b = i & 1;
        if (first) ++q;
        const int ab = q & 1;
        if (first && q >= 2 && !mbar_wait(&accr[ab], ((q >> 1) - 1) & 1, a.err)) break;
        if (!mbar_wait(&conv[b], (i >> 1) & 1, a.err)) break;
        if (!mbar_wait(&hfull[sh], (i / nh) & 1, a.err)) break;
        tc_fence_after();
        const uint64_t ad = umma_desc_sw128(smem_u32(wb(b)));
        const uint64_t bd = umma_desc_sw128(smem_u32(hb(sh)));
        const uint32_t d = tmem + 64 * ab;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (!first || kk > 0) ? 1u : 0u);
        tc_commit(&hempty[sh]);
        tc_commit(&wfree[b]);
        if (last) tc_commit(&accf[ab]);
        ++p;
        if (++c == nk) { c = 0; p = 0; }
      }
      tc_commit(done);
      mbar_wait(done, 0, a.err);   // no MMA may be in flight at teardown
    }
  } else {
    // ---- warps 0-7: fp32 -> bf16 A tile (and H_0^T for the first layer), the
    // accumulator drains and the tile epilogues
    const int t = threadIdx.x;
    const int r = t & 127, gr = t >> 7;                    // accumulator row, column group
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    GroupSync gsync{gbar, 0, a.err};
    float acc[32];                                         // blocks 2m + gr, m = 0, 1
#pragma unroll
    for (int q = 0; q < 32; ++q) acc[q] = 0.f;
    int qc = -1, drained = 0;
    // Fold segment `drained` into the registers (warp-uniform; contains tcgen05.ld).
    auto drain = [&]() -> bool {
      const int ab = drained & 1;
      if (!wait_warp(&accf[ab], (drained >> 1) & 1, a.err)) return false;
      tc_fence_after();
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb < a.Bn) {
          float v[16];
          tmem_ld16(tbase + 64 * ab + cb, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v[q]);
        }
      }
      tc_fence_before();
      mbar_arrive(&accr[ab]);
      ++drained;
      return true;
    };
    // Tile tau is complete in this CTA's registers (or in this CTA's part of it).
    // A tile split over CTAs g_first .. g_last is finished by g_first, the CTA that
    // holds its first chunk and, in stream-K order, reaches it last; every other
    // contributor writes its partial to its own slot and publishes it without
    // waiting.  The finisher adds the partials in CTA order.
    auto tile_end = [&](int tau, bool whole, float bias) -> bool {
      const int j = tau / a.o_tiles, ot = tau - j * a.o_tiles;
      if (!whole) {
        if (tau * nk < u0) {
          float* mine = a.part + (static_cast<int64_t>(g) * 128 + r) * a.Bn;
#pragma unroll
          for (int m = 0; m < 2; ++m) {
            const int cb = (2 * m + gr) * 16;
            if (cb < a.Bn) {
#pragma unroll
              for (int q = 0; q < 16; q += 4)
                __stcg(reinterpret_cast<float4*>(mine + cb + q),
                       make_float4(acc[16 * m + q], acc[16 * m + q + 1], acc[16 * m + q + 2],
                                   acc[16 * m + q + 3]));
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(pready);
#pragma unroll
          for (int q = 0; q < 32; ++q) acc[q] = 0.f;
          return true;
        }
        const int g_last = cta_of((tau + 1) * nk - 1, U, G);
        if (t == 0) {
          const bool ok = spin_acquire_eq(a.counters + tau, g_last - g, a.err);
          if (ok) a.counters[tau] = 0;   // ready for the next launch
        }
        if (!gsync()) return false;
        for (int gg = g + 1; gg <= g_last; ++gg) {
          const float* src = a.part + (static_cast<int64_t>(gg) * 128 + r) * a.Bn;
#pragma unroll
          for (int m = 0; m < 2; ++m) {
            const int cb = (2 * m + gr) * 16;
            if (cb < a.Bn) {
#pragma unroll
              for (int q = 0; q < 16; q += 4) {
                const float4 v = __ldcg(reinterpret_cast<const float4*>(src + cb + q));
                acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v.x);
                acc[16 * m + q + 1] = __fadd_rn(acc[16 * m + q + 1], v.y);
                acc[16 * m + q + 2] = __fadd_rn(acc[16 * m + q + 2], v.z);
                acc[16 * m + q + 3] = __fadd_rn(acc[16 * m + q + 3], v.w);
              }
            }
          }
        }
      }
      const int o = ot * 128 + r;
      const bool valid = o < a.out;
      if (a.mode == kFwdXent) {
#pragma unroll
        for (int q = 0; q < 32; ++q) acc[q] = __fadd_rn(acc[q], bias);
        xent_epilogue(a, j, t, r, gr, acc, reinterpret_cast<float*>(xent_sm), gsync);
      } else if (valid) {
#pragma unroll
        for (int m = 0; m < 2; ++m) {
          const int cb = (2 * m + gr) * 16;
          if (cb >= a.Bn) break;
          if (a.mode == kFwdHidden) {
            uint32_t pk[8];
#pragma unroll
            for (int q = 0; q < 16; q += 2) {
              const float h0 = fmaxf(__fadd_rn(acc[16 * m + q], bias), 0.f);
              const float h1 = fmaxf(__fadd_rn(acc[16 * m + q + 1], bias), 0.f);
              const bool in0 = cb + q < a.B, in1 = cb + q + 1 < a.B;
              pk[q / 2] = pack_bf16x2(in0 ? h0 : 0.f, in1 ? h1 : 0.f);
              const __nv_bfloat162 hh = *reinterpret_cast<__nv_bfloat162*>(&pk[q / 2]);
              if (in0) a.h_out[(static_cast<int64_t>(j) * a.Bn + cb + q) * a.pitch_out + o] = hh.x;
              if (in1) a.h_out[(static_cast<int64_t>(j) * a.Bn + cb + q + 1) * a.pitch_out + o] = hh.y;
            }
            uint4* dst = reinterpret_cast<uint4*>(a.ht_out + (static_cast<int64_t>(j) * a.out + o) * a.Kp + cb);
            dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          } else {
#pragma unroll
            for (int q = 0; q < 16; ++q)
              if (cb + q < a.B)
                a.z_out[(static_cast<int64_t>(j) * a.B + cb + q) * a.out + o] = __fadd_rn(acc[16 * m + q], bias);
          }
        }
      }
#pragma unroll
      for (int q = 0; q < 32; ++q) acc[q] = 0.f;
      return true;
    };
    bool ok = true;
    int tau = tile0, c = c0, p = 0;
    float tbias = 0.f;                 // bias of row r of the current tile, loaded early
    for (int i = 0; i < n_local && ok; ++i) {
      const int j = tau / a.o_tiles, ot = tau - j * a.o_tiles;
      const bool tlast = i == n_local - 1 || c == nk - 1;
      if (p == 0) {
        const int o = ot * 128 + r;
        tbias = o < a.out ? a.bias[static_cast<int64_t>(j) * a.ld + o] : 0.f;
      }
      const int sw = i % nw, sh = i % nh, bb = i & 1;
      if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
      if (i >= 2 && !wait_warp(&wfree[bb], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
      const float* src = reinterpret_cast<const float*>(wf(sw));
      uint8_t* dst = wb(bb);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const int f = t + kFwdConv * v;      // group of 8 floats in the [128][64] fp32 tile
        const int row = f >> 3, k = (f & 7) * 8;
        const float4 x0 = *reinterpret_cast<const float4*>(src + row * 64 + k);
        const float4 x1 = *reinterpret_cast<const float4*>(src + row * 64 + k + 4);
        *reinterpret_cast<uint4*>(dst + sw128_offset(row, k)) =
            make_uint4(pack_bf16x2(x0.x, x0.y), pack_bf16x2(x0.z, x0.w), pack_bf16x2(x1.x, x1.y),
                       pack_bf16x2(x1.z, x1.w));
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&wempty[sw]);   // the fp32 tile is no longer needed
      if (a.x_direct && ot == 0) {
        // H_0^T[k][b] for this chunk's 64 features, from the staged batch tile
        // (rows b >= B of the tile belong to later samples and are written as 0).
        if (!wait_warp(&hfull[sh], (i / nh) & 1, a.err)) { ok = false; break; }
        const uint8_t* hs = hb(sh);
        const int kk = t & 63;
        const int k = c * 64 + kk;
        if (k < a.in) {
          for (int b0 = (t >> 6) * 8; b0 < a.Bn; b0 += 32) {
            uint32_t pk[4];
#pragma unroll
            for (int q = 0; q < 8; q += 2) {
              const int b = b0 + q;
              const uint16_t lo = b < a.B ? *reinterpret_cast<const uint16_t*>(hs + sw128_offset(b, kk)) : 0;
              const uint16_t hi = b + 1 < a.B ? *reinterpret_cast<const uint16_t*>(hs + sw128_offset(b + 1, kk)) : 0;
              pk[q / 2] = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
            }
            *reinterpret_cast<uint4*>(a.ht0_out + (static_cast<int64_t>(j) * a.in + k) * a.Kp + b0) =
                make_uint4(pk[0], pk[1], pk[2], pk[3]);
          }
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&conv[bb]);
      if (p % kSegChunks == 0) ++qc;
      if (tlast) {
        while (ok && drained <= qc)
          if (!drain()) ok = false;
        if (ok) {
          const bool whole = (tau != tile0 || c0 == 0) && c == nk - 1;
          ok = __all_sync(0xffffffffu, tile_end(tau, whole, tbias));
        }
      } else if (p % kSegChunks == kSegChunks - 1 && qc >= 1 && drained < qc) {
        if (!drain()) ok = false;   // one segment behind the MMAs
      }
      ++p;
      if (++c == nk) { c = 0; p = 0; ++tau; }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kFwdTmemCols);
  }
}

// ------------------------------------------------------------------ backward
constexpr int kBwdWf32 = 64 * 128 * 4;                 // 32 KB fp32 W chunk [64 o][128 i]
constexpr int kBwdWT = 128 * 64 * 2;                   // 16 KB bf16 W^T [128 i][64 o]
constexpr int kBwdDZ = 64 * 128;                       //  8 KB bf16 dZ [Bn][64 o]
constexpr int kBwdDZT = 64 * 128;                      //  8 KB bf16 dZ^T [64 o][64 b]
constexpr int kBwdStage = kBwdWf32 + kBwdWT + kBwdDZ + kBwdDZT;   // 64 KB
constexpr int kBwdHT = 128 * 128;                      // 16 KB bf16 H^T [128 i][64 b]
constexpr int kBwdBarOff = kStages * kBwdStage + kBwdHT;
constexpr int kBwdSmem = kBwdBarOff + 256 + 1024;
constexpr uint32_t kBwdTmemCols = 256;   // dX buffers at columns 0 and 192, dW buffers at 64, 128

__global__ void __launch_bounds__(kThreads, 1)
    k_tc_backward(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_ht,
                  const __grid_constant__ CUtensorMap tm_dz, const __grid_constant__ CUtensorMap tm_dzt,
                  const TcBwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.y, i0 = blockIdx.x * 128;
  const int nc = (a.out + 63) / 64;
  uint8_t* ht = smem + kStages * kBwdStage;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kBwdBarOff);
  uint64_t* conv = full + kStages;
  uint64_t* mdone = conv + kStages;
  uint64_t* empty = mdone + kStages;
  uint64_t* tfree = empty + kStages;   // [2]
  uint64_t* htfull = tfree + 2;
  uint64_t* upd = htfull + 1;         // [kStages] updated chunk ready for the TMA store
  uint64_t* xf = upd + kStages;       // [2] dX accumulator segment complete
  uint64_t* xr = xf + 2;              // [2] dX accumulator segment drained
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xr + 2);
  auto wf = [&](int s) { return smem + s * kBwdStage; };
  auto wt = [&](int s) { return smem + s * kBwdStage + kBwdWf32; };
  auto dzb = [&](int s) { return smem + s * kBwdStage + kBwdWf32 + kBwdWT; };
  auto dztb = [&](int s) { return smem + s * kBwdStage + kBwdWf32 + kBwdWT + kBwdDZ; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&conv[s], kConv);
      mbar_init(&mdone[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&tfree[0], kConv);
    mbar_init(&tfree[1], kConv);
    mbar_init(htfull, 1);
    for (int s = 0; s < kStages; ++s) mbar_init(&upd[s], kConv);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&xf[b], 1);
      mbar_init(&xr[b], kConv);
    }
    fence_barrier_init();
  }
  if (warp == 5) {
    tmem_alloc(tmem_slot, kBwdTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 4) {
    if (lane == 0) {
      tma_prefetch_desc(&tm_w);
      tma_prefetch_desc(&tm_ht);
      tma_prefetch_desc(&tm_dz);
      tma_prefetch_desc(&tm_dzt);
      mbar_arrive_expect_tx(htfull, kBwdHT);
      tma_load_3d(ht, &tm_ht, htfull, 0, i0, j);
      const uint32_t bytes = kBwdWf32 + kBwdDZT + (a.has_dx ? a.Bn * 128 : 0);
      int issued = 0;
      for (int c = 0; c < nc; ++c) {
        const int s = c % kStages;
        if (c >= kStages && !mbar_wait(&empty[s], ((c / kStages) - 1) & 1, a.err)) break;
        mbar_arrive_expect_tx(&full[s], bytes);
        tma_load_3d(wf(s), &tm_w, &full[s], i0, c * 64, j);
        if (a.has_dx) tma_load_3d(dzb(s), &tm_dz, &full[s], c * 64, 0, j);
        tma_load_3d(dztb(s), &tm_dzt, &full[s], 0, c * 64, j);
        issued = c + 1;
      }
      mbar_wait(htfull, 0, a.err);
      for (int c = issued - kStages > 0 ? issued - kStages : 0; c < issued; ++c)
        mbar_wait(&full[c % kStages], (c / kStages) & 1, a.err);
    }
  } else if (warp == 5) {
    if (lane == 0) {
      const uint32_t idesc_dx = umma_idesc_bf16(128, a.Bn);
      const uint32_t idesc_dw = umma_idesc_bf16(128, 64);
      const int kb = (a.B + 15) / 16;   // K = B for dW
      bool ok = mbar_wait(htfull, 0, a.err);
      const uint64_t hd = umma_desc_sw128(smem_u32(ht));
      int c = 0;
      for (; ok && c < nc; ++c) {
        const int s = c % kStages, buf = c & 1;
        const int seg = c / kSegChunks, xb = seg & 1, first = c % kSegChunks == 0;
        if (a.has_dx && first && seg >= 2 && !mbar_wait(&xr[xb], ((seg >> 1) - 1) & 1, a.err)) break;
        if (!mbar_wait(&conv[s], (c / kStages) & 1, a.err)) break;
        if (c >= 2 && !mbar_wait(&tfree[buf], ((c / 2) - 1) & 1, a.err)) break;
        tc_fence_after();
        if (a.has_dx) {
          const uint64_t ad = umma_desc_sw128(smem_u32(wt(s)));
          const uint64_t bd = umma_desc_sw128(smem_u32(dzb(s)));
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16(tmem + 192 * xb, ad + 2 * kk, bd + 2 * kk, idesc_dx,
                        (!first || kk > 0) ? 1u : 0u);
        }
        const uint64_t bd = umma_desc_sw128(smem_u32(dztb(s)));
        for (int kk = 0; kk < kb; ++kk)
          tc_mma_bf16(tmem + 64 + 64 * buf, hd + 2 * kk, bd + 2 * kk, idesc_dw, kk > 0 ? 1u : 0u);
        tc_commit(&mdone[s]);
        if (a.has_dx && (c % kSegChunks == kSegChunks - 1 || c == nc - 1)) tc_commit(&xf[xb]);
      }
      // Drain: the last commit covers every MMA issued before it.
      if (c > 0) mbar_wait(&mdone[(c - 1) % kStages], ((c - 1) / kStages) & 1, a.err);
    }
  } else {
    // ---- warps 0-3: W^T for dX, the in-place SGD update, then the dX epilogue
    const int t = threadIdx.x;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    // dX accumulator promoted to registers segment by segment (see kSegChunks)
    float accx[64];
#pragma unroll
    for (int q = 0; q < 64; ++q) accx[q] = 0.f;
    int drained = 0;
    const int nseg = a.has_dx ? (nc + kSegChunks - 1) / kSegChunks : 0;
    auto drain = [&]() -> bool {
      const int xb = drained & 1;
      if (!wait_warp(&xf[xb], (drained >> 1) & 1, a.err)) return false;
      tc_fence_after();
#pragma unroll
      for (int cb = 0; cb < 64; cb += 16) {
        if (cb < a.Bn) {
          float v[16];
          tmem_ld16(tbase + 192 * xb + cb, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) accx[cb + q] = __fadd_rn(accx[cb + q], v[q]);
        }
      }
      tc_fence_before();
      mbar_arrive(&xr[xb]);
      ++drained;
      return true;
    };
    bool ok = true;
    for (int c = 0; c <= nc && ok; ++c) {
      if (c < nc) {
        const int s = c % kStages;
        if (!wait_warp(&full[s], (c / kStages) & 1, a.err)) { ok = false; break; }
        if (a.has_dx) {
          const float* src = reinterpret_cast<const float*>(wf(s));
          uint8_t* dst = wt(s);
#pragma unroll
          for (int ob = 0; ob < 8; ++ob) {
            float v[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) v[q] = src[(ob * 8 + q) * 128 + t];
            *reinterpret_cast<uint4*>(dst + sw128_offset(t, ob * 8)) =
                make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                           pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
          }
          fence_proxy_async_smem();
        }
        mbar_arrive(&conv[s]);
      }
      if (c > 0) {
        const int cp = c - 1, sp = cp % kStages, buf = cp & 1;
        if (!wait_warp(&mdone[sp], (cp / kStages) & 1, a.err)) { ok = false; break; }
        tc_fence_after();
        float* w = reinterpret_cast<float*>(wf(sp));
#pragma unroll
        for (int qb = 0; qb < 4; ++qb) {
          float d[16];
          tmem_ld16(tbase + 64 + 64 * buf + 16 * qb, d);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            float* p = w + (qb * 16 + q) * 128 + t;
            *p = __fsub_rn(*p, __fmul_rn(a.lr, d[q]));
          }
        }
        tc_fence_before();
        mbar_arrive(&tfree[buf]);
        fence_proxy_async_smem();
        mbar_arrive(&upd[sp]);
        if (t == 0) {
          if (mbar_wait(&upd[sp], (cp / kStages) & 1, a.err)) {
            tma_store_3d(&tm_w, w, i0, cp * 64, j);
            tma_store_commit();
            tma_store_wait_read_all();
          }
          mbar_arrive(&empty[sp]);
        }
        if (a.has_dx && cp % kSegChunks == kSegChunks - 1 && cp / kSegChunks >= 1 &&
            drained < cp / kSegChunks)
          if (!drain()) { ok = false; break; }
      }
    }
    while (ok && drained < nseg)
      if (!drain()) ok = false;
    if (t == 0) tma_store_wait_all();
    if (ok && a.has_dx) {
      // dX epilogue: thread t holds dH^T[i0 + t][0 .. Bn) in accx
      const int i = i0 + t;
      const bool valid = i < a.in;
      float db = 0.f;
#pragma unroll
      for (int cb = 0; cb < 64; cb += 16) {
        if (cb >= a.Bn || !valid) break;
        const float* v = accx + cb;
        uint32_t pk[8];
#pragma unroll
        for (int q = 0; q < 16; q += 2) {
          float dz[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int b = cb + q + e;
            float x = 0.f;
            if (b < a.B) {
              const __nv_bfloat16 h = *reinterpret_cast<const __nv_bfloat16*>(ht + sw128_offset(t, b));
              x = (__bfloat162float(h) > 0.f) ? v[q + e] : 0.f;
              db = __fadd_rn(db, x);
            }
            dz[e] = x;
          }
          pk[q / 2] = pack_bf16x2(dz[0], dz[1]);
          const __nv_bfloat162 hh = *reinterpret_cast<__nv_bfloat162*>(&pk[q / 2]);
          if (cb + q < a.B) a.dz_prev[(static_cast<int64_t>(j) * a.Bn + cb + q) * a.pitch_in + i] = hh.x;
          if (cb + q + 1 < a.B) a.dz_prev[(static_cast<int64_t>(j) * a.Bn + cb + q + 1) * a.pitch_in + i] = hh.y;
        }
        uint4* dst = reinterpret_cast<uint4*>(a.dzt_prev + (static_cast<int64_t>(j) * a.in + i) * a.Kp + cb);
        dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
      }
      if (valid) {
        float* bp = a.bias_prev + static_cast<int64_t>(j) * a.ld + i;
        *bp = __fsub_rn(*bp, __fmul_rn(a.lr, db));
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kBwdTmemCols);
  }
}

// ------------------------------------------------------------------ gather
// H_0[j][b][:] = X[j][(t*B + b) mod N][:], HT_0[j][k][b] = the same; one CTA per
// (64-feature slice, learner).  Rows b >= B and columns b >= B stay zero.
__global__ void __launch_bounds__(256) k_gather_bf16(const __nv_bfloat16* __restrict__ X,
                                                    int64_t N, int d0, int B, int Bn, int Kp,
                                                    int pitch0, int64_t t,
                                                    __nv_bfloat16* __restrict__ H0,
                                                    __nv_bfloat16* __restrict__ HT0) {
  __shared__ __align__(16) __nv_bfloat16 tile[64][64 + 8];
  const int j = blockIdx.y, k0 = blockIdx.x * 64;
  const int nvec = B * 8;                       // 16-byte vectors in the [B][64] slice
  for (int idx = threadIdx.x; idx < nvec; idx += blockDim.x) {
    const int b = idx >> 3, v = idx & 7;
    const int k = k0 + v * 8;
    uint4 val = make_uint4(0, 0, 0, 0);
    if (k < d0) {
      const int64_t row = (t * B + b) % N;
      val = *reinterpret_cast<const uint4*>(X + (static_cast<int64_t>(j) * N + row) * d0 + k);
      *reinterpret_cast<uint4*>(H0 + (static_cast<int64_t>(j) * Bn + b) * pitch0 + k) = val;
    }
    *reinterpret_cast<uint4*>(&tile[b][v * 8]) = val;
  }
  __syncthreads();
  const int nbv = Bn / 8;                       // 8-column groups of the transposed row
  for (int idx = threadIdx.x; idx < 64 * nbv; idx += blockDim.x) {
    const int kk = idx / nbv, bv = idx % nbv;
    const int k = k0 + kk;
    if (k >= d0) continue;
    __align__(16) __nv_bfloat16 vals[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int b = bv * 8 + q;
      vals[q] = b < B ? tile[b][kk] : __float2bfloat16_rn(0.f);
    }
    *reinterpret_cast<uint4*>(HT0 + (static_cast<int64_t>(j) * d0 + k) * Kp + bv * 8) =
        *reinterpret_cast<uint4*>(vals);
  }
}

// ------------------------------------------------------------------ cross-entropy
// Softmax cross-entropy gradient when the classes span several output tiles.
// Grid (P, class slices of 256).  Every CTA computes the per-sample statistics
// (max, sum of exponentials over all C classes; warp per sample), then each
// thread owns one class of its slice: dZ = (p - onehot(y_b)) / B in fp32 for
// every sample, the bf16 operands dZ and dZ^T, and b_L -= lr * sum_b dZ (summed
// in sample order).  Slice 0 also writes the learner's mean loss.
constexpr int kXentThreads = 256;
__global__ void __launch_bounds__(kXentThreads) k_xent_bf16(const float* __restrict__ Z,
                                                           const int32_t* __restrict__ y,
                                                           int64_t N, int64_t t, int B, int Bn,
                                                           int Kp, int C, int pitch_c, float lr,
                                                           float* bias_L, int64_t ld,
                                                           __nv_bfloat16* dZ, __nv_bfloat16* dZT,
                                                           float* loss) {
  __shared__ float row_max[64], row_sum[64], row_loss[64];
  __shared__ int row_y[64];
  const int j = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* Zj = Z + static_cast<int64_t>(j) * B * C;
  for (int b = warp; b < B; b += kXentThreads / 32) {
    const float* z = Zj + static_cast<int64_t>(b) * C;
    float m = -INFINITY;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, z[c]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    float s = 0.f;
    for (int c = lane; c < C; c += 32) s += expf(z[c] - m);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) {
      const int yb = y[static_cast<int64_t>(j) * N + (t * B + b) % N];
      row_max[b] = m;
      row_sum[b] = s;
      row_y[b] = yb;
      row_loss[b] = logf(s) + m - z[yb];
    }
  }
  __syncthreads();
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += row_loss[b];
    loss[j] = l / B;
  }
  const int c = blockIdx.y * kXentThreads + threadIdx.x;
  if (c >= C) return;
  const float fB = static_cast<float>(B);
  float db = 0.f;
  for (int b0 = 0; b0 < Bn; b0 += 8) {
    uint32_t pk[4];
#pragma unroll
    for (int q = 0; q < 8; q += 2) {
      float g2[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int b = b0 + q + e;
        float g = 0.f;
        if (b < B) {
          const float p = __fdiv_rn(expf(Zj[static_cast<int64_t>(b) * C + c] - row_max[b]), row_sum[b]);
          g = __fdiv_rn(__fsub_rn(p, row_y[b] == c ? 1.f : 0.f), fB);
          db = __fadd_rn(db, g);
          dZ[(static_cast<int64_t>(j) * Bn + b) * pitch_c + c] = __float2bfloat16_rn(g);
        }
        g2[e] = g;
      }
      pk[q / 2] = pack_bf16x2(g2[0], g2[1]);
    }
    *reinterpret_cast<uint4*>(dZT + (static_cast<int64_t>(j) * C + c) * Kp + b0) =
        make_uint4(pk[0], pk[1], pk[2], pk[3]);
  }
  float* bp = bias_L + static_cast<int64_t>(j) * ld + c;
  *bp = __fsub_rn(*bp, __fmul_rn(lr, db));
}

}  // namespace

int tc_fwd_smem_bytes() { return kFwdSmemMax; }
int tc_bwd_smem_bytes() { return kBwdSmem; }

cudaError_t tc_configure() {
  cudaError_t e = cudaFuncSetAttribute(k_tc_forward, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kFwdSmemMax);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_tc_backward, cudaFuncAttributeMaxDynamicSharedMemorySize, kBwdSmem);
}

cudaError_t launch_tc_forward(const CUtensorMap& w_fwd, const CUtensorMap& h_in,
                              const TcFwdArgs& a, int P, cudaStream_t s) {
  (void)P;
  // Cooperative: the finisher of a split tile waits for the other contributors,
  // so every CTA of the grid must be resident at once (the launch fails otherwise).
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.ctas);
  cfg.blockDim = dim3(kFwdThreads);
  cfg.dynamicSmemBytes = fwd_smem(a.mode, a.Bn);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_tc_forward, w_fwd, h_in, a);
}

cudaError_t launch_tc_backward(const CUtensorMap& w_bwd, const CUtensorMap& ht_in,
                               const CUtensorMap& dz, const CUtensorMap& dzt,
                               const TcBwdArgs& a, int P, cudaStream_t s) {
  dim3 grid((a.in + 127) / 128, P);
  k_tc_backward<<<grid, kThreads, kBwdSmem, s>>>(w_bwd, ht_in, dz, dzt, a);
  return cudaGetLastError();
}

cudaError_t launch_gather_bf16(const __nv_bfloat16* X, int64_t N, int d0, int B, int Bn,
                               int Kp, int pitch0, int64_t t, int P, __nv_bfloat16* H0,
                               __nv_bfloat16* HT0, cudaStream_t s) {
  dim3 grid((d0 + 63) / 64, P);
  k_gather_bf16<<<grid, 256, 0, s>>>(X, N, d0, B, Bn, Kp, pitch0, t, H0, HT0);
  return cudaGetLastError();
}

cudaError_t launch_xent_bf16(const float* Z, const int32_t* y, int64_t N, int64_t t, int B,
                             int Bn, int Kp, int C, int pitch_c, float lr, float* bias_L,
                             int64_t ld, __nv_bfloat16* dZ, __nv_bfloat16* dZT, float* loss,
                             int P, cudaStream_t s) {
  dim3 grid(P, (C + kXentThreads - 1) / kXentThreads);
  k_xent_bf16<<<grid, kXentThreads, 0, s>>>(Z, y, N, t, B, Bn, Kp, C, pitch_c, lr, bias_L, ld, dZ, dZT, loss);
  return cudaGetLastError();
}

}  // namespace ha
