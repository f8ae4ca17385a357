// fp32 learner step on CUDA cores: the precision mode in which every product and
// sum of the local SGD step (Algorithm 1 inner loop, Sec. 3.1) stays in fp32.
// Used for the fp32 softmax-regression workload (3072 -> 10, B = 16), whose
// tolerance forbids bf16 or tf32 operands.  The sizes are small, so these are
// plain 16x16-tiled shared-memory kernels; each output is one fp32 FMA chain
// over its reduction index in ascending order.
#include <cstdint>
#include <cuda_runtime.h>

#include "internal.h"

namespace ha {
namespace {

constexpr int T = 16;

// H0[j][b][:] = X[j][(row0 + b) mod N][:]  (row0: the batch's first row)
__global__ void k_gather_f32(const float* __restrict__ X, int64_t N, int d0, int B, int64_t row0,
                             float* __restrict__ H0) {
  const int j = blockIdx.y;
  const int64_t total = static_cast<int64_t>(B) * d0;
  for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int b = static_cast<int>(idx / d0), k = static_cast<int>(idx % d0);
    const int64_t row = (row0 + b) % N;
    H0[(static_cast<int64_t>(j) * B + b) * d0 + k] = X[(static_cast<int64_t>(j) * N + row) * d0 + k];
  }
}

// Z[j][b][o] = sum_k H[j][b][k] W[j][o][k] + bias[j][o]; ReLU for hidden layers.
__global__ void k_fwd_f32(const float* __restrict__ H, const float* __restrict__ W,
                          const float* __restrict__ bias, int64_t ld, int in, int out, int B,
                          int relu, float* __restrict__ Y) {
  __shared__ float hs[T][T + 1], ws[T][T + 1];
  const int j = blockIdx.z, b = blockIdx.y * T + threadIdx.y, o = blockIdx.x * T + threadIdx.x;
  const float* Hj = H + static_cast<int64_t>(j) * B * in;
  const float* Wj = W + static_cast<int64_t>(j) * ld;
  float acc = 0.f;
  for (int k0 = 0; k0 < in; k0 += T) {
    const int k = k0 + threadIdx.x;
    const int bb = blockIdx.y * T + threadIdx.y, oo = blockIdx.x * T + threadIdx.y;
    hs[threadIdx.y][threadIdx.x] = (bb < B && k < in) ? Hj[static_cast<int64_t>(bb) * in + k] : 0.f;
    ws[threadIdx.y][threadIdx.x] = (oo < out && k < in) ? Wj[static_cast<int64_t>(oo) * in + k] : 0.f;
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < T; ++kk) acc = fmaf(hs[threadIdx.y][kk], ws[threadIdx.x][kk], acc);
    __syncthreads();
  }
  if (b < B && o < out) {
    float z = __fadd_rn(acc, bias[static_cast<int64_t>(j) * ld + o]);
    if (relu) z = fmaxf(z, 0.f);
    Y[(static_cast<int64_t>(j) * B + b) * out + o] = z;
  }
}

// One CTA per learner: dZ = (softmax(z_b) - onehot(y_b)) / B, loss = mean CE.
__global__ void __launch_bounds__(256) k_xent_f32(const float* __restrict__ Z,
                                                 const int32_t* __restrict__ y, int64_t N,
                                                 int64_t row0, int B, int C, float* __restrict__ dZ,
                                                 float* __restrict__ loss) {
  extern __shared__ float sh[];
  float* row_max = sh;
  float* row_sum = sh + B;
  float* row_loss = sh + 2 * B;
  int* row_y = reinterpret_cast<int*>(sh + 3 * B);
  const int j = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* Zj = Z + static_cast<int64_t>(j) * B * C;
  for (int b = warp; b < B; b += blockDim.x / 32) {
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
      const int yb = y[static_cast<int64_t>(j) * N + (row0 + b) % N];
      row_max[b] = m;
      row_sum[b] = s;
      row_y[b] = yb;
      row_loss[b] = logf(s) + m - z[yb];
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += row_loss[b];
    loss[j] = l / B;
  }
  const float fB = static_cast<float>(B);
  const int64_t total = static_cast<int64_t>(B) * C;
  for (int64_t idx = threadIdx.x; idx < total; idx += blockDim.x) {
    const int b = static_cast<int>(idx / C), c = static_cast<int>(idx % C);
    const float p = __fdiv_rn(expf(Zj[idx] - row_max[b]), row_sum[b]);
    dZ[static_cast<int64_t>(j) * total + idx] = __fdiv_rn(__fsub_rn(p, row_y[b] == c ? 1.f : 0.f), fB);
  }
}

// dZprev[j][b][i] = (sum_o dZ[j][b][o] W[j][o][i]) * [Hprev[j][b][i] > 0]  (W before update)
__global__ void k_dx_f32(const float* __restrict__ dZ, const float* __restrict__ W, int64_t ld,
                         const float* __restrict__ Hprev, int in, int out, int B,
                         float* __restrict__ dZprev) {
  __shared__ float zs[T][T + 1], ws[T][T + 1];
  const int j = blockIdx.z, b = blockIdx.y * T + threadIdx.y, i = blockIdx.x * T + threadIdx.x;
  const float* dZj = dZ + static_cast<int64_t>(j) * B * out;
  const float* Wj = W + static_cast<int64_t>(j) * ld;
  float acc = 0.f;
  for (int o0 = 0; o0 < out; o0 += T) {
    const int bb = blockIdx.y * T + threadIdx.y, oo = o0 + threadIdx.x;
    zs[threadIdx.y][threadIdx.x] = (bb < B && oo < out) ? dZj[static_cast<int64_t>(bb) * out + oo] : 0.f;
    const int orow = o0 + threadIdx.y;
    ws[threadIdx.y][threadIdx.x] = (orow < out && i < in) ? Wj[static_cast<int64_t>(orow) * in + i] : 0.f;
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < T; ++kk) acc = fmaf(zs[threadIdx.y][kk], ws[kk][threadIdx.x], acc);
    __syncthreads();
  }
  if (b < B && i < in) {
    const int64_t e = (static_cast<int64_t>(j) * B + b) * in + i;
    dZprev[e] = Hprev[e] > 0.f ? acc : 0.f;
  }
}

// W[j][o][i] -= lr * sum_b dZ[j][b][o] H[j][b][i]; blocks of the first column tile
// also apply bias[j][o] -= lr * sum_b dZ[j][b][o].
__global__ void k_dw_update_f32(const float* __restrict__ dZ, const float* __restrict__ H,
                                float* __restrict__ W, float* __restrict__ bias, int64_t ld,
                                int in, int out, int B, float lr) {
  __shared__ float zs[T][T + 1], hs[T][T + 1];
  const int j = blockIdx.z, o = blockIdx.y * T + threadIdx.y, i = blockIdx.x * T + threadIdx.x;
  const float* dZj = dZ + static_cast<int64_t>(j) * B * out;
  const float* Hj = H + static_cast<int64_t>(j) * B * in;
  float acc = 0.f;
  for (int b0 = 0; b0 < B; b0 += T) {
    const int bb = b0 + threadIdx.x, orow = blockIdx.y * T + threadIdx.y;
    zs[threadIdx.y][threadIdx.x] = (bb < B && orow < out) ? dZj[static_cast<int64_t>(bb) * out + orow] : 0.f;
    const int brow = b0 + threadIdx.y;
    hs[threadIdx.y][threadIdx.x] = (brow < B && i < in) ? Hj[static_cast<int64_t>(brow) * in + i] : 0.f;
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < T; ++kk) acc = fmaf(zs[threadIdx.y][kk], hs[kk][threadIdx.x], acc);
    __syncthreads();
  }
  if (o < out && i < in) {
    float* p = W + static_cast<int64_t>(j) * ld + static_cast<int64_t>(o) * in + i;
    *p = __fsub_rn(*p, __fmul_rn(lr, acc));
  }
  if (blockIdx.x == 0 && threadIdx.x == 0 && o < out) {
    float db = 0.f;
    for (int b = 0; b < B; ++b) db = __fadd_rn(db, dZj[static_cast<int64_t>(b) * out + o]);
    float* p = bias + static_cast<int64_t>(j) * ld + o;
    *p = __fsub_rn(*p, __fmul_rn(lr, db));
  }
}

}  // namespace

cudaError_t launch_gather_f32(const float* X, int64_t N, int d0, int B, int64_t row0, int P,
                              float* H0, cudaStream_t s) {
  const int64_t total = static_cast<int64_t>(B) * d0;
  dim3 grid(static_cast<unsigned>((total + 255) / 256 < 1024 ? (total + 255) / 256 : 1024), P);
  k_gather_f32<<<grid, 256, 0, s>>>(X, N, d0, B, row0, H0);
  return cudaGetLastError();
}

cudaError_t launch_fwd_f32(const float* H, const float* W, const float* bias, int64_t ld,
                           int in, int out, int B, int relu, float* out_act, int P,
                           cudaStream_t s) {
  dim3 grid((out + T - 1) / T, (B + T - 1) / T, P), block(T, T);
  k_fwd_f32<<<grid, block, 0, s>>>(H, W, bias, ld, in, out, B, relu, out_act);
  return cudaGetLastError();
}

cudaError_t launch_xent_f32(const float* Z, const int32_t* y, int64_t N, int64_t row0, int B,
                            int C, float* dZ, float* loss, int P, cudaStream_t s) {
  const size_t sh = static_cast<size_t>(4) * B * sizeof(float);
  k_xent_f32<<<P, 256, sh, s>>>(Z, y, N, row0, B, C, dZ, loss);
  return cudaGetLastError();
}

cudaError_t launch_dx_f32(const float* dZ, const float* W, int64_t ld, const float* Hprev,
                          int in, int out, int B, float* dZprev, int P, cudaStream_t s) {
  dim3 grid((in + T - 1) / T, (B + T - 1) / T, P), block(T, T);
  k_dx_f32<<<grid, block, 0, s>>>(dZ, W, ld, Hprev, in, out, B, dZprev);
  return cudaGetLastError();
}

cudaError_t launch_dw_update_f32(const float* dZ, const float* H, float* W, float* bias,
                                 int64_t ld, int in, int out, int B, float lr, int P,
                                 cudaStream_t s) {
  dim3 grid((in + T - 1) / T, (out + T - 1) / T, P), block(T, T);
  k_dw_update_f32<<<grid, block, 0, s>>>(dZ, H, W, bias, ld, in, out, B, lr);
  return cudaGetLastError();
}

}  // namespace ha
