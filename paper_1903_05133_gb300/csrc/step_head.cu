// Last layer of the learner step when it is small (at most 16 classes) and the forward
// did not already run it (see head_body.cuh): one kernel, one thread-block cluster of
// S CTAs per learner, CTA s owning the input features [s*F, (s+1)*F).
#include "head_body.cuh"

namespace ha {
namespace {
using namespace head;

// Features per CTA (a multiple of 64) for P learners: 8 CTAs per learner (slices of at
// least 64) while all P clusters fit in one wave of the GPU's 152 SMs, else 4 (at least
// 128; more clusters of 8 than fit at once measured slower), or 8 where 4 would need
// slices over 512.
constexpr int kHeadWave = 152;
__host__ __device__ inline int head_slice(int in, int P) {
  const bool wide = P * kHeadClusterMax <= kHeadWave;
  const int per = wide ? kHeadClusterMax : kHeadClusterPref;
  int f = ((in + per - 1) / per + 63) / 64 * 64;
  if (f > 512) f = ((in + kHeadClusterMax - 1) / kHeadClusterMax + 63) / 64 * 64;
  const int fmin = wide ? 64 : 128;
  return f < fmin ? fmin : f;
}
__host__ __device__ inline int head_smem_bytes(int in, int P, int Bn) {
  return head_body_smem(head_slice(in, P), Bn);
}

template <int CT>
__global__ void __launch_bounds__(kHeadThreads) k_head(const HeadArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  grid_dep_wait();
  head_body<CT>(a, smem, blockIdx.y, blockIdx.x, gridDim.x, head_slice(a.in, gridDim.y), threadIdx.x,
                [] { __syncthreads(); });
}

template <int CT>
cudaError_t launch_cluster(const HeadArgs& a, int P, cudaStream_t s) {
  const int F = head_slice(a.in, P), S = (a.in + F - 1) / F;
  return launch_pdl(k_head<CT>, dim3(S, P), dim3(kHeadThreads), head_smem_bytes(a.in, P, a.Bn), s,
                    false, S, a);
}

}  // namespace

bool head_supported(int C, int in, int B, int P) {
  return C <= kHeadMaxC && in % 64 == 0 && B <= 64 &&
         (in + head_slice(in, P) - 1) / head_slice(in, P) <= kHeadClusterMax &&
         head_smem_bytes(in, P, 64) <= 200 * 1024;
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
