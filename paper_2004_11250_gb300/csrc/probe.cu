// Peak-rate probes: one launch keeps a single execution pipe busy on every SM,
// so the roofline fractions of the convolution kernels can be taken against a
// rate measured on the running GPU instead of a data-sheet figure.
//
//   FFMA      fp32 fused multiply-add on the CUDA cores: 4 CTAs of 256 threads
//             per SM, 16 independent dependency chains per thread (enough to
//             cover the FMA latency), 2 FLOP per multiply-add.
//   MMA_TF32  tcgen05.mma kind::tf32, M = 128, N = 256, K = 8 per instruction,
//   MMA_F16   tcgen05.mma kind::f16 (f16 operands, f32 accumulation), K = 16:
//             one CTA per SM, one thread issues back-to-back MMAs on operands in
//             shared memory into one TMEM accumulator, then waits (bounded) for
//             their completion; 2 * M * N * K FLOP per instruction.
//
// Every probe also reports the SM clock seen during the launch: the SM cycle
// counter over the global nanosecond timer of one CTA.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.h"
#include "tc_ptx.cuh"

namespace {

using namespace ppc_ptx;

constexpr int FFMA_CHAINS = 16;
constexpr int FFMA_THREADS = 256;
constexpr int FFMA_CTAS_PER_SM = 4;
constexpr int MMA_M = 128, MMA_N = 256;
constexpr int MMA_THREADS = 128;
constexpr int MMA_A_BYTES = MMA_M * 32;  // 128 rows x (8 tf32 | 16 f16)
constexpr int MMA_B_BYTES = MMA_N * 32;

struct ProbeOut {
  unsigned long long clk0, clk1, ns0, ns1;
  int timed_out;
  float sink;
};

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t)::"memory");
  return t;
}

__global__ void __launch_bounds__(FFMA_THREADS) ffma_probe_kernel(long long iters, float b, float c, ProbeOut* out) {
  float a[FFMA_CHAINS];
#pragma unroll
  for (int k = 0; k < FFMA_CHAINS; ++k) a[k] = (float)(threadIdx.x + k);
  unsigned long long clk0 = 0, ns0 = 0;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    ns0 = globaltimer();
    clk0 = clock64();
  }
  // (a loop unrolled 8 rounds deep measured ~4 % lower on GB300 than this one)
  for (long long i = 0; i < iters; ++i) {
#pragma unroll
    for (int k = 0; k < FFMA_CHAINS; ++k) a[k] = fmaf(a[k], b, c);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < FFMA_CHAINS; ++k) s += a[k];
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    out->clk1 = clock64();
    out->ns1 = globaltimer();
    out->clk0 = clk0;
    out->ns0 = ns0;
    out->timed_out = 0;
  }
  if (s == 1234.5f) out->sink = s;  // keeps the chains live; practically never taken
}

template <bool F16>
__global__ void __launch_bounds__(MMA_THREADS, 1) mma_probe_kernel(long long iters, ProbeOut* out) {
  __shared__ __align__(1024) unsigned char ops[MMA_A_BYTES + MMA_B_BYTES];
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_s;
  const int tid = threadIdx.x, warp = tid >> 5;
  for (int i = tid; i < (MMA_A_BYTES + MMA_B_BYTES) / 16; i += MMA_THREADS)
    reinterpret_cast<uint4*>(ops)[i] = make_uint4(0, 0, 0, 0);
  if (tid == 0) {
    mbar_init(su32(&done_bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tmem_s)),
                 "n"(MMA_N));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  // the zeroed operands are visible to the tensor core's (async) reads
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  const uint32_t tmem = tmem_s;
  if (tid == 0) {
    // K-major operands without swizzle: 8-row core matrices of 16 bytes, the
    // two K halves (32 bytes of K per row) rows x 16 bytes apart
    const uint64_t a = smem_desc(su32(ops), MMA_M * 16);
    const uint64_t b = smem_desc(su32(ops + MMA_A_BYTES), MMA_N * 16);
    const uint32_t id = F16 ? idesc_f16(MMA_M, MMA_N) : idesc_tf32(MMA_M, MMA_N);
    const unsigned long long ns0 = globaltimer(), clk0 = clock64();
    for (long long i = 0; i < iters; ++i) {
      if (F16)
        mma_f16(tmem, a, b, id, i > 0 ? 1u : 0u);
      else
        mma_tf32(tmem, a, b, id, i > 0 ? 1u : 0u);
    }
    mma_commit(su32(&done_bar));
    bool ok = false;
    for (long k = 0; k < PP_WAIT_POLLS && !ok; ++k) ok = mbar_try(su32(&done_bar), 0u);
    const unsigned long long clk1 = clock64(), ns1 = globaltimer();
    if (blockIdx.x == 0) {
      out->clk0 = clk0;
      out->clk1 = clk1;
      out->ns0 = ns0;
      out->ns1 = ns1;
    }
    if (!ok) atomicExch(&out->timed_out, 1);
  }
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(MMA_N));
}

}  // namespace

extern "C" pp_status pp_peak_probe(int kind, long long iters, double* tflops, double* sm_mhz, double* ms) {
  if (!tflops || !sm_mhz || !ms || iters < 1 || iters > (1LL << 24)) return PP_ERR_INVALID_ARG;
  if (kind != PP_PROBE_FFMA && kind != PP_PROBE_MMA_TF32 && kind != PP_PROBE_MMA_F16) return PP_ERR_INVALID_ARG;
  const int sms = ppc::device_sms();
  if (sms <= 0) return PP_ERR_CUDA;
  ProbeOut* d = nullptr;
  if (cudaMalloc(&d, sizeof(ProbeOut)) != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_OOM;
  }
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  bool ok = cudaMemset(d, 0, sizeof(ProbeOut)) == cudaSuccess && cudaEventCreate(&e0) == cudaSuccess &&
            cudaEventCreate(&e1) == cudaSuccess && cudaEventRecord(e0, 0) == cudaSuccess;
  double flop = 0.0;
  if (ok) {
    if (kind == PP_PROBE_FFMA) {
      const int ctas = sms * FFMA_CTAS_PER_SM;
      ffma_probe_kernel<<<ctas, FFMA_THREADS>>>(iters, 0.999f, 1e-3f, d);
      flop = 2.0 * FFMA_CHAINS * (double)iters * ctas * FFMA_THREADS;
    } else {
      const bool f16 = kind == PP_PROBE_MMA_F16;
      if (f16)
        mma_probe_kernel<true><<<sms, MMA_THREADS>>>(iters, d);
      else
        mma_probe_kernel<false><<<sms, MMA_THREADS>>>(iters, d);
      flop = 2.0 * MMA_M * MMA_N * (f16 ? 16 : 8) * (double)iters * sms;
    }
    ok = cudaGetLastError() == cudaSuccess;
  }
  ok = ok && cudaEventRecord(e1, 0) == cudaSuccess && cudaEventSynchronize(e1) == cudaSuccess;
  float t_ms = 0.f;
  ProbeOut h = {};
  ok = ok && cudaEventElapsedTime(&t_ms, e0, e1) == cudaSuccess &&
       cudaMemcpy(&h, d, sizeof(ProbeOut), cudaMemcpyDeviceToHost) == cudaSuccess;
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  cudaFree(d);
  if (!ok) {
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  if (h.timed_out) return PP_ERR_CUDA;
  *ms = t_ms;
  *tflops = t_ms > 0.f ? flop / (t_ms * 1e-3) / 1e12 : 0.0;
  *sm_mhz = h.ns1 > h.ns0 ? (double)(h.clk1 - h.clk0) / (double)(h.ns1 - h.ns0) * 1e3 : 0.0;
  return PP_OK;
}
