// Direct 3x3 convolution on the FP32 FMA pipes for layers with few input or
// few output channels (the first and last layers of the networks: VGG-16's
// 3 -> 64, the VDSR-shaped stack's 1 -> 64 and 64 -> 1 dense convolutions, the
// 16 -> 16 single layer).  For these the tensor-core kernels cannot fill an
// MMA (K = 8 channels per chunk, M = 64 or 128 filters) and their per-tile
// start-up dominates, while the FMA kernels built for pattern dispatch carry
// machinery these shapes do not need.
//
// The weights are expanded to dense [Co][Ci][9] (pruned taps and kernels are
// exact zeros, so the sum is the one of Section 2 with zero terms added).
// CTA: a 32 x 32 output tile and FBD filters; 256 threads, each owning a 2 x 2
// pixel block and accumulating FBD x 4 outputs in registers.  Input channels
// are staged CC at a time (tile plus one-pixel zero halo) together with their
// weights, double-buffered with cp.async; per channel a thread reads its 4 x 4
// input window once and runs FBD x 36 FMAs on it, the weights coming from
// shared memory as warp-wide broadcasts.  Epilogue: + bias, + skip, ReLU,
// optional 2 x 2 max pool, stored in the original channel order.
#include <cuda_runtime.h>

#include <cstring>
#include <vector>

#include "internal.h"

namespace {

constexpr int DT = 32;        // output tile edge
constexpr int DTW = DT + 2;   // staged rows (one-pixel halo)
constexpr int DCOLS = DT + 8; // staged columns: c0 - 4 .. c0 + 35 (16-byte aligned groups of 4)
constexpr int DPITCH = DCOLS; // shared-memory row pitch in floats
constexpr int DTHREADS = 256;

struct DirectParams {
  const float* x;
  float* y;
  const float* skip;
  const float* w;     // [Co][Ci][9], original filter order
  const float* bias;  // [Co] or null
  int N, Ci, Co, H, W, flags;
  int tiles_x, tiles_y;
  int vec;  // x 16-byte aligned and W a multiple of 4: rows staged in 16-byte copies
};

__device__ __forceinline__ void cp_async4(float* dst, const float* src, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(src), "r"(valid ? 4 : 0) : "memory");
}
__device__ __forceinline__ void cp_async16(float* dst, const float* src, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(valid ? 16 : 0) : "memory");
}

template <int CC, int FBD>
__global__ void __launch_bounds__(DTHREADS, FBD >= 16 ? 2 : 3) ppconv_direct_kernel(const DirectParams p) {
  // two stages of [CC][DTW][DPITCH] input and [CC][FBD][12] weights (9 taps padded to 12)
  extern __shared__ __align__(16) float dsm[];
  auto xs = reinterpret_cast<float(*)[CC][DTW][DPITCH]>(dsm);
  auto ws = reinterpret_cast<float(*)[CC][FBD][12]>(dsm + 2 * CC * DTW * DPITCH);
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  int t = (int)blockIdx.x;
  const int bx = t % p.tiles_x;
  t /= p.tiles_x;
  const int by = t % p.tiles_y;
  const int n = t / p.tiles_y;
  const int o0 = (int)blockIdx.y * FBD;
  const int r0 = by * DT, c0 = bx * DT;
  const float* xb = p.x + (size_t)n * p.Ci * p.H * p.W;
  const int nchunks = (p.Ci + CC - 1) / CC;

  // channels ch * CC .. of the input tile (zero outside the image and beyond
  // Ci) and their weights for this CTA's filters (zero beyond Co) into buffer b
  // staged column j holds image column c0 - 4 + j
  auto stage = [&](int ch, int b) {
    if (p.vec) {
      // rows of 16-byte groups: with W a multiple of 4 each group is wholly inside or outside the image
      for (int e = tid; e < CC * DTW * (DCOLS / 4); e += DTHREADS) {
        const int k = e / (DTW * (DCOLS / 4)), rem = e - k * (DTW * (DCOLS / 4));
        const int rr = rem / (DCOLS / 4), g = rem - rr * (DCOLS / 4);
        const int c = ch * CC + k, r = r0 - 1 + rr, col = c0 - 4 + 4 * g;
        const bool in = c < p.Ci && (unsigned)r < (unsigned)p.H && (unsigned)col < (unsigned)p.W;
        cp_async16(&xs[b][k][rr][4 * g], in ? xb + ((size_t)c * p.H + r) * p.W + col : p.x, in);
      }
    } else {
      for (int e = tid; e < CC * DTW * DTW; e += DTHREADS) {
        const int k = e / (DTW * DTW), rem = e - k * (DTW * DTW);
        const int rr = rem / DTW, cc = rem - rr * DTW;
        const int c = ch * CC + k, r = r0 - 1 + rr, col = c0 - 1 + cc;
        const bool in = c < p.Ci && (unsigned)r < (unsigned)p.H && (unsigned)col < (unsigned)p.W;
        cp_async4(&xs[b][k][rr][cc + 3], in ? xb + ((size_t)c * p.H + r) * p.W + col : p.x, in);
      }
    }
    for (int e = tid; e < CC * FBD * 9; e += DTHREADS) {
      const int k = e / (FBD * 9), rem = e - k * (FBD * 9);
      const int o = rem / 9, tap = rem - o * 9;
      const int c = ch * CC + k, oo = o0 + o;
      const bool in = c < p.Ci && oo < p.Co;
      cp_async4(&ws[b][k][o][tap], in ? p.w + ((size_t)oo * p.Ci + c) * 9 + tap : p.w, in);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  float acc[FBD][4];
#pragma unroll
  for (int o = 0; o < FBD; ++o)
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[o][q] = 0.f;

  // programmatic dependent launch: nothing of the previous kernel in the
  // stream is read or overwritten before this wait
  asm volatile("griddepcontrol.wait;" ::: "memory");
  stage(0, 0);
  for (int ch = 0; ch < nchunks; ++ch) {
    const int b = ch & 1;
    if (ch + 1 < nchunks) {
      stage(ch + 1, b ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < CC; ++k) {
      // the thread's 4 x 4 input window: staged rows 2 ty .. 2 ty + 3, image
      // columns c0 + 2 tx - 1 .. c0 + 2 tx + 2 (staged 2 tx + 3 .. 2 tx + 6)
      float xv[4][4];
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int q = 0; q < 4; ++q) xv[a][q] = xs[b][k][2 * ty + a][2 * tx + 3 + q];
#pragma unroll
      for (int o = 0; o < FBD; ++o) {
        const float4 w0 = *reinterpret_cast<const float4*>(&ws[b][k][o][0]);
        const float4 w1 = *reinterpret_cast<const float4*>(&ws[b][k][o][4]);
        const float w8 = ws[b][k][o][8];
        const float wt[9] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w, w8};
#pragma unroll
        for (int dy = 0; dy < 3; ++dy)
#pragma unroll
          for (int dx = 0; dx < 3; ++dx)
#pragma unroll
            for (int py = 0; py < 2; ++py)
#pragma unroll
              for (int px = 0; px < 2; ++px)
                acc[o][py * 2 + px] = fmaf(wt[dy * 3 + dx], xv[py + dy][px + dx], acc[o][py * 2 + px]);
      }
    }
    __syncthreads();  // buffer b is restaged by the next iteration's copy
  }

  // the next kernel may start its prologue (it waits for this grid to finish)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const bool relu = p.flags & PP_RELU, pool = p.flags & PP_POOL2;
  const float* skip = (p.flags & PP_ADD_SKIP) ? p.skip : nullptr;
  const int r = r0 + 2 * ty, c = c0 + 2 * tx;
#pragma unroll
  for (int o = 0; o < FBD; ++o) {
    const int oo = o0 + o;
    if (oo >= p.Co) break;
    const size_t plane = (size_t)n * p.Co + oo;
    const float bs = p.bias ? __ldg(p.bias + oo) : 0.f;
    float v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int rq = r + (q >> 1), cq = c + (q & 1);
      v[q] = acc[o][q] + bs;
      if (skip && rq < p.H && cq < p.W) v[q] += __ldg(skip + (plane * p.H + rq) * p.W + cq);
      if (relu) v[q] = fmaxf(v[q], 0.f);
    }
    if (pool) {
      // H and W are even, so a block inside the image is whole
      if (r < p.H && c < p.W)
        p.y[(plane * (p.H / 2) + r / 2) * (p.W / 2) + c / 2] = fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3]));
    } else {
#pragma unroll
      for (int py = 0; py < 2; ++py) {
        const int rq = r + py;
        if (rq >= p.H) break;
        float* yr = p.y + (plane * p.H + rq) * p.W;
        if ((p.W & 1) == 0 && c + 1 < p.W) {
          *reinterpret_cast<float2*>(yr + c) = make_float2(v[py * 2], v[py * 2 + 1]);
        } else {
          if (c < p.W) yr[c] = v[py * 2];
          if (c + 1 < p.W) yr[c + 1] = v[py * 2 + 1];
        }
      }
    }
  }
}

template <int CC, int FBD>
cudaError_t launch_one(const DirectParams& p, dim3 grid, cudaStream_t stream) {
  constexpr int bytes = 2 * (CC * DTW * DPITCH + CC * FBD * 12) * 4;
  static ppc::DeviceOnce attr_once;  // one per instantiation
  const cudaError_t ea = attr_once.run([](int) {
    return cudaFuncSetAttribute(ppconv_direct_kernel<CC, FBD>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  });
  if (ea != cudaSuccess) return ea;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.gridDim = grid;
  cfg.blockDim = dim3(DTHREADS);
  cfg.dynamicSmemBytes = bytes;
  cfg.stream = stream;
  return cudaLaunchKernelEx(&cfg, ppconv_direct_kernel<CC, FBD>, p);
}

template <int CC>
cudaError_t launch_cc(const DirectParams& p, int fbd, dim3 grid, cudaStream_t stream) {
  switch (fbd) {
    case 1: return launch_one<CC, 1>(p, grid, stream);
    case 2: return launch_one<CC, 2>(p, grid, stream);
    case 4: return launch_one<CC, 4>(p, grid, stream);
    case 8: return launch_one<CC, 8>(p, grid, stream);
    default: return launch_one<CC, 16>(p, grid, stream);
  }
}

int sm_count() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (!sms[dev] && cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return 148;
  }
  return sms[dev];
}

}  // namespace

namespace ppc {

bool direct_applicable(int Co, int Ci) {
  return (Ci <= kDirectMaxSmall || Co <= kDirectMaxSmall) && (int64_t)Co * Ci <= (int64_t(1) << 20);
}

pp_status direct_build(DirectLayout* D, const float* w_dense, const float* bias, int Co, int Ci,
                       cudaStream_t stream) {
  if (!direct_applicable(Co, Ci)) return PP_ERR_UNSUPPORTED;
  const size_t nw = (size_t)Co * Ci * 9, nb = bias ? (size_t)Co : 0;
  void* d = nullptr;
  if (cudaMalloc(&d, (nw + nb) * 4) != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_OOM;
  }
  if (cudaMemcpyAsync(d, w_dense, nw * 4, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      (nb && cudaMemcpyAsync(static_cast<float*>(d) + nw, bias, nb * 4, cudaMemcpyHostToDevice, stream) !=
                 cudaSuccess) ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    cudaFree(d);
    return PP_ERR_CUDA;
  }
  D->dmem = d;
  D->w = static_cast<const float*>(d);
  D->bias = nb ? static_cast<const float*>(d) + nw : nullptr;
  D->Co = Co;
  D->Ci = Ci;
  return PP_OK;
}

pp_status direct_launch(const DirectLayout& D, const float* x, float* y, const float* skip, int N, int H, int W,
                        int flags, cudaStream_t stream) {
  if (!D.w) return PP_ERR_UNSUPPORTED;
  DirectParams p;
  p.x = x;
  p.y = y;
  p.skip = (flags & PP_ADD_SKIP) ? skip : nullptr;
  p.w = D.w;
  p.bias = D.bias;
  p.N = N;
  p.Ci = D.Ci;
  p.Co = D.Co;
  p.H = H;
  p.W = W;
  p.flags = flags;
  p.tiles_x = (W + DT - 1) / DT;
  p.tiles_y = (H + DT - 1) / DT;
  p.vec = (W & 3) == 0 && ((uintptr_t)x & 15) == 0;
  // filters per CTA: up to 16, fewer when the layer has too few tiles to give
  // every SM a few CTAs (the input tile is then staged once per filter block)
  const int64_t nt = (int64_t)N * p.tiles_x * p.tiles_y;
  int fbd = 16;
  while (fbd > 1 && (fbd / 2 >= D.Co || nt * ((D.Co + fbd - 1) / fbd) < 2 * (int64_t)sm_count())) fbd /= 2;
  const int64_t nfb = (D.Co + fbd - 1) / fbd;
  if (nt > INT32_MAX || nfb > 65535) return PP_ERR_UNSUPPORTED;
  const dim3 grid((unsigned)nt, (unsigned)nfb);
  cudaError_t e;
  switch (D.Ci) {
    case 1: e = launch_cc<1>(p, fbd, grid, stream); break;
    case 2: e = launch_cc<2>(p, fbd, grid, stream); break;
    case 3: e = launch_cc<3>(p, fbd, grid, stream); break;
    case 4: e = launch_cc<4>(p, fbd, grid, stream); break;
    default: e = launch_cc<8>(p, fbd, grid, stream); break;  // fewer, larger copy steps
  }
  if (e != cudaSuccess) return PP_ERR_CUDA;
  return PP_OK;
}

void direct_free(DirectLayout* D) {
  if (D->dmem) cudaFree(D->dmem);
  *D = DirectLayout();
}

}  // namespace ppc
