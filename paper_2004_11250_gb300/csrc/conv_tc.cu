// Pattern-pruned 3x3 convolution as an implicit GEMM on the 5th-generation
// tensor cores (tcgen05, kind::tf32), with fp32 accuracy by 3xTF32 splitting.
//
// Method: Niu et al., IJCAI-20 demo, Section 2 (a kept kernel keeps 4 of its 9
// taps; connectivity pruning drops whole kernels) and Section 3 (fused
// activation).  The pruned weights are written densely over the 9 taps (zeros
// where a tap or kernel was pruned), so the layer is D[o][pixel] =
// sum over (input channel i, tap t) of W_t[o][i] * x[i][pixel + offset_t]: a
// dense contraction of depth 9 * Ci, of which a fraction 4 * keep / 9 is
// nonzero.  The tensor cores do ~2.25 / keep times the useful multiplies but at
// ~14x the FP32 FMA rate, which wins for the keep ratios of the workloads.
//
// Precision: tf32 keeps 10 explicit mantissa bits, far from the 1e-5 bound.
// Each operand is split v = hi + lo with hi = v with its low 13 bits cleared
// (exactly representable in tf32) and lo = v - hi (exact in fp32), and the
// product is accumulated as hi*hi + lo*hi + hi*lo in fp32 TMEM accumulators.
// The dropped lo*lo term and the tf32 truncation of lo are below 2^-20 of
// |w * x|.
//
// Per CTA (4 warps, one CTA per SM): M = 128 consecutive reordered filters, R
// output rows x TW columns of pixels (R * TW = 256 TMEM columns, one fp32
// accumulator per filter x pixel).  The K loop runs over 8-channel chunks:
//   * weights for the chunk, 9 taps x {hi, lo} x (128 x 8) in the canonical
//     K-major layout, arrive by one bulk async copy (mbarrier transaction count);
//   * the input tile for the chunk (R + 2 rows x TW + 2 columns, zero halo) is
//     staged channel-innermost with cp.async, then split into hi / lo halves in
//     place by the CTA's threads;
//   * one thread issues 9 taps x 3 passes x R row MMAs of 128 x TW x 8.  A tap
//     (dy, dx) is the same input tile with the operand start moved by dy rows
//     and dx pixels (16 bytes per pixel), so no im2col copy exists;
//   * tcgen05.commit signals an mbarrier when the chunk's MMAs have read their
//     operands, which frees that stage for the chunk after next.
// Epilogue: each thread owns one filter (TMEM lane); it reads its pixels with
// tcgen05.ld and applies bias, +skip, ReLU, 2x2 max pool, storing contiguous
// row segments.  Small grids split the chunks over a cluster and reduce the
// accumulators through distributed shared memory in rank order.
//
// Every wait on an mbarrier is bounded; on timeout the kernel records an error
// in the layer's device status word and skips the rest of its work.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"

namespace {

constexpr int TC_M = 128;          // filters per CTA (MMA M)
constexpr int KC = 8;              // input channels per chunk (MMA K for tf32)
constexpr int NTAP = 9;
constexpr int NCOL = 256;          // TMEM columns = accumulator pixels per CTA
constexpr int NTHREADS = 128;
constexpr int A_TILE = TC_M * KC * 4;             // one tap, one of hi/lo: 4 KB
constexpr int A_BYTES = NTAP * 2 * A_TILE;        // 72 KB per chunk
constexpr int MAX_SPLIT = 8;
constexpr long WAIT_LIMIT = 1L << 24;             // mbarrier polls before giving up

struct TcParams {
  const float* x;
  float* y;
  const float* skip;
  const unsigned char* a;  // [MT][nch][9][2][128 x 8] canonical tiles
  const int* perm;         // [Co]
  const float* bias;       // [Co] reordered, or null
  int* status;             // device status word (nonzero after a timed-out wait)
  int N, Ci, Co, H, W;
  int nch, MT;
  int tiles_x, tiles_y;
  int flags;
  int ksplit, cpk;
};

// Shared-memory matrix descriptor, K-major, no swizzle: core matrices of 8 rows
// x 16 bytes; lbo = byte distance between the two K halves, sbo = between
// groups of 8 rows.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo) {
  uint64_t d = (uint64_t)((addr >> 4) & 0x3FFF);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)(128 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  return d;
}

// Instruction descriptor: D f32, A and B tf32, both K-major, shape M x N.
__host__ __device__ constexpr uint32_t idesc_tf32(int m, int n) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ uint32_t su32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t a, int count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count));
}
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
               : "=r"(ok)
               : "r"(a), "r"(parity)
               : "memory");
  return ok != 0;
}
// Bounded wait; returns false on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity) {
  for (long i = 0; i < WAIT_LIMIT; ++i)
    if (mbar_try(a, parity)) return true;
  return false;
}

__device__ __forceinline__ void cp4(void* s, const void* g, bool valid) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(su32(s)), "l"(g), "r"(valid ? 4 : 0));
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;\n" ::); }
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::); }

__device__ __forceinline__ void tm_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tm_ld16(uint32_t ta, float (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7]), "=f"(v[8]),
        "=f"(v[9]), "=f"(v[10]), "=f"(v[11]), "=f"(v[12]), "=f"(v[13]), "=f"(v[14]), "=f"(v[15])
      : "r"(ta));
}
__device__ __forceinline__ void tm_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void mma_tf32(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p; }" ::"r"(d),
      "l"(a), "l"(b), "r"(id), "r"(acc));
}

template <int TW>
struct Geo {
  static constexpr int R = NCOL / TW;          // output rows per CTA
  static constexpr int BROWS = R + 2;
  static constexpr int BCOLS = TW + 2;
  static constexpr int NPIX = BROWS * BCOLS;   // pixels of the staged input tile
  static constexpr int B_HALF = NPIX * 16;     // bytes of one K half (4 channels) of one of hi / lo
  static constexpr int B_BYTES = 2 * B_HALF;   // hi or lo tile (8 channels)
  static constexpr int STAGE = A_BYTES + 2 * B_BYTES;
  static constexpr int SMEM = 2 * STAGE;
  static constexpr int RED = TC_M * NCOL * 4;  // split-K partial sums of the CTA
  static constexpr int SMEM_ALLOC = (SMEM > RED ? SMEM : RED) + 1024;
};

// Epilogue of 16 consecutive pixels (one row, columns c .. c+15 of the tile) of one filter.
__device__ __forceinline__ void store16(const TcParams& p, int n, int m_global, float (&v)[16], int row, int col) {
  if (m_global >= p.Co || row >= p.H) return;
  const int o = __ldg(p.perm + m_global);
  const float b = p.bias ? __ldg(p.bias + m_global) : 0.f;
#pragma unroll
  for (int k = 0; k < 16; ++k) v[k] += b;
  if (p.flags & PP_ADD_SKIP) {
    const float* sk = p.skip + (((size_t)n * p.Co + o) * p.H + row) * p.W;
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (col + k < p.W) v[k] += __ldg(sk + col + k);
  }
  if (p.flags & PP_RELU) {
#pragma unroll
    for (int k = 0; k < 16; ++k) v[k] = fmaxf(v[k], 0.f);
  }
  float* yo = p.y + (((size_t)n * p.Co + o) * p.H + row) * p.W;
  if (col + 16 <= p.W && (p.W & 3) == 0 && (col & 3) == 0) {
#pragma unroll
    for (int k = 0; k < 16; k += 4) *reinterpret_cast<float4*>(yo + col + k) = make_float4(v[k], v[k + 1], v[k + 2], v[k + 3]);
  } else {
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (col + k < p.W) yo[col + k] = v[k];
  }
}

// Pooled epilogue: rows row, row+1 (a, b), columns col .. col+15 -> 8 outputs.
__device__ __forceinline__ void store16_pool(const TcParams& p, int n, int m_global, float (&a)[16], float (&b)[16],
                                             int row, int col) {
  if (m_global >= p.Co || row >= p.H) return;
  const int o = __ldg(p.perm + m_global);
  const float bs = p.bias ? __ldg(p.bias + m_global) : 0.f;
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    a[k] += bs;
    b[k] += bs;
  }
  if (p.flags & PP_ADD_SKIP) {
    const float* s0 = p.skip + (((size_t)n * p.Co + o) * p.H + row) * p.W;
    const float* s1 = s0 + p.W;
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (col + k < p.W) {
        a[k] += __ldg(s0 + col + k);
        b[k] += __ldg(s1 + col + k);
      }
  }
  if (p.flags & PP_RELU) {
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      a[k] = fmaxf(a[k], 0.f);
      b[k] = fmaxf(b[k], 0.f);
    }
  }
  const int Ho = p.H / 2, Wo = p.W / 2;
  float* yo = p.y + (((size_t)n * p.Co + o) * Ho + (row >> 1)) * Wo;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int pc = (col >> 1) + k;
    if (pc < Wo) yo[pc] = fmaxf(fmaxf(a[2 * k], a[2 * k + 1]), fmaxf(b[2 * k], b[2 * k + 1]));
  }
}

template <int TW, bool SPLIT>
__global__ void __launch_bounds__(NTHREADS, 1) ppconv_tc_kernel(const TcParams p) {
  using G = Geo<TW>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_a[2];    // weights of a stage have arrived
  __shared__ __align__(8) uint64_t bar_mma[2];  // MMAs reading a stage are done
  __shared__ uint32_t tmem_s;
  __shared__ int abort_s;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x;
  const int ty = tile / p.tiles_x, tx = tile - ty * p.tiles_x;
  const int r0 = ty * G::R, c0 = tx * TW;
  const int mt = blockIdx.y;
  const int n = SPLIT ? blockIdx.z / p.ksplit : blockIdx.z;
  const int ks = SPLIT ? blockIdx.z - n * p.ksplit : 0;
  const int cbeg = ks * p.cpk;
  const int cend = min(p.nch, cbeg + p.cpk);

  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      mbar_init(su32(&bar_a[s]), 1);
      mbar_init(su32(&bar_mma[s]), 1);
    }
    abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tmem_s)),
                 "n"(NCOL));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  const uint32_t tmem = tmem_s;

  // Stage s of chunk c: weights by one bulk copy, input tile by cp.async.
  auto load = [&](int c, int s) {
    unsigned char* st = smem + s * G::STAGE;
    if (tid == 0) {
      const unsigned char* src = p.a + ((size_t)mt * p.nch + c) * A_BYTES;
      const uint32_t bar = su32(&bar_a[s]);
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(A_BYTES) : "memory");
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(su32(st)),
          "l"(src), "r"(A_BYTES), "r"(bar)
          : "memory");
    }
    float* bh = reinterpret_cast<float*>(st + A_BYTES);
    const int i0 = c * KC;
    const float* xb = p.x + (size_t)n * p.Ci * p.H * p.W;
    const int total = KC * G::NPIX;
    for (int e = tid; e < total; e += NTHREADS) {
      const int k = e / G::NPIX;
      const int pix = e - k * G::NPIX;
      const int br = pix / G::BCOLS, bc = pix - br * G::BCOLS;
      const int r = r0 - 1 + br, cc = c0 - 1 + bc, ch = i0 + k;
      const bool ok = ch < p.Ci && (unsigned)r < (unsigned)p.H && (unsigned)cc < (unsigned)p.W;
      cp4(bh + (k >> 2) * (G::NPIX * 4) + pix * 4 + (k & 3), ok ? xb + ((size_t)ch * p.H + r) * p.W + cc : p.x, ok);
    }
    cp_commit();
  };

  bool ok = true;
  if (cbeg < cend) load(cbeg, 0);
  for (int c = cbeg; c < cend; ++c) {
    const int s = (c - cbeg) & 1;
    const int use = (c - cbeg) >> 1;  // how many times stage s was used before
    unsigned char* st = smem + s * G::STAGE;
    cp_wait_all();
    __syncthreads();
    // split the input tile into hi (in place) and lo
    {
      float4* bh = reinterpret_cast<float4*>(st + A_BYTES);
      float4* bl = reinterpret_cast<float4*>(st + A_BYTES + G::B_BYTES);
      for (int e = tid; e < 2 * G::NPIX; e += NTHREADS) {
        const float4 v = bh[e];
        float4 h;
        h.x = __uint_as_float(__float_as_uint(v.x) & 0xFFFFE000u);
        h.y = __uint_as_float(__float_as_uint(v.y) & 0xFFFFE000u);
        h.z = __uint_as_float(__float_as_uint(v.z) & 0xFFFFE000u);
        h.w = __uint_as_float(__float_as_uint(v.w) & 0xFFFFE000u);
        bh[e] = h;
        bl[e] = make_float4(v.x - h.x, v.y - h.y, v.z - h.z, v.w - h.w);
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();
    if (tid == 0) {
      if (!mbar_wait(su32(&bar_a[s]), (uint32_t)(use & 1))) abort_s = 1;
      if (!abort_s) {
        tm_fence_after();
        const uint32_t abase = su32(st);
        const uint32_t bhi = su32(st + A_BYTES), blo = su32(st + A_BYTES + G::B_BYTES);
        constexpr uint32_t id = idesc_tf32(TC_M, TW);
#pragma unroll 1
        for (int t = 0; t < NTAP; ++t) {
          const int dy = t / 3, dx = t % 3;
          const uint64_t ahi = smem_desc(abase + (t * 2 + 0) * A_TILE, TC_M * 16);
          const uint64_t alo = smem_desc(abase + (t * 2 + 1) * A_TILE, TC_M * 16);
#pragma unroll 1
          for (int rr = 0; rr < G::R; ++rr) {
            const uint32_t off = (uint32_t)(((rr + dy) * G::BCOLS + dx) * 16);
            const uint64_t bdh = smem_desc(bhi + off, G::B_HALF);
            const uint64_t bdl = smem_desc(blo + off, G::B_HALF);
            const uint32_t d = tmem + (uint32_t)(rr * TW);
            const uint32_t first = (c == cbeg && t == 0) ? 0u : 1u;
            mma_tf32(d, ahi, bdh, id, first);
            mma_tf32(d, alo, bdh, id, 1u);
            mma_tf32(d, ahi, bdl, id, 1u);
          }
        }
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                         su32(&bar_mma[s]))
                     : "memory");
      }
    }
    __syncthreads();
    if (abort_s) {
      ok = false;
      break;
    }
    // Load the chunk after this one into the other stage once the MMAs that
    // read it (chunk c - 1) are done.
    if (c + 1 < cend) {
      const int s2 = s ^ 1;
      if (c > cbeg) {
        const int use2 = (c - 1 - cbeg) >> 1;
        if (!mbar_wait(su32(&bar_mma[s2]), (uint32_t)(use2 & 1))) {
          if (tid == 0) abort_s = 1;
        }
        tm_fence_after();
      }
      __syncthreads();
      if (abort_s) {
        ok = false;
        break;
      }
      load(c + 1, s2);
    }
  }
  // Wait for the last chunk's MMAs (they complete after all earlier ones).
  if (ok && cend > cbeg) {
    const int last = cend - 1 - cbeg;
    if (!mbar_wait(su32(&bar_mma[last & 1]), (uint32_t)((last >> 1) & 1))) ok = false;
    tm_fence_after();
  }
  if (!ok && tid == 0) atomicExch(p.status, 1);
  cp_wait_all();
  __syncthreads();

  // Epilogue: thread = filter (TMEM lane 32 * warp + lane); pixels along columns.
  const int m = warp * 32 + lane;
  const int mg = mt * TC_M + m;
  const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
  const bool pool = p.flags & PP_POOL2;
  if constexpr (!SPLIT) {
    if (ok) {
      if (!pool) {
#pragma unroll 1
        for (int rr = 0; rr < G::R; ++rr)
#pragma unroll 1
          for (int cc = 0; cc < TW; cc += 16) {
            float v[16];
            tm_ld16(lane_addr + (uint32_t)(rr * TW + cc), v);
            tm_wait_ld();
            store16(p, n, mg, v, r0 + rr, c0 + cc);
          }
      } else {
#pragma unroll 1
        for (int rr = 0; rr < G::R; rr += 2)
#pragma unroll 1
          for (int cc = 0; cc < TW; cc += 16) {
            float a[16], b[16];
            tm_ld16(lane_addr + (uint32_t)(rr * TW + cc), a);
            tm_ld16(lane_addr + (uint32_t)((rr + 1) * TW + cc), b);
            tm_wait_ld();
            store16_pool(p, n, mg, a, b, r0 + rr, c0 + cc);
          }
      }
    }
  } else {
    // Split over chunks: every CTA publishes its accumulators [m][column] in
    // shared memory; CTA rank r then reduces the columns with
    // (column / 16) % ksplit == r over ranks 0..ksplit-1 in order.
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    float* red = reinterpret_cast<float*>(smem);
#pragma unroll 1
    for (int col = 0; col < NCOL; col += 16) {
      float v[16];
      tm_ld16(lane_addr + (uint32_t)col, v);
      tm_wait_ld();
#pragma unroll
      for (int k = 0; k < 16; ++k)  // a CTA with no chunk (or a failed wait) contributes zeros
        red[(size_t)m * NCOL + ((col + k + m) & (NCOL - 1))] = (ok && cend > cbeg) ? v[k] : 0.f;
    }
    cluster.sync();
    const int cpr = TW / 16;  // 16-column blocks per row
#pragma unroll 1
    for (int blk = pool ? 0 : rank; blk < NCOL / 16; blk += pool ? 1 : p.ksplit) {
      const int rr = blk / cpr, cc = (blk - rr * cpr) * 16;
      if (pool && ((rr & 1) || ((blk / 2) % p.ksplit) != rank)) continue;
      float a[16], b[16];
#pragma unroll
      for (int k = 0; k < 16; ++k) a[k] = b[k] = 0.f;
#pragma unroll 1
      for (int s2 = 0; s2 < p.ksplit; ++s2) {
        const float* rem = cluster.map_shared_rank(red, s2) + (size_t)m * NCOL;
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          a[k] += rem[(blk * 16 + k + m) & (NCOL - 1)];
          if (pool) b[k] += rem[((blk + cpr) * 16 + k + m) & (NCOL - 1)];
        }
      }
      if (pool)
        store16_pool(p, n, mg, a, b, r0 + rr, c0 + cc);
      else
        store16(p, n, mg, a, r0 + rr, c0 + cc);
    }
    cluster.sync();
  }

  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(NCOL));
}

template <int TW>
cudaError_t set_attr() {
  cudaError_t e = cudaFuncSetAttribute(ppconv_tc_kernel<TW, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Geo<TW>::SMEM_ALLOC);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(ppconv_tc_kernel<TW, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              Geo<TW>::SMEM_ALLOC);
}

bool g_done[64] = {};

cudaError_t prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 64 && g_done[dev]) return cudaSuccess;
  if ((e = set_attr<16>()) != cudaSuccess) return e;
  if ((e = set_attr<32>()) != cudaSuccess) return e;
  if ((e = set_attr<64>()) != cudaSuccess) return e;
  if ((e = set_attr<128>()) != cudaSuccess) return e;
  if (dev < 64) g_done[dev] = true;
  return cudaSuccess;
}

int choose_split(int64_t base_ctas, int nch) {
  const int64_t slots = 152;  // one CTA per SM
  int best = 1;
  double best_t = 1e30;
  for (int ks = 1; ks <= MAX_SPLIT && ks <= nch; ks *= 2) {
    const double waves = (double)((base_ctas * ks + slots - 1) / slots);
    const double t = waves * (double)((nch + ks - 1) / ks) + (ks > 1 ? 1.0 : 0.0);
    if (t < best_t - 1e-9) {
      best_t = t;
      best = ks;
    }
  }
  return best;
}

template <int TW>
cudaError_t launch_tw(const TcParams& p0, int N, cudaStream_t stream) {
  TcParams p = p0;
  using G = Geo<TW>;
  p.tiles_x = (p.W + TW - 1) / TW;
  p.tiles_y = (p.H + G::R - 1) / G::R;
  const int64_t base = (int64_t)p.tiles_x * p.tiles_y * p.MT * N;
  const int ks = choose_split(base, p.nch);
  p.ksplit = ks;
  p.cpk = (p.nch + ks - 1) / ks;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.tiles_x * p.tiles_y, p.MT, N * ks);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = G::SMEM_ALLOC;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  if (ks > 1) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = ks;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, ppconv_tc_kernel<TW, true>, p);
  }
  return cudaLaunchKernelEx(&cfg, ppconv_tc_kernel<TW, false>, p);
}

}  // namespace

namespace ppc {

pp_status tc_prepare() { return prepare() == cudaSuccess ? PP_OK : PP_ERR_CUDA; }

// Dense per-tap weights of every (128-filter tile, 8-channel chunk), split into
// tf32 hi / lo, in the canonical K-major layout: element (filter m, channel k)
// of a 4 KB tile at byte (k / 4) * 2048 + m * 16 + (k % 4) * 4.
pp_status tc_build(TcLayout* T, const pp_packed* pk, cudaStream_t stream) {
  const int Co = pk->Co, Ci = pk->Ci;
  T->MT = (Co + TC_M - 1) / TC_M;
  T->nch = (Ci + KC - 1) / KC;
  const size_t total = (size_t)T->MT * T->nch * A_BYTES;
  std::vector<float> host(total / 4, 0.f);
  for (int j = 0; j < Co; ++j) {
    const int mt = j / TC_M, m = j % TC_M;
    for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e) {
      const int i = pk->kidx[e], c = i / KC, k = i % KC;
      const uint8_t* taps = &pk->taps[4 * pk->kpat[e]];
      for (int s = 0; s < 4; ++s) {
        const float w = pk->kw[(size_t)e * 4 + s];
        uint32_t bits;
        std::memcpy(&bits, &w, 4);
        bits &= 0xFFFFE000u;
        float hi;
        std::memcpy(&hi, &bits, 4);
        const float lo = w - hi;
        const int t = taps[s];
        const size_t base = ((size_t)mt * T->nch + c) * A_BYTES + (size_t)t * 2 * A_TILE;
        const size_t within = (size_t)(k / 4) * (TC_M * 16) + (size_t)m * 16 + (size_t)(k % 4) * 4;
        host[(base + within) / 4] = hi;
        host[(base + A_TILE + within) / 4] = lo;
      }
    }
  }
  void* d = nullptr;
  if (cudaMalloc(&d, total + 256) != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_OOM;
  }
  if (cudaMemsetAsync(static_cast<unsigned char*>(d) + total, 0, 256, stream) != cudaSuccess ||
      cudaMemcpyAsync(d, host.data(), total, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    cudaFree(d);
    return PP_ERR_CUDA;
  }
  T->dmem = d;
  T->dbytes = total + 256;
  T->a = static_cast<const unsigned char*>(d);
  T->status = reinterpret_cast<int*>(static_cast<unsigned char*>(d) + total);
  return PP_OK;
}

pp_status tc_launch(const TcLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N, int H,
                    int W, int flags, cudaStream_t stream) {
  if ((int64_t)N * MAX_SPLIT > 65535 || T.MT > 65535) return PP_ERR_UNSUPPORTED;
  if (prepare() != cudaSuccess) return PP_ERR_CUDA;
  TcParams p;
  p.x = x;
  p.y = y;
  p.skip = (flags & PP_ADD_SKIP) ? skip : nullptr;
  p.a = T.a;
  p.perm = M.perm;
  p.bias = M.bias;
  p.status = T.status;
  p.N = N;
  p.Ci = M.Ci;
  p.Co = M.Co;
  p.H = H;
  p.W = W;
  p.nch = T.nch;
  p.MT = T.MT;
  p.flags = flags;
  cudaError_t e;
  if (W <= 16)
    e = launch_tw<16>(p, N, stream);
  else if (W <= 32)
    e = launch_tw<32>(p, N, stream);
  else if (W <= 64)
    e = launch_tw<64>(p, N, stream);
  else
    e = launch_tw<128>(p, N, stream);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  return PP_OK;
}

pp_status tc_status(const TcLayout& T, int* device_error) {
  int v = 0;
  if (cudaMemcpy(&v, T.status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return PP_ERR_CUDA;
  *device_error = v;
  return PP_OK;
}

}  // namespace ppc
