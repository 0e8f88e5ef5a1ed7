// Pattern-pruned 3x3 convolution with accumulators in Blackwell tensor memory.
//
// Method: Niu et al., IJCAI-20 demo, Section 2 (pattern + connectivity
// pruning) and Section 3 (compact storage, filter reorder, fused activation).
// This is the kernel for layers whose patterns all belong to the ring set (the
// centre tap plus 3 consecutive of its 8 neighbours), so every pattern's taps
// are compile-time constants.
//
// Why tensor memory: a warp owns 16 filter slots x 8 pixels per lane of
// accumulators.  Which slot a kept kernel updates is data, and a register
// file cannot be indexed by data without a branch per kernel (measured on
// GB300: a warp-uniform switch or if-tree per kernel costs ~150 cycles).
// tcgen05.ld / tcgen05.st address TMEM columns with a register, so the slot
// becomes an address instead of code: load the slot's 8 accumulators, apply
// the kernel's 4 taps as 16 packed FFMA2, store them back.  The pattern is
// handled without dispatch by ordering each channel's kernels by pattern and
// running 8 static loops, one per pattern, with the taps unrolled.
//
// Per CTA (8 warps, two CTAs per SM): a 16x32 output tile and 64 consecutive
// reordered filters (4 groups of 16).  Warp w handles group w & 3 (its TMEM
// lane quadrant) on the 16x16 half w >> 2 of the tile (TMEM columns
// 128 * (w >> 2) ...).  Input channels are staged 8 at a time (tile + 1-pixel
// halo, zero padded) with cp.async, double buffered, together with each
// group's entry blob for those channels:
//   [8 x 8 bytes: per channel, cumulative entry count after each pattern]
//   [n bytes: slot of each entry, padded to 16]
//   [n x 16 bytes: the 4 weights of each entry, in the pattern's tap order]
// A lane loads its 3x10 input window once per channel and reuses it for every
// kept kernel of that channel in its group.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"

namespace {

constexpr int F = 16;          // filter slots per warp (one group)
constexpr int PX = 8;          // pixels per lane: one row segment
constexpr int NWARP = 8;
constexpr int NTHREADS = 32 * NWARP;
constexpr int GROUPS = 4;      // filter groups per CTA (one per TMEM lane quadrant)
constexpr int TILE_H = 16, TILE_W = 32;
constexpr int CC = 8;          // input channels per stage
constexpr int SROWS = TILE_H + 2;
constexpr int SCOLS = TILE_W + 2;
constexpr int SSTRIDE = 36;    // floats; 9 x 16 B, so 8 consecutive rows hit 8 distinct 16-B bank groups
constexpr int SCH = SROWS * SSTRIDE;
constexpr int IN_BYTES = CC * SCH * 4;
constexpr int EMAX = F * CC;                              // entries of a group per stage
constexpr int BLOB_MAX = 64 + EMAX + EMAX * 16;           // bounds + slots + weights
constexpr int STAGE_BYTES = IN_BYTES + GROUPS * BLOB_MAX;
constexpr int PIPE_BYTES = 2 * STAGE_BYTES;
constexpr int RED_BYTES = NWARP * 8 * PX * 32 * 4;        // split-K partials, 8 slots at a time
// Two CTAs per SM share the 512 TMEM columns; the shared-memory request alone
// keeps a third CTA off the SM so tcgen05.alloc never waits.
constexpr int SMEM_BYTES = 80 * 1024;
static_assert(PIPE_BYTES <= SMEM_BYTES && RED_BYTES <= SMEM_BYTES, "shared memory plan");
static_assert(3 * SMEM_BYTES > 228 * 1024, "at most two CTAs per SM");
constexpr int TMEM_COLS = 256;
constexpr int MAX_SPLIT = 8;

struct TmParams {
  const float* x;
  float* y;
  const float* skip;
  const uint4* blob;   // entry blobs, 16-byte units
  const int* boff;     // [G][nch + 1] blob offsets (16-byte units)
  const int* perm;
  const float* bias;
  int N, Ci, Co, H, W;
  int nch, G;
  int tiles_x;
  int flags;
  int ksplit, cpk;
  int khalf;  // 1: maps at most 16 wide; the two warps of a group split each stage's channels
};

__host__ __device__ constexpr int ring_tap(int r, int s) {
  return r == 0 ? (s == 0 ? 0 : s == 1 ? 1 : s == 2 ? 2 : 4)
       : r == 1 ? (s == 0 ? 1 : s == 1 ? 2 : s == 2 ? 4 : 5)
       : r == 2 ? (s == 0 ? 2 : s == 1 ? 4 : s == 2 ? 5 : 8)
       : r == 3 ? (s == 0 ? 4 : s == 1 ? 5 : s == 2 ? 7 : 8)
       : r == 4 ? (s == 0 ? 4 : s == 1 ? 6 : s == 2 ? 7 : 8)
       : r == 5 ? (s == 0 ? 3 : s == 1 ? 4 : s == 2 ? 6 : 7)
       : r == 6 ? (s == 0 ? 0 : s == 1 ? 3 : s == 2 ? 4 : 6)
       :          (s == 0 ? 0 : s == 1 ? 1 : s == 2 ? 3 : 4);
}

// ---- tensor memory ---------------------------------------------------------
__device__ __forceinline__ void tm_ld8(uint32_t taddr, float (&v)[PX]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7])
               : "r"(taddr));
}
__device__ __forceinline__ void tm_st8(uint32_t taddr, const float (&v)[PX]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "f"(v[0]),
               "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]));
}
__device__ __forceinline__ void tm_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tm_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// ---- cp.async --------------------------------------------------------------
__device__ __forceinline__ void cp4(void* s, const void* g, bool valid) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"((unsigned)__cvta_generic_to_shared(s)), "l"(g),
               "r"(valid ? 4 : 0));
}
__device__ __forceinline__ void cp16(void* s, const void* g) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"((unsigned)__cvta_generic_to_shared(s)), "l"(g));
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

// Input channels [i0, i0 + nvalid) of image n: rows r0-1 .. r0+16, cols c0-1 .. c0+32.
__device__ __forceinline__ void stage_input(float* s, const TmParams& p, int n, int i0, int nvalid, int r0, int c0) {
  const int total = nvalid * SROWS * SCOLS;
  const float* xb = p.x + ((size_t)n * p.Ci + i0) * p.H * p.W;
  for (int e = threadIdx.x; e < total; e += NTHREADS) {
    const int ch = e / (SROWS * SCOLS);
    const int rem = e - ch * (SROWS * SCOLS);
    const int sr = rem / SCOLS;
    const int sc = rem - sr * SCOLS;
    const int r = r0 - 1 + sr, c = c0 - 1 + sc;
    const bool ok = (unsigned)r < (unsigned)p.H && (unsigned)c < (unsigned)p.W;
    cp4(s + ch * SCH + sr * SSTRIDE + sc, ok ? xb + ((size_t)ch * p.H + r) * p.W + c : p.x, ok);
  }
}

// One kernel (4 taps of ring pattern R) on 8 pixels, as 4 x 4 packed FMAs.
// E[dy][m] = input pair (2m, 2m+1) of window row dy; O[dy][m] = (2m+1, 2m+2).
template <int R>
__device__ __forceinline__ void apply_ring(float2 (&a)[4], const float2 (&E)[3][5], const float2 (&O)[3][4],
                                           const float4& w) {
  const float ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int s = 0; s < 4; ++s) {
    const int t = ring_tap(R, s);
    const int dy = t / 3, dx = t % 3;
    const float2 wp = make_float2(ws[s], ws[s]);
#pragma unroll
    for (int m = 0; m < 4; ++m) a[m] = __ffma2_rn(wp, dx == 1 ? O[dy][m] : E[dy][m + dx / 2], a[m]);
  }
}

// All entries of one pattern for the current channel: e runs up to `end`.
template <int R>
__device__ __forceinline__ void run_pattern(int& e, int end, const unsigned char* slots, const float4* wts,
                                            uint32_t wbase, const float2 (&E)[3][5], const float2 (&O)[3][4]) {
  for (; e < end; ++e) {
    const uint32_t ta = wbase + (uint32_t)slots[e] * PX;
    const float4 w = wts[e];
    float v[PX];
    tm_ld8(ta, v);
    tm_wait_ld();
    float2 a[4] = {make_float2(v[0], v[1]), make_float2(v[2], v[3]), make_float2(v[4], v[5]),
                   make_float2(v[6], v[7])};
    apply_ring<R>(a, E, O, w);
    const float o[PX] = {a[0].x, a[0].y, a[1].x, a[1].y, a[2].x, a[2].y, a[3].x, a[3].y};
    tm_st8(ta, o);
  }
}

// Epilogue of one slot (all 32 lanes): bias, +skip, ReLU, 2x2 max pool, store.
__device__ __forceinline__ void epilogue_slot(const TmParams& p, int n, int jr, float (&v)[PX], int r, int cb,
                                              int ly) {
  const int o = __ldg(p.perm + jr);
  const float b = p.bias ? __ldg(p.bias + jr) : 0.f;
  const bool pool = p.flags & PP_POOL2;
  const int Ho = pool ? p.H / 2 : p.H, Wo = pool ? p.W / 2 : p.W;
#pragma unroll
  for (int k = 0; k < PX; ++k) v[k] += b;
  if ((p.flags & PP_ADD_SKIP) && r < p.H) {
    const float* sk = p.skip + (((size_t)n * p.Co + o) * p.H + r) * p.W;
#pragma unroll
    for (int k = 0; k < PX; ++k)
      if (cb + k < p.W) v[k] += __ldg(sk + cb + k);
  }
  if (p.flags & PP_RELU) {
#pragma unroll
    for (int k = 0; k < PX; ++k) v[k] = fmaxf(v[k], 0.f);
  }
  if (pool) {
    float u[PX];
#pragma unroll
    for (int k = 0; k < PX; ++k) u[k] = __shfl_down_sync(0xffffffffu, v[k], 1);
    if ((ly & 1) == 0 && r < p.H) {
      float* yo = p.y + (((size_t)n * p.Co + o) * Ho + (r >> 1)) * Wo;
#pragma unroll
      for (int m = 0; m < PX / 2; ++m) {
        const int pc = (cb >> 1) + m;
        if (pc < Wo) yo[pc] = fmaxf(fmaxf(v[2 * m], v[2 * m + 1]), fmaxf(u[2 * m], u[2 * m + 1]));
      }
    }
  } else if (r < p.H) {
    float* yo = p.y + (((size_t)n * p.Co + o) * Ho + r) * Wo;
    if (cb + PX <= p.W && (p.W & 3) == 0) {
      reinterpret_cast<float4*>(yo + cb)[0] = make_float4(v[0], v[1], v[2], v[3]);
      reinterpret_cast<float4*>(yo + cb)[1] = make_float4(v[4], v[5], v[6], v[7]);
    } else {
#pragma unroll
      for (int k = 0; k < PX; ++k)
        if (cb + k < p.W) yo[cb + k] = v[k];
    }
  }
}

template <bool SPLIT>
__global__ void __launch_bounds__(NTHREADS, 2) ppconv_tm_kernel(const TmParams p) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ uint32_t tmem_base_s;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int gq = warp & 3;   // group within the CTA = TMEM lane quadrant
  const int sub = warp >> 2;  // 16-column half of the tile, or (khalf) half of each stage's channels
  const int ly = lane & 15, lx = lane >> 4;
  const int ty = blockIdx.x / p.tiles_x, tx = blockIdx.x - ty * p.tiles_x;
  const int tile_w = p.khalf ? 16 : TILE_W;
  const int r0 = ty * TILE_H, c0 = tx * tile_w;
  const int cw = p.khalf ? 0 : sub * 16;  // this warp's column offset in the tile
  const int n = SPLIT ? blockIdx.z / p.ksplit : blockIdx.z;
  const int ks = SPLIT ? blockIdx.z - n * p.ksplit : 0;
  const int q = blockIdx.y * GROUPS + gq;
  const bool grp = q < p.G;                          // the group exists
  const bool compute = grp && c0 + cw < p.W;         // the warp's pixels overlap the image
  const int chb = p.khalf ? sub * (CC / 2) : 0;      // channels of each stage this warp processes
  const int che = p.khalf ? chb + CC / 2 : CC;

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     (unsigned)__cvta_generic_to_shared(&tmem_base_s)),
                 "n"(TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  const uint32_t tbase = tmem_base_s;
  const uint32_t wbase = tbase + ((uint32_t)(32 * gq) << 16) + (uint32_t)(sub * F * PX);
  {
    const float z[PX] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
    for (int j = 0; j < F; ++j) tm_st8(wbase + j * PX, z);
    tm_wait_st();
  }

  const int* boff = p.boff + (size_t)(grp ? q : 0) * (p.nch + 1);
  const int cbeg = ks * p.cpk;
  const int cend = min(p.nch, cbeg + p.cpk);

  auto issue = [&](int c) {
    unsigned char* st = smem + (c & 1) * STAGE_BYTES;
    stage_input(reinterpret_cast<float*>(st), p, n, c * CC, min(CC, p.Ci - c * CC), r0, c0);
    if (grp) {
      // the two warps of a group split the blob copy
      const int b0 = __ldg(boff + c), b1 = __ldg(boff + c + 1);
      uint4* dst = reinterpret_cast<uint4*>(st + IN_BYTES + gq * BLOB_MAX);
      for (int u = b0 + sub * 32 + lane; u < b1; u += 64) cp16(dst + (u - b0), p.blob + u);
    }
    cp_commit();
  };

  if (cbeg < cend) issue(cbeg);
  for (int c = cbeg; c < cend; ++c) {
    if (c + 1 < cend) {
      issue(c + 1);
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    if (compute) {
      const unsigned char* st = smem + (c & 1) * STAGE_BYTES;
      const float* sin = reinterpret_cast<const float*>(st) + ly * SSTRIDE + cw + lx * PX;
      const unsigned char* blob = st + IN_BYTES + gq * BLOB_MAX;
      const unsigned char* bnd = blob;  // [CC][8]
      const int ntot = bnd[CC * 8 - 1];
      const unsigned char* slots = blob + 64;
      const float4* wts = reinterpret_cast<const float4*>(blob + 64 + ((ntot + 15) & ~15));
      const int nvalid = min(che, p.Ci - c * CC);
      int e = chb > 0 ? bnd[(chb - 1) * 8 + 7] : 0;
      for (int ch = chb; ch < nvalid; ++ch) {
        const unsigned char* bc = bnd + ch * 8;
        if (bc[7] == e) continue;  // no kept kernel of this group reads channel ch
        // A slot updated in an earlier channel may be read again here: let its
        // stores land first (within one channel every slot appears once).
        tm_wait_st();
        const float* s = sin + ch * SCH;
        float2 E[3][5], O[3][4];
#pragma unroll
        for (int a = 0; a < 3; ++a) {
          const float4 u = *reinterpret_cast<const float4*>(s + a * SSTRIDE);
          const float4 v = *reinterpret_cast<const float4*>(s + a * SSTRIDE + 4);
          const float2 z = *reinterpret_cast<const float2*>(s + a * SSTRIDE + 8);
          E[a][0] = make_float2(u.x, u.y);
          E[a][1] = make_float2(u.z, u.w);
          E[a][2] = make_float2(v.x, v.y);
          E[a][3] = make_float2(v.z, v.w);
          E[a][4] = z;
          O[a][0] = make_float2(u.y, u.z);
          O[a][1] = make_float2(u.w, v.x);
          O[a][2] = make_float2(v.y, v.z);
          O[a][3] = make_float2(v.w, z.x);
        }
        run_pattern<0>(e, bc[0], slots, wts, wbase, E, O);
        run_pattern<1>(e, bc[1], slots, wts, wbase, E, O);
        run_pattern<2>(e, bc[2], slots, wts, wbase, E, O);
        run_pattern<3>(e, bc[3], slots, wts, wbase, E, O);
        run_pattern<4>(e, bc[4], slots, wts, wbase, E, O);
        run_pattern<5>(e, bc[5], slots, wts, wbase, E, O);
        run_pattern<6>(e, bc[6], slots, wts, wbase, E, O);
        run_pattern<7>(e, bc[7], slots, wts, wbase, E, O);
      }
    }
    __syncthreads();
  }
  // Every warp's accumulators are final once its stores have landed.
  tm_wait_st();
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (p.khalf) {
    // The two warps of a group hold partial sums over different channels for
    // the same pixels (same TMEM lanes): warp sub 0 adds its partner's columns.
    if (grp && sub == 0) {
      const uint32_t partner = tbase + ((uint32_t)(32 * gq) << 16) + (uint32_t)(F * PX);
#pragma unroll 1
      for (int j = 0; j < F; ++j) {
        float a[PX], b[PX];
        tm_ld8(wbase + j * PX, a);
        tm_ld8(partner + j * PX, b);
        tm_wait_ld();
#pragma unroll
        for (int k = 0; k < PX; ++k) a[k] += b[k];
        tm_st8(wbase + j * PX, a);
      }
      tm_wait_st();
    }
    tm_fence_before();
    __syncthreads();
    tm_fence_after();
  }
  const bool fin = grp && (p.khalf ? sub == 0 : compute);  // warps that finalize outputs

  const int r = r0 + ly;
  const int cb = c0 + cw + lx * PX;
  if constexpr (!SPLIT) {
    if (fin) {
#pragma unroll 1
      for (int j = 0; j < F; ++j) {
        const int jr = q * F + j;
        if (jr >= p.Co) break;  // warp-uniform
        float v[PX];
        tm_ld8(wbase + j * PX, v);
        tm_wait_ld();
        epilogue_slot(p, n, jr, v, r, cb, ly);
      }
    }
  } else {
    // Split over input chunks: in two rounds of 8 slots, publish the partial
    // sums in shared memory, then each CTA of the cluster reduces the slots
    // j with j % ksplit == its rank, reading ranks 0..ksplit-1 in order.
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    float* red = reinterpret_cast<float*>(smem);
#pragma unroll 1
    for (int half = 0; half < 2; ++half) {
#pragma unroll 1
      for (int jj = 0; jj < 8; ++jj) {
        float v[PX];
        tm_ld8(wbase + (half * 8 + jj) * PX, v);
        tm_wait_ld();
#pragma unroll
        for (int k = 0; k < PX; ++k) red[((warp * 8 + jj) * PX + k) * 32 + lane] = v[k];
      }
      cluster.sync();
      if (fin) {
#pragma unroll 1
        for (int jj = 0; jj < 8; ++jj) {
          const int j = half * 8 + jj;
          const int jr = q * F + j;
          if (jr >= p.Co) break;
          if (j % p.ksplit != rank) continue;  // warp-uniform
          float v[PX];
#pragma unroll
          for (int k = 0; k < PX; ++k) v[k] = 0.f;
#pragma unroll 1
          for (int s2 = 0; s2 < p.ksplit; ++s2) {
            const float* rem = cluster.map_shared_rank(red, s2);
#pragma unroll
            for (int k = 0; k < PX; ++k) v[k] += rem[((warp * 8 + jj) * PX + k) * 32 + lane];
          }
          epilogue_slot(p, n, jr, v, r, cb, ly);
        }
      }
      cluster.sync();
    }
  }

  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tbase), "n"(TMEM_COLS));
}

// Number of CTAs sharing one output tile (split over input chunks), chosen by
// a small cost model: resident waves (two CTAs per SM) x chunks per CTA, plus
// about one chunk of work for the cluster reduction when split.
int choose_split(int64_t base_ctas, int nch) {
  const int64_t slots = 2 * 152;
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


ppc::DeviceOnce g_attr_once;

cudaError_t prepare() {
  return g_attr_once.run([](int) {
    const cudaError_t e =
        cudaFuncSetAttribute(ppconv_tm_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(ppconv_tm_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  });
}

}  // namespace

namespace ppc {

bool tm_supports(const uint8_t* taps, int P, std::vector<int>& ring_of) {
  ring_of.assign(P, -1);
  for (int p = 0; p < P; ++p) {
    const uint16_t m = tap_mask(taps + 4 * p);
    for (int r = 0; r < 8; ++r) {
      uint8_t rt[4];
      for (int s = 0; s < 4; ++s) rt[s] = (uint8_t)ring_tap(r, s);
      if (tap_mask(rt) == m) ring_of[p] = r;
    }
    if (ring_of[p] < 0) return false;
  }
  return true;
}

pp_status tm_prepare() { return prepare() == cudaSuccess ? PP_OK : PP_ERR_CUDA; }

// Build the entry blobs of every (group, chunk) and upload them.
pp_status tm_build(TmLayout* T, const pp_packed* pk, const std::vector<int>& ring_of, cudaStream_t stream) {
  const int Co = pk->Co, Ci = pk->Ci;
  T->G = (Co + F - 1) / F;
  T->nch = (Ci + CC - 1) / CC;
  struct E {
    int ch, ring, slot;
    const float* w;
  };
  std::vector<int> boff((size_t)T->G * (T->nch + 1));
  std::vector<unsigned char> blob;
  std::vector<std::vector<E>> per_chunk(T->nch);
  for (int q = 0; q < T->G; ++q) {
    for (auto& v : per_chunk) v.clear();
    for (int j = q * F; j < std::min(Co, (q + 1) * F); ++j)
      for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e) {
        const int ch = pk->kidx[e];
        per_chunk[ch / CC].push_back(E{ch, ring_of[pk->kpat[e]], j - q * F, &pk->kw[(size_t)e * 4]});
      }
    for (int c = 0; c < T->nch; ++c) {
      std::vector<E>& es = per_chunk[c];
      std::sort(es.begin(), es.end(), [](const E& a, const E& b) {
        if (a.ch != b.ch) return a.ch < b.ch;
        if (a.ring != b.ring) return a.ring < b.ring;
        return a.slot < b.slot;
      });
      const int nent = (int)es.size();
      if (nent > EMAX) return PP_ERR_UNSUPPORTED;
      boff[(size_t)q * (T->nch + 1) + c] = (int)(blob.size() / 16);
      const size_t base = blob.size();
      const size_t slots_pad = (nent + 15) & ~15;
      blob.resize(base + 64 + slots_pad + (size_t)nent * 16, 0);
      unsigned char* b = blob.data() + base;
      int k = 0;
      for (int ch = 0; ch < CC; ++ch)
        for (int r = 0; r < 8; ++r) {
          while (k < nent && es[k].ch - c * CC == ch && es[k].ring == r) ++k;
          b[ch * 8 + r] = (unsigned char)k;
        }
      for (int i = 0; i < nent; ++i) {
        b[64 + i] = (unsigned char)es[i].slot;
        std::memcpy(b + 64 + slots_pad + (size_t)i * 16, es[i].w, 16);
      }
    }
    boff[(size_t)q * (T->nch + 1) + T->nch] = (int)(blob.size() / 16);
  }
  if (blob.empty()) blob.resize(16, 0);
  const size_t off_boff = 0;
  const size_t off_blob = (boff.size() * 4 + 255) / 256 * 256;
  const size_t total = off_blob + blob.size();
  std::vector<unsigned char> host(total, 0);
  std::memcpy(host.data() + off_boff, boff.data(), boff.size() * 4);
  std::memcpy(host.data() + off_blob, blob.data(), blob.size());
  void* d = nullptr;
  if (cudaMalloc(&d, total) != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_OOM;
  }
  if (cudaMemcpyAsync(d, host.data(), total, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    cudaFree(d);
    return PP_ERR_CUDA;
  }
  T->dmem = d;
  T->dbytes = total;
  T->boff = reinterpret_cast<int*>(static_cast<unsigned char*>(d) + off_boff);
  T->blob = reinterpret_cast<uint4*>(static_cast<unsigned char*>(d) + off_blob);
  return PP_OK;
}

pp_status tm_launch(const TmLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N, int H,
                    int W, int flags, cudaStream_t stream) {
  const int khalf = W <= 16 ? 1 : 0;
  const int tile_w = khalf ? 16 : TILE_W;
  const int tiles_y = (H + TILE_H - 1) / TILE_H, tiles_x = (W + tile_w - 1) / tile_w;
  if ((int64_t)tiles_y * tiles_x > INT32_MAX) return PP_ERR_UNSUPPORTED;
  TmParams p;
  p.khalf = khalf;
  p.x = x;
  p.y = y;
  p.skip = (flags & PP_ADD_SKIP) ? skip : nullptr;
  p.blob = T.blob;
  p.boff = T.boff;
  p.perm = M.perm;
  p.bias = M.bias;
  p.N = N;
  p.Ci = M.Ci;
  p.Co = M.Co;
  p.H = H;
  p.W = W;
  p.nch = T.nch;
  p.G = T.G;
  p.tiles_x = tiles_x;
  p.flags = flags;
  const int cgroups = (T.G + GROUPS - 1) / GROUPS;
  const int64_t base = (int64_t)tiles_y * tiles_x * cgroups * N;
  const int ks = choose_split(base, T.nch);
  p.ksplit = ks;
  p.cpk = (T.nch + ks - 1) / ks;
  if ((int64_t)N * ks > 65535 || cgroups > 65535) return PP_ERR_UNSUPPORTED;
  if (prepare() != cudaSuccess) return PP_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles_y * tiles_x, cgroups, N * ks);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  cudaError_t e;
  if (ks > 1) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = ks;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, ppconv_tm_kernel<true>, p);
  } else {
    e = cudaLaunchKernelEx(&cfg, ppconv_tm_kernel<false>, p);
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  return PP_OK;
}

}  // namespace ppc
