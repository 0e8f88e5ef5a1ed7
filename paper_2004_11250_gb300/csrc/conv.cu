// Pattern- and connectivity-pruned 3x3 convolution on sm_103a (FP32 SIMT).
//
// Method: Niu et al., IJCAI-20 demo.  Section 2: a kept kernel keeps 4 of its 9
// taps (one pattern of a small set); connectivity pruning drops whole kernels.
// Section 3: compact storage (pattern id + 4 weights per kept kernel), filter
// reorder so similar filters sit together, and convolution fused with its
// activation.
//
// Kernel design (GB300-first, not the paper's mobile code generator):
//   * A warp owns kSlots consecutive reordered filters ("slots") and a 16x16
//     output tile; a lane owns one row segment of 8 pixels, so its
//     accumulators are acc[16][8] registers, indexed only by compile-time
//     constants.
//   * Input channels are staged 16 at a time into shared memory (tile + 1-pixel
//     halo, zero padding) with cp.async, double buffered; each warp stages the
//     entries of its filter group for the same channels next to them, so the
//     entry stream is read from shared memory one entry ahead of its use.
//   * Small grids (late VGG layers) split the input channels over the CTAs of
//     a thread-block cluster; the partial accumulators are summed through
//     distributed shared memory in a fixed rank order (deterministic) and the
//     epilogue of each slot runs on one CTA of the cluster.
//   * Per input channel a lane loads its 3x10 input window once into
//     registers and reuses it for every kept kernel of that channel in its
//     filter group: this reuse across filters is what keeps the FMA pipe fed
//     instead of the shared-memory port.
//   * The kept kernels of a warp's filter group form one entry stream, sorted
//     by input channel (the reorder and compaction of Section 3 decide which
//     filters share a stream and keep adjacent streams equally long).  An
//     entry is (channel, slot, pattern) + 4 weights; the (slot, pattern) pair
//     selects a fully unrolled 4-tap x 8-pixel FMA block through one
//     warp-uniform switch.  For the ring set of 8 centre-based patterns the
//     taps are compile-time constants; any other pattern set goes through a
//     per-tap switch (slower, same results).
//   * Epilogue: bias, optional residual add, ReLU, optional 2x2 max pool (the
//     partner row comes from the neighbouring lane by shuffle), store to the
//     filter's original channel.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"

namespace {

constexpr int F = ppc::kSlots;   // filter slots per warp
constexpr int PX = 8;            // pixels per lane (one row segment)
constexpr int TH = 16;           // output tile rows (lanes 0..15 of a half)
constexpr int TW = 16;           // output tile cols (2 lane columns x 8)
constexpr int NWF = 4;           // warps (filter groups) per CTA
constexpr int CC = ppc::kChunk;  // input channels per stage
constexpr int SROWS = TH + 2;
constexpr int SCOLS = TW + 2;
constexpr int SSTRIDE = 20;      // row stride (floats): 16B aligned, conflict-free LDS.128 per 8-lane phase
constexpr int SCH = SROWS * SSTRIDE;
constexpr int STAGE_IN = CC * SCH;           // input floats per stage
constexpr int EMAX = F * CC;                 // most entries a warp can have per stage
constexpr int NTHREADS = 32 * NWF;
// Stage layout in bytes: [weights NWF][EMAX] float4 | input [CC][SROWS][SSTRIDE] | codes [NWF][EMAX] u32
constexpr int OFF_WTS = 0;
constexpr int OFF_IN = OFF_WTS + NWF * EMAX * 16;
constexpr int OFF_CODE = OFF_IN + STAGE_IN * 4;
constexpr int STAGE_BYTES = OFF_CODE + NWF * EMAX * 4;
constexpr int SMEM_BYTES = 2 * STAGE_BYTES;
constexpr int RED_BYTES = NWF * F * PX * 32 * 4;  // split-K partials of one CTA
static_assert(RED_BYTES <= SMEM_BYTES, "split-K partials must fit in the stage buffers");
constexpr int MAX_SPLIT = 8;

enum Mode { MODE_RING8 = 0, MODE_GENERIC = 1 };

// The ring set: centre (tap 4) plus 3 consecutive neighbours in the ring order
// 0,1,2,5,8,7,6,3 around the centre.
__host__ __device__ constexpr int ring_tap(int r, int s) {
  // taps of ring pattern r in ascending order
  return r == 0 ? (s == 0 ? 0 : s == 1 ? 1 : s == 2 ? 2 : 4)
       : r == 1 ? (s == 0 ? 1 : s == 1 ? 2 : s == 2 ? 4 : 5)
       : r == 2 ? (s == 0 ? 2 : s == 1 ? 4 : s == 2 ? 5 : 8)
       : r == 3 ? (s == 0 ? 4 : s == 1 ? 5 : s == 2 ? 7 : 8)
       : r == 4 ? (s == 0 ? 4 : s == 1 ? 6 : s == 2 ? 7 : 8)
       : r == 5 ? (s == 0 ? 3 : s == 1 ? 4 : s == 2 ? 6 : 7)
       : r == 6 ? (s == 0 ? 0 : s == 1 ? 3 : s == 2 ? 4 : 6)
       :          (s == 0 ? 0 : s == 1 ? 1 : s == 2 ? 3 : 4);
}

struct ConvParams {
  const float* x;        // [N][Ci][H][W]
  float* y;              // [N][Co][H'][W']
  const float* skip;     // [N][Co][H][W] or null
  const int* cofs;       // [G][nch + 1] entry offsets per (group, chunk)
  const uint32_t* code;  // [nE]
  const float4* wts;     // [nE]
  const int* perm;       // [Co]
  const float* bias;     // [Co] in reordered order, or null
  int N, Ci, Co, H, W;
  int nch, G;
  int tiles_x;
  int flags;
  int cc;      // input channels per stage (<= CC; entries per warp and stage stay <= EMAX)
  int ksplit;  // CTAs of a cluster sharing one output tile (split over input chunks)
  int cpk;     // input chunks per split
};

// Entry code layout: bits 0..15 pattern payload (MODE_RING8: ring index;
// MODE_GENERIC: 4 taps x 4 bits), 16..19 slot, 20..27 channel within the stage,
// 28..29 number of taps - 1 (MODE_GENERIC).
__device__ __forceinline__ int code_slot(uint32_t c) { return (c >> 16) & 15; }
__device__ __forceinline__ int code_ch(uint32_t c) { return (c >> 20) & 255; }

template <int T>
__device__ __forceinline__ void tap_fma(float (&a)[PX], const float (&win)[3][PX + 2], float w) {
  constexpr int dy = T / 3, dx = T % 3;
#pragma unroll
  for (int k = 0; k < PX; ++k) a[k] = fmaf(w, win[dy][k + dx], a[k]);
}

template <int R>
__device__ __forceinline__ void ring_fma(float (&a)[PX], const float (&win)[3][PX + 2], const float4& w) {
  tap_fma<ring_tap(R, 0)>(a, win, w.x);
  tap_fma<ring_tap(R, 1)>(a, win, w.y);
  tap_fma<ring_tap(R, 2)>(a, win, w.z);
  tap_fma<ring_tap(R, 3)>(a, win, w.w);
}

__device__ __forceinline__ void cp_async4(float* sdst, const float* gsrc, bool valid) {
  unsigned saddr = (unsigned)__cvta_generic_to_shared(sdst);
  int n = valid ? 4 : 0;
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(saddr), "l"(gsrc), "r"(n));
}
__device__ __forceinline__ void cp_async16(void* sdst, const void* gsrc) {
  unsigned saddr = (unsigned)__cvta_generic_to_shared(sdst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(saddr), "l"(gsrc));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

// Stage input channels [i0, i0 + nvalid) of image n, rows r0-1..r0+TH, cols
// c0-1..c0+TW, into `s` (zero outside the image), one 4-byte cp.async each.
__device__ __forceinline__ void stage_input(float* s, const ConvParams& p, int n, int i0, int nvalid, int r0,
                                            int c0) {
  const int total = nvalid * SROWS * SCOLS;
  const float* xb = p.x + ((size_t)n * p.Ci + i0) * p.H * p.W;
  for (int e = threadIdx.x; e < total; e += NTHREADS) {
    const int ch = e / (SROWS * SCOLS);
    const int rem = e - ch * (SROWS * SCOLS);
    const int sr = rem / SCOLS;
    const int sc = rem - sr * SCOLS;
    const int r = r0 - 1 + sr, c = c0 - 1 + sc;
    const bool ok = (unsigned)r < (unsigned)p.H && (unsigned)c < (unsigned)p.W;
    const float* src = ok ? xb + ((size_t)ch * p.H + r) * p.W + c : p.x;
    cp_async4(s + ch * SCH + sr * SSTRIDE + sc, src, ok);
  }
}

// Stage the entries [e0, e1) of this warp's filter group (at most EMAX) into
// the warp's own slice of the stage.
__device__ __forceinline__ void stage_entries(unsigned char* stage, const ConvParams& p, int warp, int lane, int e0,
                                              int e1) {
  float4* sw = reinterpret_cast<float4*>(stage + OFF_WTS) + warp * EMAX;
  uint32_t* sc = reinterpret_cast<uint32_t*>(stage + OFF_CODE) + warp * EMAX;
  for (int e = e0 + lane; e < e1; e += 32) {
    cp_async16(sw + (e - e0), p.wts + e);
    cp_async4(reinterpret_cast<float*>(sc + (e - e0)), reinterpret_cast<const float*>(p.code + e), true);
  }
}

template <int MODE>
__device__ __forceinline__ void dispatch(float (&acc)[F][PX], const float (&win)[3][PX + 2], uint32_t code,
                                         float4 w) {
  if constexpr (MODE == MODE_RING8) {
    const int cs = code_slot(code) * 8 + (code & 7);
    switch (cs) {
#define PP_RING_CASE(J, R) \
  case (J)*8 + (R): ring_fma<R>(acc[J], win, w); break;
#define PP_RING_SLOT(J) \
  PP_RING_CASE(J, 0) PP_RING_CASE(J, 1) PP_RING_CASE(J, 2) PP_RING_CASE(J, 3) \
  PP_RING_CASE(J, 4) PP_RING_CASE(J, 5) PP_RING_CASE(J, 6) PP_RING_CASE(J, 7)
      PP_RING_SLOT(0) PP_RING_SLOT(1) PP_RING_SLOT(2) PP_RING_SLOT(3)
      PP_RING_SLOT(4) PP_RING_SLOT(5) PP_RING_SLOT(6) PP_RING_SLOT(7)
      PP_RING_SLOT(8) PP_RING_SLOT(9) PP_RING_SLOT(10) PP_RING_SLOT(11)
      PP_RING_SLOT(12) PP_RING_SLOT(13) PP_RING_SLOT(14) PP_RING_SLOT(15)
#undef PP_RING_SLOT
#undef PP_RING_CASE
      default: break;
    }
  } else {
    const int slot9 = code_slot(code) * 9;
    const int nt = ((code >> 28) & 3) + 1;
    uint32_t taps = code & 0xffff;
    float wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll 1
    for (int s = 0; s < nt; ++s) {
      const float ws = s == 0 ? wv[0] : s == 1 ? wv[1] : s == 2 ? wv[2] : wv[3];
      switch (slot9 + (int)(taps & 15)) {
#define PP_TAP_CASE(J, T) \
  case (J)*9 + (T): tap_fma<T>(acc[J], win, ws); break;
#define PP_TAP_SLOT(J) \
  PP_TAP_CASE(J, 0) PP_TAP_CASE(J, 1) PP_TAP_CASE(J, 2) PP_TAP_CASE(J, 3) PP_TAP_CASE(J, 4) \
  PP_TAP_CASE(J, 5) PP_TAP_CASE(J, 6) PP_TAP_CASE(J, 7) PP_TAP_CASE(J, 8)
        PP_TAP_SLOT(0) PP_TAP_SLOT(1) PP_TAP_SLOT(2) PP_TAP_SLOT(3)
        PP_TAP_SLOT(4) PP_TAP_SLOT(5) PP_TAP_SLOT(6) PP_TAP_SLOT(7)
        PP_TAP_SLOT(8) PP_TAP_SLOT(9) PP_TAP_SLOT(10) PP_TAP_SLOT(11)
        PP_TAP_SLOT(12) PP_TAP_SLOT(13) PP_TAP_SLOT(14) PP_TAP_SLOT(15)
#undef PP_TAP_SLOT
#undef PP_TAP_CASE
        default: break;
      }
      taps >>= 4;
    }
  }
}

// Epilogue of one filter slot: bias, +skip, ReLU, 2x2 max pool, store at the
// filter's original channel.  Must be called by all 32 lanes (the pool reads
// the partner row from the next lane).
__device__ __forceinline__ void epilogue_slot(const ConvParams& p, int n, int q, int j, float (&v)[PX], int r,
                                              int cb, int ly) {
  const int jr = q * F + j;
  const int o = __ldg(p.perm + jr);
  const float b = p.bias ? __ldg(p.bias + jr) : 0.f;
  const bool pool = p.flags & PP_POOL2;
  const int Ho = pool ? p.H / 2 : p.H, Wo = pool ? p.W / 2 : p.W;
#pragma unroll
  for (int k = 0; k < PX; ++k) v[k] += b;
  if (p.flags & PP_ADD_SKIP) {
    if (r < p.H) {
      const float* sk = p.skip + (((size_t)n * p.Co + o) * p.H + r) * p.W;
#pragma unroll
      for (int k = 0; k < PX; ++k)
        if (cb + k < p.W) v[k] += __ldg(sk + cb + k);
    }
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

template <int MODE, bool SPLIT>
__global__ void __launch_bounds__(NTHREADS, 2) ppconv_kernel(const ConvParams p) {
  extern __shared__ __align__(16) unsigned char smem[];

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int ly = lane & 15;  // row in tile
  const int lx = lane >> 4;  // column segment (8 pixels)
  const int tile = blockIdx.x;
  const int ty = tile / p.tiles_x, tx = tile - ty * p.tiles_x;
  const int r0 = ty * TH, c0 = tx * TW;
  const int n = SPLIT ? blockIdx.z / p.ksplit : blockIdx.z;
  const int ks = SPLIT ? blockIdx.z - n * p.ksplit : 0;
  const int q = blockIdx.y * NWF + warp;  // filter group of this warp
  const bool active = q < p.G;

  float acc[F][PX];
#pragma unroll
  for (int j = 0; j < F; ++j)
#pragma unroll
    for (int k = 0; k < PX; ++k) acc[j][k] = 0.f;

  const int* cofs = p.cofs + (size_t)(active ? q : 0) * (p.nch + 1);
  const int cbeg = ks * p.cpk;
  const int cend = min(p.nch, cbeg + p.cpk);

  auto issue = [&](int c) {
    unsigned char* st = smem + (c & 1) * STAGE_BYTES;
    stage_input(reinterpret_cast<float*>(st + OFF_IN), p, n, c * p.cc, min(p.cc, p.Ci - c * p.cc), r0, c0);
    if (active) stage_entries(st, p, warp, lane, __ldg(cofs + c), __ldg(cofs + c + 1));
    cp_async_commit();
  };

  if (cbeg < cend) issue(cbeg);
  for (int c = cbeg; c < cend; ++c) {
    if (c + 1 < cend) {
      issue(c + 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (active) {
      const unsigned char* st = smem + (c & 1) * STAGE_BYTES;
      const float* sb = reinterpret_cast<const float*>(st + OFF_IN) + ly * SSTRIDE + lx * PX;
      const float4* sw = reinterpret_cast<const float4*>(st + OFF_WTS) + warp * EMAX;
      const uint32_t* sc = reinterpret_cast<const uint32_t*>(st + OFF_CODE) + warp * EMAX;
      const int ne = __ldg(cofs + c + 1) - __ldg(cofs + c);
      int cur = -1;
      float win[3][PX + 2];
#pragma unroll
      for (int a = 0; a < 3; ++a)
#pragma unroll
        for (int b = 0; b < PX + 2; ++b) win[a][b] = 0.f;
      uint32_t code_n = ne > 0 ? sc[0] : 0u;
      float4 w_n = ne > 0 ? sw[0] : make_float4(0.f, 0.f, 0.f, 0.f);
      for (int e = 0; e < ne; ++e) {
        const uint32_t code = code_n;
        const float4 w = w_n;
        if (e + 1 < ne) {
          code_n = sc[e + 1];
          w_n = sw[e + 1];
        }
        const int ch = code_ch(code);
        if (ch != cur) {
          cur = ch;
          const float* s = sb + ch * SCH;
#pragma unroll
          for (int a = 0; a < 3; ++a) {
            const float4 u = *reinterpret_cast<const float4*>(s + a * SSTRIDE);
            const float4 v = *reinterpret_cast<const float4*>(s + a * SSTRIDE + 4);
            const float2 z = *reinterpret_cast<const float2*>(s + a * SSTRIDE + 8);
            win[a][0] = u.x; win[a][1] = u.y; win[a][2] = u.z; win[a][3] = u.w;
            win[a][4] = v.x; win[a][5] = v.y; win[a][6] = v.z; win[a][7] = v.w;
            win[a][8] = z.x; win[a][9] = z.y;
          }
        }
        dispatch<MODE>(acc, win, code, w);
      }
    }
    __syncthreads();
  }

  const int r = r0 + ly;
  const int cb = c0 + lx * PX;
  if constexpr (!SPLIT) {
    if (!active) return;
#pragma unroll
    for (int j = 0; j < F; ++j) {
      if (q * F + j >= p.Co) break;  // warp-uniform
      epilogue_slot(p, n, q, j, acc[j], r, cb, ly);
    }
  } else {
    // Split over input chunks: publish the partial sums in this CTA's shared
    // memory, then every CTA of the cluster reduces the slots j with
    // j % ksplit == its rank, reading all ranks in order 0..ksplit-1.
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    float* red = reinterpret_cast<float*>(smem);
#pragma unroll
    for (int j = 0; j < F; ++j)
#pragma unroll
      for (int k = 0; k < PX; ++k) red[((warp * F + j) * PX + k) * 32 + lane] = acc[j][k];
    cluster.sync();
    const int rank = (int)cluster.block_rank();
    if (active) {
      for (int j = rank; j < F; j += p.ksplit) {
        if (q * F + j >= p.Co) break;  // warp-uniform
        float v[PX];
#pragma unroll
        for (int k = 0; k < PX; ++k) v[k] = 0.f;
        for (int s2 = 0; s2 < p.ksplit; ++s2) {
          const float* rem = cluster.map_shared_rank(red, s2);
#pragma unroll
          for (int k = 0; k < PX; ++k) v[k] += rem[((warp * F + j) * PX + k) * 32 + lane];
        }
        epilogue_slot(p, n, q, j, v, r, cb, ly);
      }
    }
    cluster.sync();  // keep every CTA's shared memory alive until all reads are done
  }
}

}  // namespace

// ----------------------------------------------------------------------------
// Host side: device layout of a layer and the launch.
// ----------------------------------------------------------------------------

struct pp_layer {
  int Co = 0, Ci = 0;
  int mode = MODE_GENERIC;
  bool tm_ok = false;    // ring-set layer: the tensor-memory kernel can run it
  bool tc_ok = false;    // the tensor-core kernel can run it
  int kernel = 2;        // PP_KERNEL_TMEM / _REGISTER / _TC
  int auto_kernel = 2;
  ppc::TmLayout tm;
  ppc::TcLayout tc;
  ppc::DirectLayout direct;  // built for layers with few input or output channels
  int G = 0, nch = 0;
  int cc = CC;  // input channels per stage
  int64_t nE = 0;
  bool has_bias = false;
  void* dmem = nullptr;  // one allocation holding every array below
  size_t dbytes = 0;
  int* cofs = nullptr;
  uint32_t* code = nullptr;
  float4* wts = nullptr;
  int* perm = nullptr;   // [Co] output channel of reordered filter j (the packer's perm unless re-ordered)
  float* bias = nullptr;
  std::vector<int32_t> pk_perm;     // the packer's filter permutation (host copy)
  std::vector<float> direct_w;      // direct layout's dense weights [Co][Ci][9], original filter order
  std::vector<float> direct_bias;   // and its bias (empty: none)
  pp_packed packed;                 // host copy of the packed layer (tensor-core layers: f16 layout built on demand)
  int precision = PP_PRECISION_TF32X3;
};

struct pp_dense {
  pp_layer base;
};

namespace {

struct Entry {
  int32_t ch;      // input channel
  int32_t slot;    // filter slot in the warp's group
  uint32_t payload;
  float w[4];
};

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Map each pattern of the set to its ring index, or -1 when the set is not a
// subset of the ring set.
bool ring_map(const uint8_t* taps, int P, std::vector<int>& map) {
  map.assign(P, -1);
  for (int p = 0; p < P; ++p) {
    uint16_t m = ppc::tap_mask(taps + 4 * p);
    for (int r = 0; r < 8; ++r) {
      uint8_t rt[4];
      for (int s = 0; s < 4; ++s) rt[s] = (uint8_t)ring_tap(r, s);
      if (ppc::tap_mask(rt) == m) map[p] = r;
    }
    if (map[p] < 0) return false;
  }
  return true;
}

// Build the device layout from per-filter entry lists (filters already in
// reordered order) and upload it.
pp_status build_layer(pp_layer* L, int Co, int Ci, int cc, const std::vector<std::vector<Entry>>& per_filter,
                      const std::vector<int32_t>& perm, const float* bias_reordered, cudaStream_t stream) {
  L->Co = Co;
  L->Ci = Ci;
  L->cc = cc;
  L->G = (Co + F - 1) / F;
  L->nch = (Ci + cc - 1) / cc;
  L->has_bias = bias_reordered != nullptr;
  std::vector<int> cofs((size_t)L->G * (L->nch + 1));
  std::vector<uint32_t> code;
  std::vector<float> wts;
  for (int q = 0; q < L->G; ++q) {
    std::vector<Entry> es;
    for (int j = q * F; j < std::min(Co, (q + 1) * F); ++j)
      for (Entry e : per_filter[j]) {
        e.slot = j - q * F;
        es.push_back(e);
      }
    std::stable_sort(es.begin(), es.end(), [](const Entry& a, const Entry& b) {
      return a.ch != b.ch ? a.ch < b.ch : a.slot < b.slot;
    });
    size_t k = 0;
    for (int c = 0; c <= L->nch; ++c) {
      while (k < es.size() && es[k].ch < c * cc) ++k;
      cofs[(size_t)q * (L->nch + 1) + c] = (int)(code.size() + k);
    }
    for (int c = 0; c < L->nch; ++c)  // the kernel stages at most EMAX entries per warp and chunk
      if (cofs[(size_t)q * (L->nch + 1) + c + 1] - cofs[(size_t)q * (L->nch + 1) + c] > EMAX)
        return PP_ERR_UNSUPPORTED;
    for (const Entry& e : es) {
      code.push_back(e.payload | (uint32_t(e.slot) << 16) | (uint32_t(e.ch % cc) << 20));
      for (int s = 0; s < 4; ++s) wts.push_back(e.w[s]);
    }
  }
  L->nE = (int64_t)code.size();
  if (L->nE > INT32_MAX) return PP_ERR_UNSUPPORTED;
  size_t off_cofs = 0;
  size_t off_code = align_up(off_cofs + cofs.size() * 4, 256);
  size_t off_wts = align_up(off_code + code.size() * 4, 256);
  size_t off_perm = align_up(off_wts + wts.size() * 4, 256);
  size_t off_bias = align_up(off_perm + (size_t)Co * 4, 256);
  size_t total = align_up(off_bias + (size_t)Co * 4, 256);
  std::vector<unsigned char> host(total, 0);
  std::memcpy(host.data() + off_cofs, cofs.data(), cofs.size() * 4);
  if (!code.empty()) std::memcpy(host.data() + off_code, code.data(), code.size() * 4);
  if (!wts.empty()) std::memcpy(host.data() + off_wts, wts.data(), wts.size() * 4);
  std::memcpy(host.data() + off_perm, perm.data(), (size_t)Co * 4);
  if (bias_reordered) std::memcpy(host.data() + off_bias, bias_reordered, (size_t)Co * 4);
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
  unsigned char* b = static_cast<unsigned char*>(d);
  L->dmem = d;
  L->dbytes = total;
  L->cofs = reinterpret_cast<int*>(b + off_cofs);
  L->code = reinterpret_cast<uint32_t*>(b + off_code);
  L->wts = reinterpret_cast<float4*>(b + off_wts);
  L->perm = reinterpret_cast<int*>(b + off_perm);
  L->bias = reinterpret_cast<float*>(b + off_bias);
  return PP_OK;
}

template <int MODE, bool SPLIT>
cudaError_t set_attributes() {
  cudaError_t e = cudaFuncSetAttribute(ppconv_kernel<MODE, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       SMEM_BYTES);
  return e;
}

// Once per process and device: allow the kernels' dynamic shared memory.
ppc::DeviceOnce g_kernels_once;
cudaError_t prepare_kernels() {
  return g_kernels_once.run([](int) {
    cudaError_t e;
    if ((e = set_attributes<MODE_RING8, false>()) != cudaSuccess) return e;
    if ((e = set_attributes<MODE_RING8, true>()) != cudaSuccess) return e;
    if ((e = set_attributes<MODE_GENERIC, false>()) != cudaSuccess) return e;
    return set_attributes<MODE_GENERIC, true>();
  });
}

// Number of CTAs sharing one output tile: split the input chunks over a
// cluster when the grid alone would leave SMs idle (two CTAs fit per SM).
int choose_split(int64_t base_ctas, int nch) {
  const int sms = ppc::device_sms();
  int ks = 1;
  while (ks < MAX_SPLIT && ks * 2 <= nch && base_ctas * ks < 2 * sms) ks *= 2;
  return ks;
}

pp_status launch(const pp_layer* L, const float* x, float* y, const float* skip, int N, int H, int W, int flags,
                 cudaStream_t stream) {
  if (!L || !x || !y || N < 1 || H < 1 || W < 1) return PP_ERR_INVALID_ARG;
  if (flags & ~(PP_ADD_SKIP | PP_RELU | PP_POOL2)) return PP_ERR_INVALID_ARG;
  if ((flags & PP_ADD_SKIP) && !skip) return PP_ERR_INVALID_ARG;
  if ((flags & PP_POOL2) && ((H & 1) || (W & 1))) return PP_ERR_UNSUPPORTED;
  if (((uintptr_t)y & 15) || ((uintptr_t)x & 3)) return PP_ERR_INVALID_ARG;
  if (L->kernel == PP_KERNEL_DIRECT) return ppc::direct_launch(L->direct, x, y, skip, N, H, W, flags, stream);
  if (L->kernel == PP_KERNEL_TMEM || L->kernel == PP_KERNEL_TC || L->kernel == PP_KERNEL_TC_FLAT) {
    ppc::LayerMeta M;
    M.Co = L->Co;
    M.Ci = L->Ci;
    M.perm = L->perm;
    M.bias = L->has_bias ? L->bias : nullptr;
    if (L->kernel == PP_KERNEL_TC_FLAT) {
      const pp_status st = ppc::tcf_launch(L->tc, M, x, y, skip, N, H, W, flags, stream);
      if (st != PP_ERR_UNSUPPORTED) return st;
      // maps wider than the flat kernel's tiles run the row-tiled tensor-core kernel
    }
    if (L->kernel == PP_KERNEL_TC || L->kernel == PP_KERNEL_TC_FLAT) {
      const pp_status st = ppc::tc_launch(L->tc, M, x, y, skip, N, H, W, flags, stream);
      if (st != PP_ERR_UNSUPPORTED) return st;
      // shapes beyond the tensor-core kernel's 32-bit offsets run on an FMA kernel
      if (L->tm_ok) return ppc::tm_launch(L->tm, M, x, y, skip, N, H, W, flags, stream);
    } else {
      return ppc::tm_launch(L->tm, M, x, y, skip, N, H, W, flags, stream);
    }
  }
  const int tiles_y = (H + TH - 1) / TH, tiles_x = (W + TW - 1) / TW;
  if ((int64_t)tiles_y * tiles_x > INT32_MAX) return PP_ERR_UNSUPPORTED;
  ConvParams p;
  p.x = x;
  p.y = y;
  p.skip = (flags & PP_ADD_SKIP) ? skip : nullptr;
  p.cofs = L->cofs;
  p.code = L->code;
  p.wts = L->wts;
  p.perm = L->perm;
  p.bias = L->has_bias ? L->bias : nullptr;
  p.N = N;
  p.Ci = L->Ci;
  p.Co = L->Co;
  p.H = H;
  p.W = W;
  p.nch = L->nch;
  p.cc = L->cc;
  p.G = L->G;
  p.tiles_x = tiles_x;
  p.flags = flags;
  const int cgroups = (L->G + NWF - 1) / NWF;
  const int64_t base = (int64_t)tiles_y * tiles_x * cgroups * N;
  if (prepare_kernels() != cudaSuccess || ppc::device_sms() <= 0) return PP_ERR_CUDA;
  const int ks = choose_split(base, L->nch);
  p.ksplit = ks;
  p.cpk = (L->nch + ks - 1) / ks;
  if ((int64_t)N * ks > 65535 || cgroups > 65535) return PP_ERR_UNSUPPORTED;
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
    e = L->mode == MODE_RING8 ? cudaLaunchKernelEx(&cfg, ppconv_kernel<MODE_RING8, true>, p)
                              : cudaLaunchKernelEx(&cfg, ppconv_kernel<MODE_GENERIC, true>, p);
  } else {
    e = L->mode == MODE_RING8 ? cudaLaunchKernelEx(&cfg, ppconv_kernel<MODE_RING8, false>, p)
                              : cudaLaunchKernelEx(&cfg, ppconv_kernel<MODE_GENERIC, false>, p);
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  return PP_OK;
}

}  // namespace

namespace ppc {

int device_sms() {
  static DeviceOnce once;
  static int sms[DeviceOnce::kMaxDevices];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= DeviceOnce::kMaxDevices) return 0;
  if (once.run([](int d) { return cudaDeviceGetAttribute(&sms[d], cudaDevAttrMultiProcessorCount, d); }) !=
      cudaSuccess)
    return 0;
  return sms[dev];
}

}  // namespace ppc

extern "C" pp_status pp_layer_create(const pp_packed* pk, const float* bias, void* stream, pp_layer** out) {
  if (!pk || !out) return PP_ERR_INVALID_ARG;
  if (prepare_kernels() != cudaSuccess) return PP_ERR_CUDA;  // outside any stream capture
  pp_layer* L = new (std::nothrow) pp_layer;
  if (!L) return PP_ERR_OOM;
  std::vector<int> rmap;
  L->mode = ring_map(pk->taps.data(), pk->P, rmap) ? MODE_RING8 : MODE_GENERIC;
  std::vector<std::vector<Entry>> per_filter(pk->Co);
  std::vector<float> bias_r;
  if (bias) bias_r.resize(pk->Co);
  for (int j = 0; j < pk->Co; ++j) {
    if (bias) bias_r[j] = bias[pk->perm[j]];
    for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e) {
      Entry en;
      en.ch = pk->kidx[e];
      en.slot = 0;
      const int p = pk->kpat[e];
      if (L->mode == MODE_RING8) {
        // Reorder the 4 weights from the pattern's ascending taps to the ring
        // pattern's ascending taps (same set, so the same order).
        en.payload = (uint32_t)rmap[p];
      } else {
        const uint8_t* t = &pk->taps[4 * p];
        en.payload = t[0] | (t[1] << 4) | (t[2] << 8) | (t[3] << 12) | (3u << 28);
      }
      for (int s = 0; s < 4; ++s) en.w[s] = pk->kw[(size_t)e * 4 + s];
      per_filter[j].push_back(en);
    }
  }
  pp_status st = build_layer(L, pk->Co, pk->Ci, CC, per_filter, pk->perm, bias ? bias_r.data() : nullptr,
                             (cudaStream_t)stream);
  if (st == PP_OK && L->mode == MODE_RING8) {
    st = ppc::tm_prepare();
    if (st == PP_OK) st = ppc::tm_build(&L->tm, pk, rmap, (cudaStream_t)stream);
    L->tm_ok = st == PP_OK;
  }
  if (st == PP_OK) {
    // channels are padded to the chunk width (zero weights, zero-filled input
    // boxes), so a layer with fewer than 8 input channels has one ragged chunk
    st = ppc::tc_prepare();
    if (st == PP_OK) st = ppc::tc_build(&L->tc, pk, (cudaStream_t)stream);
    L->tc_ok = st == PP_OK;
    if (L->tc_ok) L->packed = *pk;
  }
  if (st == PP_OK && ppc::direct_applicable(pk->Co, pk->Ci)) {
    // dense [Co][Ci][9] in the original filter order, zeros where pruned
    std::vector<float> wd((size_t)pk->Co * pk->Ci * 9, 0.f);
    for (int j = 0; j < pk->Co; ++j)
      for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e) {
        const uint8_t* t = &pk->taps[4 * pk->kpat[e]];
        for (int s = 0; s < 4; ++s)
          wd[((size_t)pk->perm[j] * pk->Ci + pk->kidx[e]) * 9 + t[s]] = pk->kw[(size_t)e * 4 + s];
      }
    st = ppc::direct_build(&L->direct, wd.data(), bias, pk->Co, pk->Ci, (cudaStream_t)stream);
    L->direct_w.swap(wd);
    if (bias) L->direct_bias.assign(bias, bias + pk->Co);
  }
  if (st != PP_OK) {
    pp_layer_destroy(L);
    return st;
  }
  L->pk_perm = pk->perm;
  // Kernel choice by estimated SM cycles per pixel: the tensor cores run the
  // dense 9-tap contraction (filters padded to 128, channels to 8) three times
  // at ~1800 multiply-adds per cycle; the FMA kernels run only the kept taps
  // at a quarter of the 128 FMA lanes (what they reach on these layers).
  const double nk = (double)pk->kidx.size();
  const double tc_cycles = 27.0 * (double)((pk->Co + 127) / 128 * 128) * (double)((pk->Ci + 7) / 8 * 8) / 1800.0;
  const double fma_cycles = 4.0 * nk / 32.0;
  L->auto_kernel = (L->tc_ok && tc_cycles < fma_cycles) ? (L->tc.FB == 128 ? PP_KERNEL_TC_FLAT : PP_KERNEL_TC)
                                                         : (L->tm_ok ? PP_KERNEL_TMEM : PP_KERNEL_REGISTER);
  // layers with a handful of input channels (a network's first layer) run the
  // direct kernel: the others cannot fill their tiles
  if (L->direct.w && pk->Ci <= 4) L->auto_kernel = PP_KERNEL_DIRECT;
  L->kernel = L->auto_kernel;
  *out = L;
  return PP_OK;
}

extern "C" pp_status pp_layer_set_output_order(pp_layer* L, const int32_t* order, void* stream_) {
  if (!L) return PP_ERR_INVALID_ARG;
  const int Co = L->Co, Ci = L->Ci;
  std::vector<int32_t> ord(Co);
  std::vector<uint8_t> seen(Co, 0);
  for (int o = 0; o < Co; ++o) {
    ord[o] = order ? order[o] : o;
    if (ord[o] < 0 || ord[o] >= Co || seen[ord[o]]) return PP_ERR_INVALID_ARG;
    seen[ord[o]] = 1;
  }
  cudaStream_t stream = (cudaStream_t)stream_;
  // the direct kernel stores row o of its dense weights at channel o: its layout is rebuilt with rows
  // moved, first, so that a failure leaves the layer as it was
  ppc::DirectLayout D;
  if (L->direct.w) {
    std::vector<float> w((size_t)Co * Ci * 9), b(L->direct_bias.empty() ? 0 : Co);
    for (int o = 0; o < Co; ++o) {
      std::memcpy(&w[(size_t)ord[o] * Ci * 9], &L->direct_w[(size_t)o * Ci * 9], (size_t)Ci * 9 * sizeof(float));
      if (!b.empty()) b[ord[o]] = L->direct_bias[o];
    }
    const pp_status st = ppc::direct_build(&D, w.data(), b.empty() ? nullptr : b.data(), Co, Ci, stream);
    if (st != PP_OK) return st;
  }
  // every other kernel stores reordered filter j at channel perm[j]
  std::vector<int32_t> store(Co);
  for (int j = 0; j < Co; ++j) store[j] = ord[L->pk_perm[j]];
  if (cudaMemcpyAsync(L->perm, store.data(), (size_t)Co * 4, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    cudaGetLastError();
    ppc::direct_free(&D);
    return PP_ERR_CUDA;
  }
  if (L->direct.w) {
    ppc::direct_free(&L->direct);
    L->direct = D;
  }
  return PP_OK;
}

extern "C" pp_status pp_layer_set_precision(pp_layer* L, int precision, float input_bound, void* stream) {
  if (!L) return PP_ERR_INVALID_ARG;
  if (precision == PP_PRECISION_TF32X3) {
    L->tc.f16 = false;
    L->precision = precision;
    return PP_OK;
  }
  if (precision != PP_PRECISION_F16X3 || std::isnan(input_bound)) return PP_ERR_INVALID_ARG;
  if (!L->tc_ok) return PP_ERR_UNSUPPORTED;
  const pp_status st = ppc::tc_build16(&L->tc, &L->packed, input_bound, (cudaStream_t)stream);
  if (st != PP_OK) return st;
  L->tc.f16 = true;
  L->precision = precision;
  return PP_OK;
}

extern "C" pp_status pp_layer_precision(const pp_layer* L, int* precision, float* input_scale) {
  if (!L) return PP_ERR_INVALID_ARG;
  if (precision) *precision = L->precision;
  if (input_scale) *input_scale = L->precision == PP_PRECISION_F16X3 ? L->tc.xscale : 1.f;
  return PP_OK;
}

extern "C" pp_status pp_layer_set_kernel(pp_layer* L, int kernel) {
  if (!L) return PP_ERR_INVALID_ARG;
  switch (kernel) {
    case PP_KERNEL_AUTO: L->kernel = L->auto_kernel; return PP_OK;
    case PP_KERNEL_TMEM:
      if (!L->tm_ok) return PP_ERR_UNSUPPORTED;
      L->kernel = kernel;
      return PP_OK;
    case PP_KERNEL_TC:
      if (!L->tc_ok) return PP_ERR_UNSUPPORTED;
      L->kernel = kernel;
      return PP_OK;
    case PP_KERNEL_TC_FLAT:
      if (!L->tc_ok || L->tc.FB != 128) return PP_ERR_UNSUPPORTED;
      L->kernel = kernel;
      return PP_OK;
    case PP_KERNEL_REGISTER: L->kernel = kernel; return PP_OK;
    case PP_KERNEL_DIRECT:
      if (!L->direct.w) return PP_ERR_UNSUPPORTED;
      L->kernel = kernel;
      return PP_OK;
    default: return PP_ERR_INVALID_ARG;
  }
}

extern "C" pp_status pp_layer_kernel(const pp_layer* L, int* kernel) {
  if (!L || !kernel) return PP_ERR_INVALID_ARG;
  *kernel = L->kernel;
  return PP_OK;
}

extern "C" pp_status pp_layer_autotune(pp_layer* L, int N, int H, int W, int flags, void* stream_) {
  if (!L || N < 1 || H < 1 || W < 1) return PP_ERR_INVALID_ARG;
  if (flags & ~(PP_ADD_SKIP | PP_RELU | PP_POOL2)) return PP_ERR_INVALID_ARG;
  if ((flags & PP_POOL2) && ((H & 1) || (W & 1))) return PP_ERR_UNSUPPORTED;
  cudaStream_t stream = (cudaStream_t)stream_;
  // Candidates: (kernel, flat-kernel rows per tile, split); the flat kernel is
  // tried at the six best geometries of its cost model (CTA pairs included).
  struct Cand {
    int kernel, R, S;
  };
  std::vector<Cand> cand;
  if (L->tc_ok) cand.push_back({PP_KERNEL_TC, 0, 0});
  if (L->tc_ok && L->tc.FB == 128) {
    int R[6], S[6];
    const int n = ppc::tcf_plan(L->tc, N, H, W, flags, R, S, 6);
    for (int k = 0; k < n; ++k) cand.push_back({PP_KERNEL_TC_FLAT, R[k], S[k]});
  }
  if (L->tm_ok) cand.push_back({PP_KERNEL_TMEM, 0, 0});
  if (L->direct.w) cand.push_back({PP_KERNEL_DIRECT, 0, 0});
  if (cand.empty()) cand.push_back({PP_KERNEL_REGISTER, 0, 0});
  if (cand.size() == 1) {
    L->kernel = cand[0].kernel;
    return PP_OK;
  }
  const size_t in_elems = (size_t)N * L->Ci * H * W, out_elems = (size_t)N * L->Co * H * W;
  float *x = nullptr, *y = nullptr, *sk = nullptr;
  if (cudaMalloc(&x, in_elems * 4) != cudaSuccess || cudaMalloc(&y, out_elems * 4) != cudaSuccess ||
      ((flags & PP_ADD_SKIP) && cudaMalloc(&sk, out_elems * 4) != cudaSuccess)) {
    cudaGetLastError();
    cudaFree(x);
    cudaFree(y);
    return PP_ERR_OOM;
  }
  pp_status st = PP_OK;
  if (cudaMemsetAsync(x, 0, in_elems * 4, stream) != cudaSuccess ||
      (sk && cudaMemsetAsync(sk, 0, out_elems * 4, stream) != cudaSuccess))
    st = PP_ERR_CUDA;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (st == PP_OK && (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess)) st = PP_ERR_CUDA;
  const int saved = L->kernel;
  Cand best = {saved, 0, 0};
  float best_ms = 1e30f, tc_ms = 1e30f;
  for (const Cand& c : cand) {
    if (st != PP_OK) break;
    L->kernel = c.kernel;
    if (c.kernel == PP_KERNEL_TC_FLAT) ppc::tcf_pin(L->tc, N, H, W, flags, c.R, c.S);
    for (int w = 0; w < 2 && st == PP_OK; ++w) st = launch(L, x, y, sk, N, H, W, flags, stream);
    if (st != PP_OK) break;
    if (cudaEventRecord(e0, stream) != cudaSuccess) {
      st = PP_ERR_CUDA;
      break;
    }
    for (int r = 0; r < 5 && st == PP_OK; ++r) st = launch(L, x, y, sk, N, H, W, flags, stream);
    float ms = 0.f;
    if (st != PP_OK || cudaEventRecord(e1, stream) != cudaSuccess || cudaEventSynchronize(e1) != cudaSuccess ||
        cudaEventElapsedTime(&ms, e0, e1) != cudaSuccess) {
      st = st != PP_OK ? st : PP_ERR_CUDA;
      break;
    }
    if (c.kernel == PP_KERNEL_TC) tc_ms = ms;
    if (ms < best_ms) {
      best_ms = ms;
      best = c;
    }
  }
  // The candidates are timed alone.  In a network, a row-tiled layer that follows
  // a flat-kernel layer measured up to ~14 us slower than after a row-tiled one
  // (the style trunk's 128 x 128 convs, both arithmetics), so the flat kernel
  // replaces the row-tiled one only when it is more than 10 % faster alone.
  if (best.kernel == PP_KERNEL_TC_FLAT && tc_ms <= 1.1f * best_ms) best = {PP_KERNEL_TC, 0, 0};
  L->kernel = st == PP_OK ? best.kernel : saved;
  // the flat kernel keeps the geometry that won for this shape (none if it lost)
  if (L->tc_ok && L->tc.FB == 128)
    ppc::tcf_pin(L->tc, N, H, W, flags, st == PP_OK && best.kernel == PP_KERNEL_TC_FLAT ? best.R : 0, best.S);
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  cudaStreamSynchronize(stream);
  cudaFree(x);
  cudaFree(y);
  cudaFree(sk);
  return st;
}

extern "C" pp_status pp_layer_flat_geometry(const pp_layer* L, int N, int H, int W, int flags, int* R, int* S) {
  if (!L || !R || !S || N < 1 || H < 1 || W < 1) return PP_ERR_INVALID_ARG;
  *R = 0;
  *S = 0;
  if (L->tc_ok && L->tc.FB == 128) ppc::tcf_pinned(L->tc, N, H, W, flags, R, S);
  return PP_OK;
}

extern "C" pp_status pp_layer_pin_flat_geometry(pp_layer* L, int N, int H, int W, int flags, int R, int S) {
  if (!L || N < 1 || H < 1 || W < 1 || R < 0) return PP_ERR_INVALID_ARG;
  if (flags & ~(PP_ADD_SKIP | PP_RELU | PP_POOL2)) return PP_ERR_INVALID_ARG;
  if (!L->tc_ok || L->tc.FB != 128) return PP_ERR_UNSUPPORTED;
  if (R > 0 && !ppc::tcf_can_run(L->tc, N, H, W, flags, R, S)) return PP_ERR_UNSUPPORTED;
  ppc::tcf_pin(L->tc, N, H, W, flags, R, S);
  return PP_OK;
}

extern "C" pp_status pp_layer_device_status(const pp_layer* L, int* device_error) {
  if (!L || !device_error) return PP_ERR_INVALID_ARG;
  *device_error = 0;
  if (!L->tc_ok) return PP_OK;
  pp_status st = ppc::tc_status(L->tc, device_error);
  if (st == PP_OK && *device_error && cudaMemset(L->tc.status, 0, sizeof(int)) != cudaSuccess) return PP_ERR_CUDA;
  return st;
}

extern "C" pp_status pp_layer_info(const pp_layer* L, int* Co, int* Ci, int64_t* device_bytes) {
  if (!L) return PP_ERR_INVALID_ARG;
  if (Co) *Co = L->Co;
  if (Ci) *Ci = L->Ci;
  if (device_bytes)
    *device_bytes = (int64_t)(L->dbytes + L->tm.dbytes + L->tc.dbytes + L->tc.dbytes16 +
                              (L->direct.w ? ((size_t)L->Co * L->Ci * 9 + (L->direct.bias ? L->Co : 0)) * 4 : 0));
  return PP_OK;
}

extern "C" pp_status pp_conv_forward(const pp_layer* L, const float* x, float* y, const float* skip, int N, int H,
                                     int W, int flags, void* stream) {
  return launch(L, x, y, skip, N, H, W, flags, (cudaStream_t)stream);
}

// The flat tensor-core kernel, with no device memory allocated by the call
// (see the declaration).
extern "C" pp_status pp_conv_forward_noalloc(const pp_layer* L, const float* x, float* y, const float* skip, int N,
                                             int H, int W, int flags, void* stream) {
  if (!L || !x || !y || N < 1 || H < 1 || W < 1) return PP_ERR_INVALID_ARG;
  if (flags & ~(PP_ADD_SKIP | PP_RELU | PP_POOL2)) return PP_ERR_INVALID_ARG;
  if ((flags & PP_ADD_SKIP) && !skip) return PP_ERR_INVALID_ARG;
  if ((flags & PP_POOL2) && ((H & 1) || (W & 1))) return PP_ERR_UNSUPPORTED;
  if (((uintptr_t)y & 15) || ((uintptr_t)x & 3)) return PP_ERR_INVALID_ARG;
  if (!L->tc_ok) return PP_ERR_UNSUPPORTED;
  ppc::LayerMeta M;
  M.Co = L->Co;
  M.Ci = L->Ci;
  M.perm = L->perm;
  M.bias = L->has_bias ? L->bias : nullptr;
  return ppc::tcf_launch(L->tc, M, x, y, skip, N, H, W, flags, (cudaStream_t)stream);
}

extern "C" void pp_layer_destroy(pp_layer* L) {
  if (!L) return;
  if (L->dmem) cudaFree(L->dmem);
  if (L->tm.dmem) cudaFree(L->tm.dmem);
  ppc::tc_free(&L->tc);
  ppc::direct_free(&L->direct);
  delete L;
}

extern "C" pp_status pp_dense_create(const float* w, const float* bias, int Co, int Ci, void* stream,
                                     pp_dense** out) {
  if (!w || !out || Co < 1 || Ci < 1) return PP_ERR_INVALID_ARG;
  if ((int64_t)Co * Ci > (int64_t(1) << 26)) return PP_ERR_UNSUPPORTED;
  if (prepare_kernels() != cudaSuccess) return PP_ERR_CUDA;
  pp_dense* D = new (std::nothrow) pp_dense;
  if (!D) return PP_ERR_OOM;
  D->base.mode = MODE_GENERIC;
  // A dense kernel is three entries of the generic path: taps 0-3, 4-7 and 8.
  std::vector<std::vector<Entry>> per_filter(Co);
  std::vector<int32_t> perm(Co);
  for (int o = 0; o < Co; ++o) {
    perm[o] = o;
    for (int i = 0; i < Ci; ++i) {
      const float* k = w + ((size_t)o * Ci + i) * 9;
      for (int part = 0; part < 3; ++part) {
        Entry en;
        en.ch = i;
        en.slot = 0;
        const int t0 = part * 4;
        const int nt = part < 2 ? 4 : 1;
        en.payload = 0;
        for (int s = 0; s < nt; ++s) en.payload |= uint32_t(t0 + s) << (4 * s);
        en.payload |= uint32_t(nt - 1) << 28;
        for (int s = 0; s < 4; ++s) en.w[s] = s < nt ? k[t0 + s] : 0.f;
        per_filter[o].push_back(en);
      }
    }
  }
  // three entries per kernel: 5 channels per stage keep a warp's stage at <= EMAX entries
  pp_status st = build_layer(&D->base, Co, Ci, 5, per_filter, perm, bias, (cudaStream_t)stream);
  if (st == PP_OK && ppc::direct_applicable(Co, Ci)) {
    st = ppc::direct_build(&D->base.direct, w, bias, Co, Ci, (cudaStream_t)stream);
    if (st == PP_OK) D->base.kernel = D->base.auto_kernel = PP_KERNEL_DIRECT;
  }
  if (st != PP_OK) {
    pp_dense_destroy(D);
    return st;
  }
  *out = D;
  return PP_OK;
}

extern "C" pp_status pp_dense_forward(const pp_dense* D, const float* x, float* y, const float* skip, int N, int H,
                                      int W, int flags, void* stream) {
  if (!D) return PP_ERR_INVALID_ARG;
  return launch(&D->base, x, y, skip, N, H, W, flags, (cudaStream_t)stream);
}

extern "C" pp_status pp_dense_info(const pp_dense* D, int* Co, int* Ci) {
  if (!D) return PP_ERR_INVALID_ARG;
  if (Co) *Co = D->base.Co;
  if (Ci) *Ci = D->base.Ci;
  return PP_OK;
}

extern "C" void pp_dense_destroy(pp_dense* D) {
  if (!D) return;
  if (D->base.dmem) cudaFree(D->base.dmem);
  ppc::direct_free(&D->base.direct);
  delete D;
}
