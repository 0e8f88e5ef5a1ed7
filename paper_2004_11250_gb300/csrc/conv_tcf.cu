// Pattern-pruned 3x3 convolution on the tensor cores, "flat" variant for maps
// at most 128 pixels wide, with the input-channel loop optionally split over a
// thread-block cluster.
//
// The layer is the same dense contraction as in conv_tc.cu (pruned taps and
// kernels written as zeros, Section 2; 3xTF32 split for fp32 accuracy), with a
// different mapping of the output tile onto one MMA:
//   * M = 128 consecutive reordered filters (TMEM lanes);
//   * N = the pixels of R whole output rows, flattened.  The input tile for a
//     chunk of 8 channels is staged as R + 2 rows of BCOLS >= W + 2 pixels (zero
//     halo, BCOLS a multiple of 8), one 16-byte K-major row per pixel.  Output
//     pixel (r, c) of the tile is MMA column j = r * BCOLS + c, and its tap
//     (dy, dx) reads staged pixel j + dy * BCOLS + dx, so a tap is the whole
//     staged tile with the operand start moved by dy * BCOLS + dx pixels: one
//     MMA of N = R * BCOLS (rounded up to 16, at most 256) per tap and pass.
//     Columns c >= W of each row are computed and discarded.
// Against one MMA per output row (N = tile width) this makes narrow maps
// (14 ... 128 pixels) run full-width MMAs and halves the shared-memory operand
// traffic per multiply-add.
//
// Split: when the layer has fewer output tiles than SMs, S CTAs of a cluster
// share a tile, each summing a contiguous range of the channel chunks.  Each
// copies its fp32 partial tile from TMEM into its own shared memory, a cluster
// barrier orders those writes before the reads, and each CTA then finishes 1/S
// of the tile's filters: it reads the S partials of those filters through
// distributed shared memory, adds them in rank order (deterministic), then
// bias, skip, ReLU, pool, and stores y.  No global workspace is used.
//
// CTA pairs (geometries S | PP_FLAT_PAIRED): the two filter blocks of a tile
// run on two CTAs of a cluster as one M = 256 MMA (cta_group::2), each CTA
// holding its own block's weights and staging half of the tile's columns; the
// even CTA issues every MMA (see the kernel's PAIR parameter).
//
// Precision: 3xTF32 (as conv_tc.cu), or, for layers set to PP_PRECISION_F16X3,
// an fp16 split (F16 instantiations): each operand v is held as hi = f16(v) and
// lo = f16((v - hi) * 2^11), the weights scaled per filter and the input per
// layer by powers of two so that both stay in fp16's normal range; a chunk is
// 16 channels (the K of kind::f16) and each tap runs w_hi x_hi into one
// accumulator and w_lo x_hi + w_hi x_lo into a second one (TMEM columns 128 ..
// 255 of the buffer for tiles of at most 128 columns; for wider tiles, which are
// single-buffered, the other buffer), combined in the epilogue as (acc1 + 2^-11 acc2) times the
// filter's inverse scale.  The dropped lo x lo term and the rounding of the lo
// parts are each below 2^-22 of |w * x|.  Inputs that overflow fp16 after
// scaling (|x s| >= 65520) or are not finite are flagged by the loaders in the
// device status word.
//
// Roles (one CTA per SM): warps 0-7 stage the operands (thread 0 also issues
// the input-box copies), warp 8 allocates TMEM and one of its threads issues
// the MMAs, waiting once per chunk (the stage's full barrier counts the loaders
// and the weight copies), warps 9-16 are the epilogue (two per TMEM lane
// quadrant), and in the cluster-split and f16 instantiations warp 17 copies
// the weights, three groups of 3 taps per chunk into a ring of group slots,
// each slot refilled as soon as its MMAs complete.  The unsplit tf32
// instantiation has no warp 17: loader thread 0 copies each chunk's weights
// whole once its stage is free.  Without a split the CTA is persistent
// over tiles with two TMEM accumulator buffers, so a tile's epilogue overlaps
// the next tile's MMAs.  Every mbarrier wait is bounded; a timeout sets the
// layer's device status word and the CTA skips the rest of its work (every
// thread still reaches the cluster barrier).
#include <cooperative_groups.h>
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>

#include "internal.h"
#include "tc_ptx.cuh"

namespace {

using namespace ppc_ptx;

constexpr int KC = 8;                 // input channels per chunk (MMA K for tf32; 16 for f16)
constexpr int ACC2 = 128;             // f16, double-buffered: column offset of the second accumulator in a buffer
constexpr int NTAP = 9;
constexpr int FB = 128;               // filters per block (MMA M)
constexpr int NMAX = 256;             // TMEM columns of one accumulator buffer
constexpr int NLOAD = 256;            // loader threads (warps 0-7)
constexpr int MMA_WARP = 8;
constexpr int EPI_WARP0 = 9;          // warps 9-16
constexpr int NEPI = 256;
constexpr int WPROD_WARP = 17;        // the weight producer (weight-ring instantiations)
constexpr int NTHREADS = 576;         // with the producer warp; 544 without
constexpr int WMAX = 128;             // widest map handled
constexpr int W_TILE = FB * KC * 4;   // one tap, hi or lo: 128 x 8 fp32 (or 128 x 16 f16)
constexpr int TAP_BYTES = 2 * W_TILE;          // one tap's hi and lo rows
constexpr int W_BYTES = NTAP * TAP_BYTES;        // the weights of one chunk
constexpr int NGRP = 3;                          // weight groups per chunk (3 taps each)
constexpr int GRP_BYTES = W_BYTES / NGRP;        // a slot of the weight ring
constexpr int WSL_MAX = 7;                       // slots of the weight ring (7, else 6 when short of space)
constexpr int PIX_MAX = 544;          // staged pixels per K half, padding included
constexpr int IN_MAX = 2 * PIX_MAX * 16;  // largest hi (or lo) operand of one chunk
constexpr int SMEM_ALLOC = 231424;    // dynamic shared memory (static use stays below 1 KB)
constexpr int SMEM_USE = SMEM_ALLOC - 1024;  // after aligning the base to 1024
constexpr int ITEMS_MAX = (2 * PIX_MAX + NLOAD - 1) / NLOAD;  // (K half, pixel) items per loader thread
constexpr long WAIT_LIMIT = PP_WAIT_POLLS;  // mbarrier polls before a wait gives up
constexpr int MAX_SPLIT = 16;
static_assert(2 * (W_BYTES + 2 * IN_MAX) <= SMEM_USE, "shared memory plan");
static_assert(GRP_BYTES % 1024 == 0, "weight-ring slots keep 1024-byte alignment");
static_assert(FB * NMAX * 4 <= SMEM_USE, "split reduction buffer");

// Weights by the producer warp into the ring of 3-tap groups: the cluster-split
// and f16 instantiations.  The unsplit tf32 one (persistent over several tiles)
// measured faster with each chunk's weights copied whole by the loaders' thread
// 0 into two fixed chunk slots (the ring's first 6 group slots) once the stage
// is free, and without the producer warp (an 18th warp, even idle, slowed it).
template <bool SPLIT, bool F16>
__host__ __device__ constexpr bool weight_ring() { return SPLIT || F16; }
template <bool SPLIT, bool F16>
__host__ __device__ constexpr int flat_threads() { return weight_ring<SPLIT, F16>() ? NTHREADS : NTHREADS - 32; }

struct FlatParams {
  const float* rscale;      // f16: per reordered filter, 1 / (weight scale x input scale)
  float xscale;             // f16: power of two applied to x before the split
  const float* x;
  float* y;
  const float* skip;
  const unsigned char* wt;  // [nfb][nch][9][2][128 x 8] canonical tiles
  const int* perm;
  const float* bias;
  int* status;
  int N, Ci, Co, H, W;
  int nch, nfb, flags, use_tma;
  int bcols, R, ncols, npix, npixa, raw_w, raw_bytes;
  int wsl;                  // slots of the weight ring (6 or 7 groups of 3 taps) at the start of shared memory
  int xoff, xstage, lo_off; // input operand stage s at xoff + s * xstage: hi, then lo at lo_off
  int sep, raw_off, raw_slot;  // input boxes in a ring of their own: sep (2 or 1) slots at raw_off; 0 = none
                               // (slot of chunk g: g & (sep - 1))
  int plane;                // box over x viewed as [N][Ci][H * W]: the staged rows packed, raw_w = box width
  int tiles_y, ntiles, split;
  uint32_t idesc;
  // TMEM accumulator buffers (2: a tile's epilogue overlaps the next tile's MMAs;
  // 1: f16 tiles wider than ACC2 columns, whose second accumulator takes the
  // other buffer's columns) and the f16 second accumulator's column offset
  int nbuf, acc2;
};

struct Tile {
  int n, r0, fb;
};
__device__ __forceinline__ Tile tile_of(const FlatParams& p, int t) {
  Tile T;
  T.fb = t % p.nfb;
  t /= p.nfb;
  T.r0 = (t % p.tiles_y) * p.R;
  T.n = t / p.tiles_y;
  return T;
}

// Second phase of a cluster split: this CTA owns filters [m0, m0 + nm) of the
// tile and sums, for each of them, the S partial tiles of the cluster (read in
// rank order from each CTA's shared memory), then applies the epilogue.  Work
// items are 4 adjacent accumulator columns of one filter (pooled: 2 rows x 4
// columns, i.e. 2 pooled outputs), spread over all threads of the CTA; each
// item issues its S 16-byte loads before it sums them.
// The S partials of a tile are in cluster CTAs rofs, rofs + rstride, ... (rstride
// 2 with CTA pairs: the even and the odd CTAs hold different filter blocks).
template <int S>
__device__ __forceinline__ void split_reduce(const FlatParams& p, const Tile& T, int m0, int nm, float* part,
                                             const int* o_s, const float* b_s, int tid, int rstride, int rofs) {
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  const float* src[S];
#pragma unroll
  for (int s = 0; s < S; ++s) src[s] = cl.map_shared_rank(part, s * rstride + rofs);
  const int pst = p.ncols + 4;
  const bool relu = p.flags & PP_RELU;
  const float* skip = (p.flags & PP_ADD_SKIP) ? p.skip : nullptr;
  auto sum = [&](int off) -> float4 {
    float4 v[S];
#pragma unroll
    for (int s = 0; s < S; ++s) v[s] = *reinterpret_cast<const float4*>(src[s] + off);
    float4 a = v[0];
#pragma unroll
    for (int s = 1; s < S; ++s) {
      a.x += v[s].x;
      a.y += v[s].y;
      a.z += v[s].z;
      a.w += v[s].w;
    }
    return a;
  };
  if (!(p.flags & PP_POOL2)) {
    const int qw = (p.W + 3) >> 2, ipf = p.R * qw;
    for (int it = tid; it < nm * ipf; it += NTHREADS) {
      const int ml = it / ipf, rest = it - ml * ipf;
      const int ro = rest / qw, cx = (rest - ro * qw) * 4;
      const int row = T.r0 + ro, o = o_s[ml];
      if (row >= p.H || o < 0) continue;
      const float4 a = sum((m0 + ml) * pst + ro * p.bcols + cx);
      const size_t yoff = (((size_t)T.n * p.Co + o) * p.H + row) * p.W + cx;
      float v[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        v[k] += b_s[ml];
        if (skip && cx + k < p.W) v[k] += __ldg(skip + yoff + k);
        if (relu) v[k] = fmaxf(v[k], 0.f);
      }
      float* y = p.y + yoff;
      if ((p.W & 3) == 0) {
        *reinterpret_cast<float4*>(y) = make_float4(v[0], v[1], v[2], v[3]);
      } else if ((p.W & 1) == 0) {
        *reinterpret_cast<float2*>(y) = make_float2(v[0], v[1]);
        if (cx + 2 < p.W) *reinterpret_cast<float2*>(y + 2) = make_float2(v[2], v[3]);
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (cx + k < p.W) y[k] = v[k];
      }
    }
  } else {
    const int Ho = p.H / 2, Wo = p.W / 2;
    const int qw = (Wo + 1) >> 1, ipf = (p.R / 2) * qw;
    for (int it = tid; it < nm * ipf; it += NTHREADS) {
      const int ml = it / ipf, rest = it - ml * ipf;
      const int pr = rest / qw, pc = (rest - pr * qw) * 2;
      const int orow = T.r0 / 2 + pr, o = o_s[ml];
      if (orow >= Ho || o < 0) continue;
      const int off = (m0 + ml) * pst + 2 * pr * p.bcols + 2 * pc;
      const float4 a = sum(off), b = sum(off + p.bcols);
      const size_t plane = (size_t)T.n * p.Co + o;
      // window d of pooled output e: row 2 pr + (d >> 1), column 2 (pc + e) + (d & 1)
      const float win[2][4] = {{a.x, a.y, b.x, b.y}, {a.z, a.w, b.z, b.w}};
      float out[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        float mx = 0.f;
#pragma unroll
        for (int d = 0; d < 4; ++d) {
          float v = win[e][d] + b_s[ml];
          if (skip && pc + e < Wo)
            v += __ldg(skip + (plane * p.H + 2 * orow + (d >> 1)) * p.W + 2 * (pc + e) + (d & 1));
          if (relu) v = fmaxf(v, 0.f);
          mx = d == 0 ? v : fmaxf(mx, v);
        }
        out[e] = mx;
      }
      float* y = p.y + (plane * Ho + orow) * Wo + pc;
      if ((Wo & 1) == 0) {
        *reinterpret_cast<float2*>(y) = make_float2(out[0], out[1]);
      } else {
        y[0] = out[0];
        if (pc + 1 < Wo) y[1] = out[1];
      }
    }
  }
}

// PAIR: the CTAs of a cluster form pairs (cluster ranks 2k, 2k + 1) that run
// two filter blocks of the same tile and channel range with cta_group::2 MMAs
// (M = 256): each CTA holds its own block's weights (A) and stages half of
// the tile's pixels (B columns 0 .. N/2-1 in the even CTA, N/2 .. N-1 in the
// odd one); the even CTA's MMA thread issues for both, once the odd CTA has
// reported its stage full, and its commits arrive in both CTAs.  Pairs run in
// cluster-split mode (one tile per CTA).
template <bool SPLIT, bool F16, bool PAIR>
__global__ void __launch_bounds__(flat_threads<SPLIT, F16>(), 1) ppconv_tcf_kernel(const FlatParams p, const __grid_constant__ CUtensorMap xmap) {
  static_assert(SPLIT || !PAIR, "CTA pairs run in cluster-split mode");
  constexpr bool WR = weight_ring<SPLIT, F16>();
  constexpr int KCH = F16 ? 16 : KC;  // input channels per chunk
  constexpr int CPH = KCH / 2;         // channels per K half (16 bytes of one pixel row of an operand)
  extern __shared__ unsigned char smem_raw[];
  // Offset from the shared array itself (not an integer round trip), so the
  // compiler keeps every access below in the shared state space.
  unsigned char* smem = smem_raw + ((1024u - (su32(smem_raw) & 1023u)) & 1023u);
  __shared__ __align__(8) uint64_t full[2], raw_full[2], empty[2], acc_full[2], acc_empty[2], done_bar;
  __shared__ __align__(8) uint64_t wempty[WSL_MAX];  // a weight-ring slot has been read by its MMAs
  __shared__ __align__(8) uint64_t pfull[2];  // PAIR, even CTA: the odd CTA's stage is full
  __shared__ uint32_t tmem_s;
  __shared__ volatile int abort_s;
  __shared__ int o_s[FB / 2];    // split phase: original index of each owned filter (-1 beyond Co)
  __shared__ float b_s[FB / 2];  // and its bias

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  auto wait = [&](uint64_t* bar, uint32_t parity) -> bool {
    const uint32_t a = su32(bar);
    for (long i = 0; i < WAIT_LIMIT; ++i) {
      if (mbar_try(a, parity)) return true;
      if ((i & 255) == 255 && abort_s) return false;
    }
    abort_s = 1;
    atomicOr(p.status, ppc::kStatusTimeout);
    return false;
  };

  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      // a stage is full once every loader thread has stored its part of the
      // input operands and the chunk's weight copies (one more arrival each,
      // with its bytes: the three group copies, or without the ring the whole
      // chunk) have landed: the MMA thread waits on one barrier per chunk
      mbar_init(su32(&full[s]), NLOAD + (WR ? NGRP : 1));
      mbar_init(su32(&raw_full[s]), 1);
      mbar_init(su32(&empty[s]), 1);
      mbar_init(su32(&acc_full[s]), 1);
      mbar_init(su32(&acc_empty[s]), NEPI);
    }
    mbar_init(su32(&done_bar), 1);
    if (WR)
      for (int k = 0; k < WSL_MAX; ++k) mbar_init(su32(&wempty[k]), 1);
    mbar_init(su32(&pfull[0]), 1);
    mbar_init(su32(&pfull[1]), 1);
    abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == MMA_WARP) {
    if (PAIR) {  // both CTAs of the pair allocate together
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tmem_s)),
                   "n"(2 * NMAX));
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tmem_s)),
                   "n"(2 * NMAX));
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
  }
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  const uint32_t tmem = tmem_s;

  // This CTA's tiles and channel-chunk range.  Cluster rank crank: split rank
  // srank, and with pairs the position pp in the pair (0: issues the MMAs).
  const int csize = PAIR ? 2 * p.split : p.split;
  const int crank = SPLIT ? (int)blockIdx.x % csize : 0;
  const int pp = PAIR ? (crank & 1) : 0;
  const int srank = PAIR ? (crank >> 1) : crank;
  int nmine, c_beg, c_end;
  if (SPLIT) {
    nmine = 1;
    c_beg = srank * p.nch / p.split;
    c_end = (srank + 1) * p.nch / p.split;
  } else {
    nmine = p.ntiles > (int)blockIdx.x ? (p.ntiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
    c_beg = 0;
    c_end = p.nch;
  }
  auto tile_index = [&](int i) -> int {
    return SPLIT ? (int)blockIdx.x / csize : (int)blockIdx.x + i * (int)gridDim.x;
  };
  // with pairs a tile index names a pair of filter blocks (p.nfb counts pairs)
  auto my_tile = [&](int t) -> Tile {
    Tile T = tile_of(p, t);
    if (PAIR) T.fb = 2 * T.fb + pp;
    return T;
  };
  const int brows = p.R + 2;

  if (warp < MMA_WARP) {
    // ------------------------------------------------------------ loaders
    // Chunk sequence g = 0 .. nall-1 of this CTA (tiles in order, each over the
    // CTA's chunk range).
    const int nchm = c_end - c_beg;
    const int nall = nmine * nchm;
    // Each loader thread's (K half, pixel) items are the same for every chunk:
    // their offsets in the input box and in the operand tiles are computed once.
    int roff[ITEMS_MAX], doff[ITEMS_MAX], rowcol[ITEMS_MAX];
#pragma unroll
    for (int b = 0; b < ITEMS_MAX; ++b) {
      const int it = b * NLOAD + tid;
      const int kh = it >= p.npix ? 1 : 0;
      const int pix = it - kh * p.npix;
      // operand row pix holds staged pixel pix (+ N/2 in the odd CTA of a pair);
      // staged pixels past the box's rows only feed dropped columns: zeros
      const int sp = PAIR ? pix + pp * (p.ncols >> 1) : pix;
      const int br = sp / p.bcols, bc = sp - br * p.bcols;
      const bool has = it < 2 * p.npix, inbox = !PAIR || br < brows;
      // 4-D box: columns from -4, zero filled outside the image.  Packed rows
      // (plane): row br of the tile starts br * W elements into the box (after
      // the tile's alignment shift, added per tile); the halo columns, which
      // the packed rows do not hold, are zeros.
      roff[b] = !(has && inbox) ? -1
                     : (p.plane ? ((bc >= 1 && bc <= p.W) ? kh * CPH * p.raw_w + br * p.W + bc - 1 : -1)
                                : (kh * CPH * brows + br) * p.raw_w + bc + 3);
      doff[b] = has ? kh * p.npixa + pix : -1;
      rowcol[b] = (kh << 30) | ((inbox ? br : 0x7FFF) << 15) | bc;  // row 0x7FFF: outside the image
    }
    const int cstride = p.plane ? p.raw_w : brows * p.raw_w;  // between two channels of the box
    // Packed rows: the box starts at element (r0 - 1) W rounded down to a
    // multiple of 4 (16 bytes, as a tensor-map copy requires); the remainder is
    // the tile's shift into the box.
    auto plane_shift = [&](const Tile& T) -> int { return p.plane ? ((T.r0 - 1) * p.W) & 3 : 0; };
    // Input box of chunk gg (thread 0): [8 channels][rows r0-1 ..][columns -4 ..];
    // zero fill outside the image is the convolution's padding.
    auto issue_raw = [&](int gg, unsigned char* dst) {
      const int i = gg / nchm, c = c_beg + gg % nchm;
      const Tile T = my_tile(tile_index(i));
      mbar_arrive_expect_tx(su32(&raw_full[gg & 1]), (uint32_t)p.raw_bytes);
      if (p.plane) {
        const int x0 = (T.r0 - 1) * p.W - plane_shift(T);
        asm volatile(
            "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, "
            "%4}], [%5];" ::"r"(su32(dst)),
            "l"(reinterpret_cast<uint64_t>(&xmap)), "r"(x0), "r"(c * KCH), "r"(T.n), "r"(su32(&raw_full[gg & 1]))
            : "memory");
        return;
      }
      asm volatile(
          "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, "
          "%4, %5}], [%6];" ::"r"(su32(dst)),
          "l"(reinterpret_cast<uint64_t>(&xmap)), "r"(-4), "r"(T.r0 - 1), "r"(c * KCH), "r"(T.n),
          "r"(su32(&raw_full[gg & 1]))
          : "memory");
    };
    // With a ring of their own the boxes are copied one or two chunks ahead of use
    // (as many as the ring has slots), not only once the chunk's stage is free.
    int g = 0, raw_issued = 0, w_issued = 0;
    // Without the ring: the weights of chunk gg, whole, into chunk slot s (the
    // ring's group slots 3 s .. 3 s + 2), on the stage's full barrier (thread 0).
    auto issue_w = [&](int gg, int s) {
      const Tile T = my_tile(tile_index(gg / nchm));
      const unsigned char* src = p.wt + ((size_t)T.fb * p.nch + c_beg + gg % nchm) * W_BYTES;
      mbar_arrive_expect_tx(su32(&full[s]), W_BYTES);
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
              su32(smem + (size_t)s * W_BYTES)),
          "l"(src), "r"(W_BYTES), "r"(su32(&full[s]))
          : "memory");
    };
    // The weights do not depend on the previous kernel in the stream: without
    // the ring the first two chunks' copies start before waiting for it
    // (programmatic dependent launch); everything that reads x comes after.
    if (!WR && tid == 0)
      for (; w_issued < 2 && w_issued < nall; ++w_issued) issue_w(w_issued, w_issued);
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (tid == 0 && p.use_tma && p.sep)
      for (; raw_issued < p.sep && raw_issued < nall; ++raw_issued)
        issue_raw(raw_issued, smem + p.raw_off + raw_issued * p.raw_slot);
    bool stop = false;  // identical in every loader thread (decided by group_any)
    uint32_t range_bad = 0;  // f16: nonzero once an input is non-finite or overflows fp16 after scaling
    for (int i = 0; i < nmine && !stop; ++i) {
      const Tile T = my_tile(tile_index(i));
      const float* xb = p.x + (size_t)T.n * p.Ci * p.H * p.W;
      const int tsh = plane_shift(T);
      for (int c = c_beg; c < c_end; ++c, ++g) {
        const int s = g & 1, use = g >> 1;
        // Without a tensor map the chunk's input values are fetched into
        // registers first: that needs no free stage, so it overlaps the wait.
        // With a box ring the box has a slot of its own and lands ahead of time,
        // so it is read into registers before the stage is free too, while the
        // MMAs of the two previous chunks still read it; f16 also splits it
        // there (the tf32 split is cheap and follows the stage wait).
        // v holds an item's input values, or (f16, read early) its packed hi words then lo words
        float v[ITEMS_MAX][CPH];
        const bool early = p.use_tma && p.sep;
        if (early) {
          if (group_any<NLOAD>(!wait(&raw_full[s], (uint32_t)(use & 1)))) {
            stop = true;
            break;
          }
          const float* raw = reinterpret_cast<const float*>(smem + p.raw_off + (size_t)(g & (p.sep - 1)) * p.raw_slot);
#pragma unroll
          for (int b = 0; b < ITEMS_MAX; ++b) {
            if constexpr (F16) {
              // split as soon as read: only the packed halves stay live
              float u[CPH];
#pragma unroll
              for (int k = 0; k < CPH; ++k) u[k] = roff[b] >= 0 ? raw[roff[b] + tsh + k * cstride] : 0.f;
              uint4 h = make_uint4(0, 0, 0, 0), l = h;
              if (doff[b] >= 0) range_bad |= split_f16x8(u, p.xscale, h, l);
              v[b][0] = __uint_as_float(h.x);
              v[b][1] = __uint_as_float(h.y);
              v[b][2] = __uint_as_float(h.z);
              v[b][3] = __uint_as_float(h.w);
              v[b][4] = __uint_as_float(l.x);
              v[b][5] = __uint_as_float(l.y);
              v[b][6] = __uint_as_float(l.z);
              v[b][7] = __uint_as_float(l.w);
            } else {
#pragma unroll
              for (int k = 0; k < CPH; ++k) v[b][k] = roff[b] >= 0 ? raw[roff[b] + tsh + k * cstride] : 0.f;
            }
          }
          // the slot is rewritten next by a tensor-map copy (async proxy): each thread orders its reads of
          // it before that copy with a proxy fence, then the loader barrier lets thread 0 issue it
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          group_sync<NLOAD>();
          if (tid == 0 && raw_issued < nall && raw_issued == g + p.sep) {
            issue_raw(raw_issued, smem + p.raw_off + (size_t)(raw_issued & (p.sep - 1)) * p.raw_slot);
            ++raw_issued;
          }
        }
        if (!p.use_tma) {
#pragma unroll
          for (int b = 0; b < ITEMS_MAX; ++b) {
            const int kh = rowcol[b] >> 30, br = (rowcol[b] >> 15) & 0x7FFF, bc = rowcol[b] & 0x7FFF;
            const int r = T.r0 - 1 + br, cc = bc - 1;
            const bool inside = doff[b] >= 0 && (unsigned)r < (unsigned)p.H && (unsigned)cc < (unsigned)p.W;
#pragma unroll
            for (int k = 0; k < CPH; ++k) {
              const int ch = c * KCH + kh * CPH + k;
              v[b][k] = (inside && ch < p.Ci) ? __ldg(xb + ((size_t)ch * p.H + r) * p.W + cc) : 0.f;
            }
          }
        }
        if (group_any<NLOAD>(use > 0 && !wait(&empty[s], (uint32_t)((use - 1) & 1)))) {
          stop = true;
          break;
        }
        unsigned char* st = smem + p.xoff + (size_t)s * p.xstage;
        float4* hi = reinterpret_cast<float4*>(st);
        float4* lo = reinterpret_cast<float4*>(st + p.lo_off);
        if (tid == 0) {
          if (!WR && g >= 2) {
            issue_w(g, s);
            ++w_issued;
          }
          if (p.use_tma && !p.sep) {
            issue_raw(g, reinterpret_cast<unsigned char*>(lo));  // lands in the lo operand, split in place below
            ++raw_issued;
          }
        }
        if (p.use_tma && !early) {
          if (group_any<NLOAD>(!wait(&raw_full[s], (uint32_t)(use & 1)))) {
            stop = true;
            break;
          }
          const float* raw = p.sep ? reinterpret_cast<const float*>(smem + p.raw_off + (size_t)(g & (p.sep - 1)) * p.raw_slot)
                                   : reinterpret_cast<const float*>(lo);
#pragma unroll
          for (int b = 0; b < ITEMS_MAX; ++b)
#pragma unroll
            for (int k = 0; k < CPH; ++k) v[b][k] = roff[b] >= 0 ? raw[roff[b] + tsh + k * cstride] : 0.f;
          // A ring slot is rewritten next by a tensor-map copy (async proxy): each
          // thread orders its reads of the slot before that copy with a proxy fence.
          if (p.sep) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          group_sync<NLOAD>();  // the whole box is in registers before its buffer is reused
          if (p.sep && tid == 0 && raw_issued < nall && raw_issued == g + p.sep) {
            issue_raw(raw_issued, smem + p.raw_off + (size_t)(raw_issued & (p.sep - 1)) * p.raw_slot);
            ++raw_issued;
          }
        }
#pragma unroll
        for (int b = 0; b < ITEMS_MAX; ++b) {
          if (doff[b] >= 0) {
            const int dst = doff[b];
            if constexpr (F16) {
              uint4 h, l;
              if (early) {
                h = make_uint4(__float_as_uint(v[b][0]), __float_as_uint(v[b][1]), __float_as_uint(v[b][2]),
                               __float_as_uint(v[b][3]));
                l = make_uint4(__float_as_uint(v[b][4]), __float_as_uint(v[b][5]), __float_as_uint(v[b][6]),
                               __float_as_uint(v[b][7]));
              } else {
                range_bad |= split_f16x8(&v[b][0], p.xscale, h, l);
              }
              reinterpret_cast<uint4*>(hi)[dst] = h;
              reinterpret_cast<uint4*>(lo)[dst] = l;
            } else {
              float4 h;
              h.x = tf32_hi(v[b][0]);
              h.y = tf32_hi(v[b][1]);
              h.z = tf32_hi(v[b][2]);
              h.w = tf32_hi(v[b][3]);
              hi[dst] = h;
              lo[dst] = make_float4(v[b][0] - h.x, v[b][1] - h.y, v[b][2] - h.z, v[b][3] - h.w);
            }
          }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive(su32(&full[s]));
      }
    }
    if (F16 && range_bad != 0) atomicOr(p.status, ppc::kStatusF16Range);
    if (tid == 0) {
      // No copy may still be writing shared memory when the CTA exits: wait
      // (bounded) for the last copies issued into each stage.  (After a timeout
      // a stage's barrier may lack loader arrivals and never complete; the
      // bounded wait then outlasts any copy still in flight.)
      for (int gg = raw_issued > 2 ? raw_issued - 2 : 0; gg < raw_issued; ++gg)
        for (long k = 0; k < WAIT_LIMIT && !mbar_try(su32(&raw_full[gg & 1]), (uint32_t)((gg >> 1) & 1)); ++k) {
        }
      for (int gg = w_issued > 2 ? w_issued - 2 : 0; gg < w_issued; ++gg)
        for (long k = 0; k < WAIT_LIMIT && !mbar_try(su32(&full[gg & 1]), (uint32_t)((gg >> 1) & 1)); ++k) {
        }
    }
    __syncwarp();
  } else if (warp == MMA_WARP) {
    // ------------------------------------------------------------ MMA issuer
    // (with pairs: in the even CTA; the odd CTA's thread reports its stages full)
    const uint16_t pmask = (uint16_t)(3u << (crank & ~1));  // PAIR: both CTAs of this pair
    if (PAIR && lane == 0 && pp == 1) {
      int g = 0;
      bool ok = true;
      for (int c = c_beg; c < c_end && ok; ++c, ++g) {
        const int s = g & 1, use = g >> 1;
        ok = wait(&full[s], (uint32_t)(use & 1));
        if (ok) mbar_arrive_remote(map_rank(su32(&pfull[s]), (uint32_t)(crank ^ 1)));
      }
      asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    } else if (lane == 0) {
      int g = 0, wslot = 0;  // chunk count and the weight-ring slot of the next group
      for (int i = 0; i < nmine && !abort_s; ++i) {
        const int b = p.nbuf == 2 ? (i & 1) : 0, ub = p.nbuf == 2 ? (i >> 1) : i;
        if (ub > 0 && !wait(&acc_empty[b], (uint32_t)((ub - 1) & 1))) break;
        tm_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * NMAX);
        const uint32_t d2 = d + (uint32_t)p.acc2;  // f16: the second accumulator
        bool okc = true;
        for (int c = c_beg; c < c_end; ++c, ++g) {
          const int s = g & 1, use = g >> 1;
          if (!wait(&full[s], (uint32_t)(use & 1)) || (PAIR && !wait(&pfull[s], (uint32_t)(use & 1)))) {
            okc = false;
            break;
          }
          tm_fence_after();
          const unsigned char* st = smem + p.xoff + (size_t)s * p.xstage;
          // descriptors hold address / 16 in their low 14 bits (operands lie below
          // 256 KB), so moving an operand by k pixels of 16 bytes adds k
          const uint64_t xh0 = smem_desc(su32(st), (uint32_t)p.npixa * 16);
          const uint64_t xl0 = smem_desc(su32(st + p.lo_off), (uint32_t)p.npixa * 16);
          // the chunk's three weight groups: consecutive slots of the ring
          int gs[NGRP];
#pragma unroll
          for (int k = 0; k < NGRP; ++k) {
            gs[k] = wslot;
            wslot = wslot + 1 == p.wsl ? 0 : wslot + 1;
          }
          const uint32_t acc0 = c == c_beg ? 0u : 1u;  // the range's first chunk overwrites the accumulators
#pragma unroll
          for (int t = 0; t < NTAP; ++t) {
            const uint64_t off = (uint64_t)((t / 3) * p.bcols + t % 3);
            // hi and lo rows of a tap in each K half; lo rows follow the hi rows
            const uint64_t whi = smem_desc(su32(smem + (size_t)gs[t / 3] * GRP_BYTES + (t % 3) * TAP_BYTES), 2 * FB * 16);
            const uint64_t wlo = whi + (uint64_t)FB;
            if (PAIR) {
              if (F16) {
                mma_f16_pair(d, whi, xh0 + off, p.idesc, t == 0 ? acc0 : 1u);
                mma_f16_pair(d2, wlo, xh0 + off, p.idesc, t == 0 ? acc0 : 1u);
                mma_f16_pair(d2, whi, xl0 + off, p.idesc, 1u);
              } else {
                mma_tf32_pair(d, whi, xh0 + off, p.idesc, t == 0 ? acc0 : 1u);
                mma_tf32_pair(d, wlo, xh0 + off, p.idesc, 1u);
                mma_tf32_pair(d, whi, xl0 + off, p.idesc, 1u);
              }
            } else if (F16) {
              // acc1 += w_hi x_hi; acc2 += w_lo x_hi + w_hi x_lo (both lo parts scaled by 2^11)
              mma_f16(d, whi, xh0 + off, p.idesc, t == 0 ? acc0 : 1u);
              mma_f16(d2, wlo, xh0 + off, p.idesc, t == 0 ? acc0 : 1u);
              mma_f16(d2, whi, xl0 + off, p.idesc, 1u);
            } else {
              mma_tf32(d, whi, xh0 + off, p.idesc, t == 0 ? acc0 : 1u);
              mma_tf32(d, wlo, xh0 + off, p.idesc, 1u);
              mma_tf32(d, whi, xl0 + off, p.idesc, 1u);
            }
            if (WR && t % 3 == 2) {  // the group's slot is free for the producer once these MMAs complete
              if (PAIR)
                mma_commit_pair(su32(&wempty[gs[t / 3]]), pmask);
              else
                mma_commit(su32(&wempty[gs[t / 3]]));
            }
          }
          if (PAIR)
            mma_commit_pair(su32(&empty[s]), pmask);
          else
            mma_commit(su32(&empty[s]));
        }
        if (!okc) break;
        if (PAIR)
          mma_commit_pair(su32(&acc_full[b]), pmask);
        else
          mma_commit(su32(&acc_full[b]));
      }
      // every MMA issued by this thread is complete before TMEM is released
      // the next kernel in the stream may start its prologue (it waits for this
      // grid to complete before it reads anything this grid writes)
      asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
      if (PAIR)
        mma_commit_pair(su32(&done_bar), pmask);
      else
        mma_commit(su32(&done_bar));
      wait(&done_bar, 0u);
    }
    __syncwarp();
  } else if (warp == WPROD_WARP) {
    // ------------------------------------------------------------ weight producer
    // A chunk's weights are three groups of 3 tap tiles (24 KB each), copied
    // into a ring of p.wsl slots.  Group k of a chunk is copied as soon as the
    // MMAs of the group that held its slot before have completed; with 7 slots
    // (2 1/3 chunks) the last group of chunk g is copied while the MMAs of
    // chunk g - 2 still run, not only once they all have.  The three copies
    // arrive (with their bytes) on the stage's full barrier, so the MMA thread
    // still waits once per chunk; the copies of chunk g go out only after the
    // barrier's previous phase (chunk g - 2) has completed.
    if (WR && lane == 0) {
      const int nchm = c_end - c_beg;
      const int nall = nmine * nchm;
      int slot = 0, use = 0, issued = 0;  // ring position, its round, groups issued
      bool ok = true;
      for (int gg = 0; gg < nall && ok; ++gg) {
        const int s = gg & 1;
        if (gg >= 2) ok = wait(&full[s], (uint32_t)(((gg - 2) >> 1) & 1));
        const Tile T = my_tile(tile_index(gg / nchm));
        const unsigned char* src = p.wt + ((size_t)T.fb * p.nch + c_beg + gg % nchm) * W_BYTES;
        for (int k = 0; k < NGRP && ok; ++k) {
          if (use > 0) ok = wait(&wempty[slot], (uint32_t)((use - 1) & 1));
          if (!ok) break;
          mbar_arrive_expect_tx(su32(&full[s]), GRP_BYTES);
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                  su32(smem + (size_t)slot * GRP_BYTES)),
              "l"(src + (size_t)k * GRP_BYTES), "r"(GRP_BYTES), "r"(su32(&full[s]))
              : "memory");
          ++issued;
          if (++slot == p.wsl) {
            slot = 0;
            ++use;
          }
        }
      }
      // No copy may still be writing shared memory when the CTA exits: wait
      // (bounded) for the last two chunks' barriers (after a timeout a
      // barrier may lack loader arrivals; the bounded wait outlasts any copy).
      const int last = (issued + NGRP - 1) / NGRP;  // chunks with at least one group issued
      for (int gg = last > 2 ? last - 2 : 0; gg < last; ++gg)
        for (long w = 0; w < WAIT_LIMIT && !mbar_try(su32(&full[gg & 1]), (uint32_t)((gg >> 1) & 1)); ++w) {
        }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;                     // TMEM lane quadrant of this warp
    const int half = (warp - EPI_WARP0) >> 2;   // the two warps of a quadrant share the work
    const bool pool = p.flags & PP_POOL2;
    const bool relu = p.flags & PP_RELU;
    const float* skip = (p.flags & PP_ADD_SKIP) ? p.skip : nullptr;
    for (int i = 0; i < nmine; ++i) {
      const int b = p.nbuf == 2 ? (i & 1) : 0, ub = p.nbuf == 2 ? (i >> 1) : i;
      // the whole warp leaves together: its TMEM loads are warp-collective
      if (!__all_sync(0xffffffffu, wait(&acc_full[b], (uint32_t)(ub & 1)))) break;
      tm_fence_after();
      const Tile T = my_tile(tile_index(i));
      const uint32_t lanebase = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * NMAX);
      const uint32_t lane2 = lanebase + (uint32_t)p.acc2;  // f16: the second accumulator
      const int m = 32 * q + lane;  // filter within the block = TMEM lane
      // f16: the filter's inverse scale (the layout holds nfb x FB entries, padding included)
      const float rs = F16 ? __ldg(p.rscale + T.fb * FB + m) : 1.f;
      if (SPLIT) {
        // this CTA's partial tile into its own shared memory (free once the
        // accumulators are ready): row m of [128][ncols + 4], padded so a warp's
        // 16-byte stores to 32 rows spread over the banks
        // (4 TMEM loads per wait; the bounds are warp-uniform, as the
        // warp-collective loads require)
        float* prow = reinterpret_cast<float*>(smem) + m * (p.ncols + 4);
        for (int cb0 = half * 8; cb0 < p.ncols; cb0 += 64) {
          float a[4][8], a2[4][8];
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (cb0 + 16 * u < p.ncols) {
              tm_ld8(lanebase + (uint32_t)(cb0 + 16 * u), a[u]);
              if constexpr (F16) tm_ld8(lane2 + (uint32_t)(cb0 + 16 * u), a2[u]);
            }
          tm_wait_ld();
          if constexpr (F16) {
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int k = 0; k < 8; ++k) a[u][k] = fmaf(a2[u][k], 0x1p-11f, a[u][k]) * rs;
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int cb = cb0 + 16 * u;
            if (cb < p.ncols) {
              *reinterpret_cast<float4*>(prow + cb) = make_float4(a[u][0], a[u][1], a[u][2], a[u][3]);
              *reinterpret_cast<float4*>(prow + cb + 4) = make_float4(a[u][4], a[u][5], a[u][6], a[u][7]);
            }
          }
        }
      } else {
        const int jr = T.fb * FB + m;
        const bool valid = jr < p.Co;
        const int o = valid ? __ldg(p.perm + jr) : 0;
        const float bs = (valid && p.bias) ? __ldg(p.bias + jr) : 0.f;
        const size_t plane = (size_t)T.n * p.Co + o;
        const bool vec = (p.W & 3) == 0;
        if (!pool) {
          for (int rr = half; rr < p.R; rr += 2) {
            const int row = T.r0 + rr;
            if (row >= p.H) break;
            float* yr = p.y + (plane * p.H + row) * p.W;
            const float* sr = skip ? skip + (plane * p.H + row) * p.W : nullptr;
            for (int cb = 0; cb < p.W; cb += 8) {
              float a[8], a2[8];
              tm_ld8(lanebase + (uint32_t)(rr * p.bcols + cb), a);
              if constexpr (F16) tm_ld8(lane2 + (uint32_t)(rr * p.bcols + cb), a2);
              tm_wait_ld();
              if constexpr (F16) {
#pragma unroll
                for (int k = 0; k < 8; ++k) a[k] = fmaf(a2[k], 0x1p-11f, a[k]) * rs;
              }
              if (valid) {
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                  a[k] += bs;
                  if (sr && cb + k < p.W) a[k] += __ldg(sr + cb + k);
                  if (relu) a[k] = fmaxf(a[k], 0.f);
                }
                if (vec && cb + 8 <= p.W) {
                  *reinterpret_cast<float4*>(yr + cb) = make_float4(a[0], a[1], a[2], a[3]);
                  *reinterpret_cast<float4*>(yr + cb + 4) = make_float4(a[4], a[5], a[6], a[7]);
                } else {
#pragma unroll
                  for (int k = 0; k < 8; ++k)
                    if (cb + k < p.W) yr[cb + k] = a[k];
                }
              }
            }
          }
        } else {
          const int Ho = p.H / 2, Wo = p.W / 2;
          for (int rr = 2 * half; rr < p.R; rr += 4) {
            const int row = T.r0 + rr;
            if (row >= p.H) break;
            float* yr = p.y + (plane * Ho + row / 2) * Wo;
            const float* s0 = skip ? skip + (plane * p.H + row) * p.W : nullptr;
            for (int cb = 0; cb < p.W; cb += 8) {
              float a[8], bb[8], a2[8], bb2[8];
              tm_ld8(lanebase + (uint32_t)(rr * p.bcols + cb), a);
              tm_ld8(lanebase + (uint32_t)((rr + 1) * p.bcols + cb), bb);
              if constexpr (F16) {
                tm_ld8(lane2 + (uint32_t)(rr * p.bcols + cb), a2);
                tm_ld8(lane2 + (uint32_t)((rr + 1) * p.bcols + cb), bb2);
              }
              tm_wait_ld();
              if constexpr (F16) {
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                  a[k] = fmaf(a2[k], 0x1p-11f, a[k]) * rs;
                  bb[k] = fmaf(bb2[k], 0x1p-11f, bb[k]) * rs;
                }
              }
              if (valid) {
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                  a[k] += bs;
                  bb[k] += bs;
                  if (s0 && cb + k < p.W) {
                    a[k] += __ldg(s0 + cb + k);
                    bb[k] += __ldg(s0 + p.W + cb + k);
                  }
                  if (relu) {
                    a[k] = fmaxf(a[k], 0.f);
                    bb[k] = fmaxf(bb[k], 0.f);
                  }
                }
#pragma unroll
                for (int k = 0; k < 4; ++k)
                  if (cb + 2 * k < p.W)
                    yr[cb / 2 + k] = fmaxf(fmaxf(a[2 * k], a[2 * k + 1]), fmaxf(bb[2 * k], bb[2 * k + 1]));
              }
            }
          }
        }
      }
      tm_fence_before();
      mbar_arrive(su32(&acc_empty[b]));
    }
  }

  if (SPLIT) {
    // Every thread of every CTA of the cluster arrives at both cluster
    // barriers, also after an early stop, so they always complete.  The first
    // (release / acquire at cluster scope) orders every CTA's partial tile in
    // its shared memory, and the filter table below, before the reads; the
    // second keeps each CTA's shared memory alive until the others have read it.
    // This CTA finishes filters [m0, m1) of the tile (at most FB / 2 of them);
    // their original indices and biases are fetched now, so the loads overlap
    // the barrier wait.
    const int tile = (int)blockIdx.x / csize, rstride = PAIR ? 2 : 1;
    const int m0 = srank * FB / p.split, m1 = (srank + 1) * FB / p.split, nm = m1 - m0;
    const Tile T = my_tile(tile);
    if (tid < nm) {
      const int jr = T.fb * FB + m0 + tid;
      o_s[tid] = jr < p.Co ? __ldg(p.perm + jr) : -1;
      b_s[tid] = (jr < p.Co && p.bias) ? __ldg(p.bias + jr) : 0.f;
    }
    __syncwarp();
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
    if (!abort_s) {
      float* part = reinterpret_cast<float*>(smem);
      switch (p.split) {
        case 2: split_reduce<2>(p, T, m0, nm, part, o_s, b_s, tid, rstride, pp); break;
        case 4: split_reduce<4>(p, T, m0, nm, part, o_s, b_s, tid, rstride, pp); break;
        case 8: split_reduce<8>(p, T, m0, nm, part, o_s, b_s, tid, rstride, pp); break;
        default: split_reduce<16>(p, T, m0, nm, part, o_s, b_s, tid, rstride, pp); break;
      }
    }
    __syncwarp();
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
  }

  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (warp == MMA_WARP) {
    if (PAIR)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(2 * NMAX));
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(2 * NMAX));
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

struct DeviceState {
  int sms = 0;
  int max_clusters[MAX_SPLIT + 1] = {};  // co-resident clusters of each size (0: size unusable)
  EncodeTiledFn encode = nullptr;
};
DeviceState g_dev[ppc::DeviceOnce::kMaxDevices];
ppc::DeviceOnce g_dev_once;  // fills g_dev[dev] once per device (its ready flag publishes it)

cudaError_t init_device(int dev) {
  DeviceState& D = g_dev[dev];
  cudaError_t e = cudaDeviceGetAttribute(&D.sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(ppconv_tcf_kernel<false, false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_ALLOC)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(ppconv_tcf_kernel<true, false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_ALLOC)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(ppconv_tcf_kernel<false, true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_ALLOC)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(ppconv_tcf_kernel<true, true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_ALLOC)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(ppconv_tcf_kernel<true, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_ALLOC)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(ppconv_tcf_kernel<true, true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_ALLOC)) != cudaSuccess)
    return e;
  // then only portable sizes (up to 8) can be used
  if (cudaFuncSetAttribute(ppconv_tcf_kernel<true, false, false>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
      cudaSuccess)
    cudaGetLastError();
  if (cudaFuncSetAttribute(ppconv_tcf_kernel<true, true, false>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
      cudaSuccess)
    cudaGetLastError();
  if (cudaFuncSetAttribute(ppconv_tcf_kernel<true, false, true>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
      cudaSuccess)
    cudaGetLastError();
  if (cudaFuncSetAttribute(ppconv_tcf_kernel<true, true, true>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
      cudaSuccess)
    cudaGetLastError();
  for (int s = 2; s <= MAX_SPLIT; s *= 2) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = (unsigned)s;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3((unsigned)s);
    cfg.blockDim = dim3(NTHREADS);
    cfg.dynamicSmemBytes = SMEM_ALLOC;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    // split launches run 576 threads in both precisions, one CTA per SM, with the same shared memory
    if (cudaOccupancyMaxActiveClusters(&n, ppconv_tcf_kernel<true, false, false>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      n = 0;
    }
    D.max_clusters[s] = n;
  }
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    D.encode = reinterpret_cast<EncodeTiledFn>(fn);
  else
    cudaGetLastError();  // without the entry point every launch uses per-thread loads
  return cudaSuccess;
}

// The current device's state, set up on first use (thread-safe), or null.
DeviceState* prepare() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= ppc::DeviceOnce::kMaxDevices) return nullptr;
  if (g_dev_once.run(init_device) != cudaSuccess) return nullptr;
  return &g_dev[dev];
}

struct FlatGeo {
  int bcols = 0, R = 0, ncols = 0, npix = 0, npixa = 0, raw_w = 0, raw_bytes = 0, tiles_y = 0, ntiles = 0, split = 1;
  int wsl = 0, xoff = 0, xstage = 0, lo_off = 0, sep = 0, raw_off = 0, raw_slot = 0;
  bool pair = false;  // CTA pairs over two filter blocks (ntiles then counts pairs of blocks)
  double cost = 1e300;
  // the split as the geometry API reports it (PP_FLAT_PAIRED set for pairs)
  int code() const { return split | (pair ? PP_FLAT_PAIRED : 0); }
};

// Geometry of one launch: rows per tile and split, by a model of the time in
// SM cycles: an MMA of N columns takes the longer of its multiply-adds at
// ~1850 per cycle and its operand reads (4 KB of weights + 32 N bytes of
// input) at 128 shared-memory bytes per cycle; a chunk also needs its 73.7 KB
// of weights from L2 (~48 bytes per cycle) and at least ~1500 cycles of
// staging latency with two stages; a start-up and pipeline fill of ~5000
// cycles; the split's partial-tile round trip through L2 at ~64 bytes per
// cycle; and clusters beyond those co-resident on the GPU run in later waves.
// Every geometry the kernel can run for this shape, best first by the model;
// fills up to maxn entries and returns how many.
// f16: nch counts 16-channel chunks and the input box holds 16 channels; a tile
// of at most 128 columns keeps its second accumulator in the same TMEM buffer
// (double-buffered), a wider one puts it in the other buffer (single-buffered:
// its epilogue is not overlapped with the CTA's next tile).
int flat_candidates(int N, int H, int W, int nch, int nfb, bool pool, bool allow_split, const DeviceState& D,
                    FlatGeo* out, int maxn, bool f16) {
  if (W < 1 || W > WMAX || H < 1 || maxn < 1) return 0;
  const int bcols = (W + 2 + 7) / 8 * 8;
  const int nmax = NMAX;  // f16 tiles wider than ACC2 run single-buffered (below)
  const int kch = f16 ? 16 : KC;
  const int rmax = nmax / bcols;
  if (rmax < 1 || (pool && rmax < 2)) return 0;
  int n = 0;
  for (int r0 = rmax; r0 >= 1; --r0) {
    int R = std::min(r0, H);
    int ty = (H + R - 1) / R;
    R = (H + ty - 1) / ty;  // balance the rows over the tiles
    if (pool) {
      R += R & 1;
      if (R > rmax) R = rmax & ~1;
      if (R < 2) break;
    }
    ty = (H + R - 1) / R;
    for (int pair = 0; pair < 2; ++pair) {
      // pairs: two filter blocks per tile, cluster of 2 S, each CTA stages half of the tile's columns
      if (pair && (!allow_split || (nfb & 1))) continue;
      FlatGeo G;
      G.pair = pair != 0;
      G.bcols = bcols;
      G.R = R;
      G.ncols = (R * bcols + 15) / 16 * 16;
      G.npix = pair ? (G.ncols / 2 + 2 * bcols + 2 + 7) / 8 * 8 : (R + 2) * bcols;
      G.npixa = G.npix + 16;
      G.raw_w = bcols + 4;
      G.raw_bytes = kch * (R + 2) * G.raw_w * 4;
      G.tiles_y = ty;
      const int64_t nt = (int64_t)ty * (pair ? nfb / 2 : nfb) * N;
      const int in_bytes = (2 * G.npixa * 16 + 127) / 128 * 128;
      G.raw_slot = (G.raw_bytes + 127) / 128 * 128;
      // shared memory: the weight ring (7 groups of 3 taps, else 6), two input operand stages (hi, lo),
      // and a ring of two input-box slots, else one (copied one chunk ahead), else the box lands in lo
      G.xstage = 2 * in_bytes;
      G.lo_off = in_bytes;
      const auto fits = [&](int wsl, int sep) {
        return wsl * GRP_BYTES + 2 * G.xstage + sep * G.raw_slot <= SMEM_USE;
      };
      G.sep = fits(6, 2) ? 2 : (fits(6, 1) ? 1 : 0);
      if (!G.sep) G.xstage = in_bytes + std::max(in_bytes, G.raw_slot);
      G.wsl = fits(WSL_MAX, G.sep) ? WSL_MAX : 6;
      G.xoff = G.wsl * GRP_BYTES;
      G.raw_off = G.xoff + 2 * G.xstage;
      if (G.npixa > PIX_MAX || !fits(G.wsl, G.sep) || G.ncols > nmax || nt > INT32_MAX / MAX_SPLIT) continue;
      // f16 with more than ACC2 columns: the second accumulator takes the other TMEM buffer, so the
      // tile is single-buffered (a CTA's next tile starts its MMAs once this one's epilogue has read
      // the accumulators); not for pairs
      const bool wide = f16 && G.ncols > ACC2;
      if (wide && pair) continue;
      G.ntiles = (int)nt;
      const double mma = 27.0 * std::max(G.ncols * 128.0 * 8.0 / 1850.0, 32.0 + G.ncols / 4.0);
      // pairs: each SM reads half the input operand bytes per MMA and issues half the MMAs; modelled as 0.8
      // of the chunk time (the input operand reads are ~20 % of a chunk's shared-memory traffic)
      const double per_chunk = std::max(std::max(mma, W_BYTES / 48.0), 1500.0) * (pair ? 0.8 : 1.0);
      // (split mode owns at most FB / 2 filters per CTA in its second phase: pairs split at least 2 ways)
      for (int s = pair ? 2 : 1; s <= MAX_SPLIT; s *= 2) {
        const int cs = pair ? 2 * s : s;  // cluster size
        if (cs > MAX_SPLIT) break;
        if (cs > 1 && (!allow_split || s > nch || D.max_clusters[cs] <= 0 || (int64_t)G.ntiles * cs > D.sms)) continue;
        double cost;
        if (cs == 1) {
          const double waves = std::ceil((double)G.ntiles / D.sms);
          // single-buffered: every tile's epilogue but the last is no longer hidden behind MMAs
          cost = waves * nch * per_chunk + 5000.0 + (wide ? (waves - 1) * 16.0 * G.ncols : 0.0);
        } else {
          // clusters beyond those that fit on the GPU at once run in a later wave
          const double waves = std::ceil((double)G.ntiles / D.max_clusters[cs]);
          cost = waves * (std::ceil((double)nch / s) * per_chunk + 5000.0 + 16.0 * G.ncols);
        }
        G.split = s;
        G.cost = cost;
        bool dup = false;
        for (int k = 0; k < n; ++k) dup = dup || (out[k].R == G.R && out[k].code() == G.code());
        if (dup) continue;
        // insert in cost order, keeping the best maxn
        if (n == maxn && out[n - 1].cost <= cost) continue;
        int k = n < maxn ? n++ : maxn - 1;  // a full list drops its worst entry
        while (k > 0 && out[k - 1].cost > cost) {
          out[k] = out[k - 1];
          --k;
        }
        out[k] = G;
      }
    }
  }
  return n;
}

bool flat_geometry(int N, int H, int W, int nch, int nfb, bool pool, bool allow_split, const DeviceState& D,
                   FlatGeo* out, bool f16) {
  return flat_candidates(N, H, W, nch, nfb, pool, allow_split, D, out, 1, f16) == 1;
}

// The geometry (R, split) for this shape if the model can run it.
bool flat_pick(int N, int H, int W, int nch, int nfb, bool pool, const DeviceState& D, int R, int S, FlatGeo* out,
               bool f16) {
  FlatGeo all[160];
  const int n = flat_candidates(N, H, W, nch, nfb, pool, true, D, all, 160, f16);
  for (int k = 0; k < n; ++k)
    if (all[k].R == R && all[k].code() == S) {
      *out = all[k];
      return true;
    }
  return false;
}

// The geometry pinned by timing for this shape, if any.
bool pinned_geometry(const ppc::TcLayout& T, int N, int H, int W, int flags, const DeviceState& D, FlatGeo* out) {
  const ppc::TcState* st = T.state;
  if (!st || st->R <= 0 || st->key[0] != N || st->key[1] != H || st->key[2] != W || st->key[3] != flags) return false;
  return flat_pick(N, H, W, T.f16 ? T.nch16 : T.nch, T.nfb, flags & PP_POOL2, D, st->R, st->S, out, T.f16);
}

pp_status launch_geo(const FlatGeo& G, const DeviceState& Dref, const ppc::TcLayout& T, const ppc::LayerMeta& M,
                     const float* x, float* y, const float* skip, int N, int H, int W, int flags, cudaStream_t stream);

}  // namespace

namespace ppc {

pp_status tcf_launch(const TcLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N, int H,
                     int W, int flags, cudaStream_t stream) {
  if (T.FB != FB) return PP_ERR_UNSUPPORTED;
  DeviceState* D = prepare();
  if (!D) return PP_ERR_CUDA;
  const bool pool = flags & PP_POOL2;
  FlatGeo G;
  if (!pinned_geometry(T, N, H, W, flags, *D, &G) &&
      !flat_geometry(N, H, W, T.f16 ? T.nch16 : T.nch, T.nfb, pool, true, *D, &G, T.f16))
    return PP_ERR_UNSUPPORTED;
  return launch_geo(G, *D, T, M, x, y, skip, N, H, W, flags, stream);
}

}  // namespace ppc

namespace {

pp_status launch_geo(const FlatGeo& G, const DeviceState& Dref, const ppc::TcLayout& T, const ppc::LayerMeta& M,
                     const float* x, float* y, const float* skip, int N, int H, int W, int flags, cudaStream_t stream) {
  const DeviceState* D = &Dref;
  const bool f16 = T.f16;
  const int kch = f16 ? 16 : KC;
  FlatParams p;
  p.rscale = T.rscale;
  p.xscale = T.xscale;
  p.x = x;
  p.y = y;
  p.skip = (flags & PP_ADD_SKIP) ? skip : nullptr;
  p.wt = f16 ? T.a16 : T.a;
  p.perm = M.perm;
  p.bias = M.bias;
  p.status = T.status;
  p.N = N;
  p.Ci = M.Ci;
  p.Co = M.Co;
  p.H = H;
  p.W = W;
  p.nch = f16 ? T.nch16 : T.nch;
  p.nfb = G.pair ? T.nfb / 2 : T.nfb;  // pairs: the tile index names a pair of filter blocks
  p.flags = flags;
  p.bcols = G.bcols;
  p.R = G.R;
  p.ncols = G.ncols;
  p.npix = G.npix;
  p.npixa = G.npixa;
  p.raw_w = G.raw_w;
  p.raw_bytes = G.raw_bytes;
  // without the weight ring (unsplit tf32): two whole-chunk weight slots, 6 group slots
  const bool ring = G.split > 1 || G.pair || f16;
  p.wsl = ring ? G.wsl : 6;
  p.xoff = p.wsl * GRP_BYTES;
  p.xstage = G.xstage;
  p.lo_off = G.lo_off;
  p.sep = G.sep;
  p.raw_off = p.xoff + 2 * G.xstage;
  p.raw_slot = G.raw_slot;
  p.tiles_y = G.tiles_y;
  p.ntiles = G.ntiles;
  p.split = G.split;
  const bool wide = f16 && G.ncols > ACC2;  // single-buffered f16 tile
  p.nbuf = wide ? 1 : 2;
  p.acc2 = wide ? NMAX : ACC2;
  const int mrows = G.pair ? 2 * FB : FB;  // pairs: one M = 256 MMA over both CTAs' filter blocks
  p.idesc = f16 ? idesc_f16(mrows, G.ncols) : idesc_tf32(mrows, G.ncols);
  CUtensorMap xmap;
  std::memset(&xmap, 0, sizeof(xmap));
  p.use_tma = 0;
  p.plane = 0;
  const bool can_map = (reinterpret_cast<uintptr_t>(x) & 15) == 0 && D->encode;
  if (can_map && (W & 3) == 0) {
    // 4-D map over x viewed as [N][Ci][H][W] (W innermost), box [1][8][R+2][BCOLS+4]
    const cuuint64_t dims[4] = {(cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)M.Ci, (cuuint64_t)N};
    const cuuint64_t strides[3] = {(cuuint64_t)W * 4, (cuuint64_t)W * H * 4, (cuuint64_t)W * H * M.Ci * 4};
    const cuuint32_t box[4] = {(cuuint32_t)G.raw_w, (cuuint32_t)(G.R + 2), (cuuint32_t)kch, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    p.use_tma = D->encode(&xmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float*>(x), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
                      ? 1
                      : 0;
  } else if (can_map && ((size_t)H * W) % 4 == 0) {
    // Rows not 16-byte aligned but planes are: a 3-D map over x viewed as
    // [N][Ci][H * W] and a box of the tile's R + 2 rows packed, plus up to 3
    // elements of alignment shift (the halo columns are zeros in the loaders).
    const int boxw = ((G.R + 2) * W + 3 + 3) / 4 * 4;
    if (boxw <= 256 && kch * boxw * 4 <= G.raw_slot) {
      const cuuint64_t dims[3] = {(cuuint64_t)H * W, (cuuint64_t)M.Ci, (cuuint64_t)N};
      const cuuint64_t strides[2] = {(cuuint64_t)H * W * 4, (cuuint64_t)H * W * M.Ci * 4};
      const cuuint32_t box[3] = {(cuuint32_t)boxw, (cuuint32_t)kch, 1};
      const cuuint32_t estr[3] = {1, 1, 1};
      if (D->encode(&xmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(x), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS) {
        p.use_tma = 1;
        p.plane = 1;
        p.raw_w = boxw;
        p.raw_bytes = kch * boxw * 4;
      }
    }
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[2];
  // programmatic dependent launch: the kernel waits (griddepcontrol.wait) for
  // the previous one before touching its inputs and outputs
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.blockDim = dim3(ring ? flat_threads<true, false>() : flat_threads<false, false>());
  cfg.dynamicSmemBytes = SMEM_ALLOC;
  cfg.stream = stream;
  cudaError_t e;
  if (G.pair) {
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = (unsigned)(2 * G.split);
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
    cfg.gridDim = dim3((unsigned)(G.ntiles * 2 * G.split));
    e = f16 ? cudaLaunchKernelEx(&cfg, ppconv_tcf_kernel<true, true, true>, p, xmap)
            : cudaLaunchKernelEx(&cfg, ppconv_tcf_kernel<true, false, true>, p, xmap);
  } else if (G.split > 1) {
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = (unsigned)G.split;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
    cfg.gridDim = dim3((unsigned)(G.ntiles * G.split));
    e = f16 ? cudaLaunchKernelEx(&cfg, ppconv_tcf_kernel<true, true, false>, p, xmap)
            : cudaLaunchKernelEx(&cfg, ppconv_tcf_kernel<true, false, false>, p, xmap);
  } else {
    cfg.gridDim = dim3((unsigned)std::min(G.ntiles, D->sms));
    e = f16 ? cudaLaunchKernelEx(&cfg, ppconv_tcf_kernel<false, true, false>, p, xmap)
            : cudaLaunchKernelEx(&cfg, ppconv_tcf_kernel<false, false, false>, p, xmap);
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  return PP_OK;
}

}  // namespace

namespace ppc {

int tcf_plan(const TcLayout& T, int N, int H, int W, int flags, int* R, int* S, int maxn) {
  if (T.FB != FB || maxn < 1) return 0;
  DeviceState* D = prepare();
  if (!D) return 0;
  FlatGeo G[16];
  const int n = flat_candidates(N, H, W, T.f16 ? T.nch16 : T.nch, T.nfb, flags & PP_POOL2, true, *D, G,
                                std::min(maxn, 16), T.f16);
  for (int k = 0; k < n; ++k) {
    R[k] = G[k].R;
    S[k] = G[k].code();
  }
  return n;
}

bool tcf_can_run(const TcLayout& T, int N, int H, int W, int flags, int R, int S) {
  if (T.FB != FB) return false;
  DeviceState* D = prepare();
  FlatGeo G;
  return D && flat_pick(N, H, W, T.f16 ? T.nch16 : T.nch, T.nfb, flags & PP_POOL2, *D, R, S, &G, T.f16);
}

void tcf_pinned(const TcLayout& T, int N, int H, int W, int flags, int* R, int* S) {
  const TcState* st = T.state;
  const bool hit = st && st->R > 0 && st->key[0] == N && st->key[1] == H && st->key[2] == W && st->key[3] == flags;
  *R = hit ? st->R : 0;
  *S = hit ? st->S : 0;
}

void tcf_pin(const TcLayout& T, int N, int H, int W, int flags, int R, int S) {
  if (!T.state) return;
  TcState* st = T.state;
  st->key[0] = N;
  st->key[1] = H;
  st->key[2] = W;
  st->key[3] = flags;
  st->R = R;
  st->S = S;
}

}  // namespace ppc
