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
// Per CTA (17 warps, one CTA per SM, persistent over tiles): warps 0-7 stage
// the operands, warp 8 owns the TMEM (two accumulator buffers of 256 columns,
// so one tile's epilogue overlaps the next tile's MMAs) and one of its threads
// issues the MMAs, warps 9-16 are the epilogue; tf32 128-filter tiles add warp
// 17, which produces the weights.  The K loop runs over 8-channel chunks,
// double buffered:
//   * weights for the chunk, 9 taps x {hi, lo} x (FB x 8) in the canonical
//     K-major layout, arrive by bulk async copies whose transaction counts
//     complete on the stage's full barrier with the loaders' arrivals, so the
//     MMA thread waits once per chunk: most tiles copy them whole into the
//     stage; tf32 128-filter tiles copy them in three groups of 3 taps into a
//     ring of group slots, each slot refilled as soon as its MMAs complete;
//   * the input box for the chunk (tile rows + 2, columns + halo, 8 channels;
//     zero fill outside the image is the padding) arrives by a tensor-map copy
//     (per-thread loads when x is not 16-byte aligned or W % 4 != 0), and the
//     loader threads transpose it channel-innermost while splitting hi / lo;
//   * a tap (dy, dx) is the same staged tile with the operand start moved by dy
//     rows and dx pixels (16 bytes per pixel), so no im2col copy exists.
//     Filter-major tiles (ORI_FP) run 3 MMAs per tap and row segment
//     (w_hi x_hi, w_lo x_hi, w_hi x_lo); pixel-major tiles (ORI_PF, ORI_PFR) run
//     2 (x_hi [w_hi | w_lo] as one 2 FB-wide operand, then x_lo w_hi);
//   * tcgen05.commit signals an mbarrier when the chunk's MMAs have read their
//     operands, which frees that stage for the chunk after next.
// fp16 split (layers set to PP_PRECISION_F16X3, F16 instantiations): operands
// held as hi = f16(v) and lo = f16((v - hi) * 2^11) (weights scaled per filter,
// the input per layer, by powers of two), 16-channel chunks (the K of
// kind::f16), w_hi x_hi into one accumulator and w_lo x_hi + w_hi x_lo into a
// second one (pixel-major: the lo half of the merged operand's columns and the
// x_lo MMA; filter-major: the row segment's second TW columns), combined in the
// epilogue as (acc1 + 2^-11 acc2) times the filter's inverse scale; inputs that
// overflow fp16 after scaling (or are not finite) are flagged in the device
// status word.
// Epilogue: bias, +skip, ReLU, 2x2 max pool from tcgen05.ld, stores to each
// filter's original channel.  This kernel has no channel split: layers with
// more than 64 filters on maps at most 128 wide can also run the flat kernel
// (conv_tcf.cu), which splits the chunks of small grids over a cluster.
//
// Every wait on an mbarrier is bounded; on timeout the kernel records an error
// in the layer's device status word and skips the rest of its work.
#include <cooperative_groups.h>
#include <cuda.h>
#include <cuda_runtime.h>

#include <cuda_fp16.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"
#include "tc_ptx.cuh"

namespace {

using namespace ppc_ptx;

constexpr int KC = 8;              // input channels per chunk (MMA K for tf32)
constexpr int NTAP = 9;
constexpr int NCOL = 256;          // TMEM columns of one accumulator buffer
constexpr int NLOAD = 256;         // loader threads (warps 0-7)
constexpr int MMA_WARP = 8;        // warp 8: TMEM owner and MMA issuer
constexpr int EPI_WARP0 = 9;       // warps 9-16: epilogue, two per TMEM lane quadrant
constexpr int NEPI = 256;          // epilogue threads
constexpr int WPROD_WARP = 17;     // warp 17: weight producer (weight-ring instantiations only)
constexpr int NGRP = 3;            // weight-ring groups per chunk
constexpr int TPG = NTAP / NGRP;   // taps per weight-ring group
constexpr int WSL_MAX = 12;        // weight-ring slots at most (4 chunks)
constexpr int LBATCH = 4;          // loader items whose global loads are in flight together
constexpr long WAIT_LIMIT = PP_WAIT_POLLS;  // mbarrier polls before a wait gives up
// dynamic shared memory a CTA may request: 227 KB less room for the kernel's static barriers
constexpr int SMEM_LIMIT = 232448 - 256;

// Orientation of the GEMM on the tensor core.
//   ORI_FP: M = 128 filters, N = TW pixels of one output row (narrow maps)
//   ORI_PF: M = 128 pixels of one output row, N = FB filters (wide maps)
//   ORI_PFR: pixel-major with whole rows flattened: M = 128 staged pixels =
//     128 / TW rows of TW >= W + 2 columns (TW = 16, 32 or 64; the columns
//     past W are computed and dropped), for narrow maps of 64-filter layers
enum { ORI_FP = 0, ORI_PF = 1, ORI_PFR = 2 };

struct TcParams {
  const float* rscale;      // f16: per reordered filter, 1 / (weight scale x input scale)
  float xscale;             // f16: power of two applied to x before the split
  const float* x;
  float* y;
  const float* skip;
  const unsigned char* wt;  // [nfb][nch][9][2][FB x 8] canonical tiles
  const int* perm;          // [Co]
  const float* bias;        // [Co] reordered, or null
  int* status;              // device status word (nonzero after a timed-out wait)
  int N, Ci, Co, H, W;
  int nch, nfb, FB;
  int tiles_x, tiles_y, ntiles;
  int flags;
  int use_tma;  // input tiles by tensor-map copy (W % 4 == 0, aligned x), else per-thread loads
};

// Geometry of one instantiation.  TW pixels per output row segment, FB filters
// per block, R row segments per tile (one accumulator column range each).
template <int ORI, int TW, int FB, bool F16>
struct Geo {
  static_assert(ORI == ORI_FP ? FB == 128 : (ORI == ORI_PF ? TW == 128 : (128 % TW == 0 && FB == 64)),
                "orientation needs a 128-row M side");
  static constexpr int KCH = F16 ? 16 : KC;  // input channels per chunk
  static constexpr int CPH = KCH / 2;        // channels per K half (16 bytes of a pixel's operand row)
  // MRG (pixel-major): the hi and lo weight tiles of a tap are one 2 FB-wide B
  // operand, so x_hi * [w_hi | w_lo] is one N = 2 FB MMA (the lo part lands in
  // accumulator columns FB .. 2 FB - 1 and the epilogue adds the two halves);
  // x_lo * w_hi is an N = FB MMA.  Two MMAs instead of three read the pixel
  // tile twice instead of three times.
  static constexpr bool MRG = ORI != ORI_FP;
  // accumulator columns per row segment (f16 filter-major: a second accumulator of TW columns follows)
  static constexpr int SEGC = ORI == ORI_FP ? (F16 ? 2 * TW : TW) : (MRG ? 2 * FB : FB);
  static constexpr int ACC2 = ORI == ORI_FP ? TW : FB;   // f16: offset of the second accumulator in a segment
  static constexpr int NSEG = NCOL / SEGC;                // MMA row segments per tile
  static constexpr int RSEG = ORI == ORI_PFR ? 128 / TW : 1;  // output rows per segment
  static constexpr int R = NSEG * RSEG;                   // output rows per tile
  static constexpr int BROWS = R + 2, BCOLS = ORI == ORI_PFR ? TW : TW + 2;
  static constexpr int NPIX = BROWS * BCOLS;              // staged input pixels
  // flattened rows: the last segment's operand for the (2, 2) tap runs 2
  // pixels past the staged tile (junk columns only); 16 pixels of slack
  static constexpr int NPIXA = ORI == ORI_PFR ? NPIX + 16 : NPIX;
  static constexpr int IN_HALF = NPIXA * 16;              // one K half (4 channels) of hi or lo
  // hi or lo operand of a chunk; a multiple of 128 bytes, so the lo area (where the input box lands
  // when it has no slot of its own) starts where a tensor-map copy may write
  static constexpr int IN_BYTES = (2 * IN_HALF + 127) / 128 * 128;
  // tensor-map box width: columns c0-4 .. (staged column bc is box column bc + 3),
  // a multiple of 4 so each box row is whole 16-byte units
  static constexpr int RAW_W = (BCOLS + 3 + 3) / 4 * 4;
  static constexpr int RAW = KCH * BROWS * RAW_W * 4;     // box [KCH channels][BROWS][RAW_W], landed in the lo area
  static constexpr int LO_BYTES = IN_BYTES > RAW ? IN_BYTES : RAW;
  static constexpr int W_TILE = FB * KC * 4;              // one tap, one of hi / lo (FB x 8 fp32 or FB x 16 f16)
  static constexpr int W_BYTES = NTAP * 2 * W_TILE;       // weights of one chunk
  // WR: the weights sit in a ring of WSL groups of TPG taps (GRP bytes each, two
  // chunks at least, up to WSL_MAX as shared memory allows) ahead of the two
  // input operand stages, filled by the producer warp; a group's slot is
  // refilled as soon as its MMAs complete.  Used by the tf32 128-filter tiles,
  // where it measured faster; the others (the 64-filter tiles are shared-memory
  // bound at 9 taps of N = 128 + 64 MMAs) keep each chunk's weights in its
  // operand stage, copied whole by the loaders' thread 0 once the stage is free,
  // and run without the producer warp (an 18th warp, even idle, measured slower
  // there).
  static constexpr bool WR = FB == 128 && !F16;
  static constexpr int NTHREADS = WR ? 576 : 544;
  static constexpr int GRP = W_BYTES / NGRP;
  // SEP: the raw boxes get a ring of their own (NRAW = two slots, or one when
  // two do not fit), so the copy for chunk g + NRAW starts as soon as chunk g's
  // box has been read instead of waiting for the MMAs that read the stage; used
  // whenever it fits in shared memory.  The two raw_full barriers alternate
  // between chunks whatever the slot count.
  static constexpr int STAGE_SEP = W_BYTES + 2 * IN_BYTES;
  static constexpr int NRAW = 2 * STAGE_SEP + 2 * RAW + 1024 <= SMEM_LIMIT ? 2
                              : (2 * STAGE_SEP + RAW + 1024 <= SMEM_LIMIT ? 1 : 0);
  static constexpr bool SEP = NRAW > 0;
  static constexpr int XSTAGE = SEP ? 2 * IN_BYTES : IN_BYTES + LO_BYTES;  // input operands (hi, lo) of a stage
  static constexpr int STAGE = WR ? XSTAGE : W_BYTES + XSTAGE;  // stage stride; without WR its weights come first
  static constexpr int WSL_FIT = (SMEM_LIMIT - 1024 - 2 * XSTAGE - NRAW * RAW) / GRP;
  static constexpr int WSL = WR ? (WSL_FIT < WSL_MAX ? WSL_FIT : WSL_MAX) : 0;
  static constexpr int XOFF = WR ? WSL * GRP : W_BYTES;  // stage s's input operands at XOFF + s * STAGE
  static constexpr int RAW_OFF = WR ? XOFF + 2 * STAGE : 2 * STAGE;  // raw slots (SEP)
  static constexpr int SMEM_ALLOC = RAW_OFF + NRAW * RAW + 1024;
  static constexpr int ITEMS = (2 * NPIX + NLOAD - 1) / NLOAD;  // (K half, pixel) items per loader thread
  static_assert(SMEM_ALLOC <= SMEM_LIMIT, "shared memory plan");
  static_assert(W_BYTES % 128 == 0 && IN_BYTES % 128 == 0 && RAW % 128 == 0 && STAGE % 128 == 0 && GRP % 128 == 0,
                "tensor-map copies need 128-byte aligned shared-memory destinations");
  static_assert(!WR || WSL >= 2 * NGRP, "the weight ring holds two chunks at least");
  static constexpr uint32_t IDESC = F16 ? (ORI == ORI_FP ? idesc_f16(128, TW) : idesc_f16(128, FB))
                                        : (ORI == ORI_FP ? idesc_tf32(128, TW) : idesc_tf32(128, FB));
  static constexpr uint32_t IDESC2 = F16 ? idesc_f16(128, 2 * FB) : idesc_tf32(128, 2 * FB);  // MRG: [w_hi | w_lo]
  static constexpr int WLBO = 2 * FB * 16;  // weights: bytes between K halves (hi and lo rows of a tap in each)
};

struct Tile {
  int n, r0, c0, fb;
};
__device__ __forceinline__ Tile tile_of(const TcParams& p, int t, int R, int TW) {
  Tile T;
  T.fb = t % p.nfb;
  t /= p.nfb;
  const int tx = t % p.tiles_x;
  t /= p.tiles_x;
  const int ty = t % p.tiles_y;
  T.n = t / p.tiles_y;
  T.r0 = ty * R;
  T.c0 = tx * TW;
  return T;
}

template <int ORI, int TW, int FB, bool F16>
__global__ void __launch_bounds__(Geo<ORI, TW, FB, F16>::NTHREADS, 1) ppconv_tc_kernel(const TcParams p, const __grid_constant__ CUtensorMap xmap) {
  using G = Geo<ORI, TW, FB, F16>;
  // slots of the box ring (its uses sit behind G::SEP; 1 keeps the modulo defined where the ring is absent)
  constexpr int RING = G::NRAW > 0 ? G::NRAW : 1;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // Offset from the shared array itself (not an integer round trip), so the
  // compiler keeps every access below in the shared state space.
  unsigned char* smem = smem_raw + ((1024u - (su32(smem_raw) & 1023u)) & 1023u);
  __shared__ __align__(8) uint64_t full[2], empty[2], acc_full[2], acc_empty[2], done_bar, raw_full[2];
  __shared__ __align__(8) uint64_t wempty[G::WR ? WSL_MAX : 1];  // a weight-ring slot has been read by its MMAs
  __shared__ uint32_t tmem_s;
  __shared__ volatile int abort_s;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // Bounded wait that gives up early once another role has aborted.
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
      // full: every loader thread's operand stores plus the chunk's weight
      // copies (one more arrival each, with its bytes: the whole chunk, or its
      // NGRP ring groups), so the MMA thread waits once per chunk
      mbar_init(su32(&full[s]), NLOAD + (G::WR ? NGRP : 1));
      mbar_init(su32(&empty[s]), 1);
      mbar_init(su32(&acc_full[s]), 1);
      mbar_init(su32(&acc_empty[s]), NEPI);
      mbar_init(su32(&raw_full[s]), 1);
    }
    mbar_init(su32(&done_bar), 1);
    if (G::WR)
      for (int k = 0; k < WSL_MAX; ++k) mbar_init(su32(&wempty[k]), 1);
    abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == MMA_WARP) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tmem_s)),
                 "n"(2 * NCOL));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  const uint32_t tmem = tmem_s;
  const int nmine = p.ntiles > (int)blockIdx.x ? (p.ntiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;

  if (warp < MMA_WARP) {
    // ------------------------------------------------------------ loaders
    // Thread 0 issues the copies: the weights (bulk, on full[s]) unless the
    // producer warp does (WR) and, with a tensor map, the raw input box (on
    // raw_full); all loader threads then transpose the box into the hi / lo
    // operand tiles and arrive on full[s].
    const int nall = nmine * p.nch;  // chunks of this CTA
    auto issue_raw = [&](int gg, unsigned char* dst) {  // thread 0 only
      const int i = gg / p.nch, c = gg - i * p.nch;
      const Tile T = tile_of(p, (int)blockIdx.x + i * (int)gridDim.x, G::R, TW);
      // box [8 channels][rows r0-1 ..][columns c0-4 ..]; outside the image the
      // copy fills zeros, which is the convolution's zero padding
      mbar_arrive_expect_tx(su32(&raw_full[gg & 1]), G::RAW);
      asm volatile(
          "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, "
          "%4, %5}], [%6];" ::"r"(su32(dst)),
          "l"(reinterpret_cast<uint64_t>(&xmap)), "r"(T.c0 - 4), "r"(T.r0 - 1), "r"(c * G::KCH), "r"(T.n),
          "r"(su32(&raw_full[gg & 1]))
          : "memory");
    };
    int raw_issued = 0, w_issued = 0;  // thread 0's counts of issued copies
    // Weights of chunk gg into stage s (thread 0).
    auto issue_w = [&](int gg, int s) {
      const Tile T = tile_of(p, (int)blockIdx.x + (gg / p.nch) * (int)gridDim.x, G::R, TW);
      const unsigned char* src = p.wt + ((size_t)T.fb * p.nch + gg % p.nch) * G::W_BYTES;
      mbar_arrive_expect_tx(su32(&full[s]), G::W_BYTES);
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
              su32(smem + s * G::STAGE)),
          "l"(src), "r"(G::W_BYTES), "r"(su32(&full[s]))
          : "memory");
    };
    // The weights do not depend on the previous kernel in the stream: the first
    // two chunks' copies start before waiting for it (programmatic dependent
    // launch), everything that reads x comes after the wait.
    if (!G::WR && tid == 0)
      for (; w_issued < 2 && w_issued < nall; ++w_issued) issue_w(w_issued, w_issued);
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (tid == 0 && p.use_tma && G::SEP)
      for (; raw_issued < G::NRAW && raw_issued < nall; ++raw_issued)
        issue_raw(raw_issued, smem + G::RAW_OFF + raw_issued * G::RAW);
    int g = 0;  // chunk sequence number of this CTA
    bool stop = false;  // identical in every loader thread (decided by loader_any)
    uint32_t range_bad = 0;  // f16: nonzero once an input is non-finite or overflows fp16 after scaling
    for (int i = 0; i < nmine && !stop; ++i) {
      const Tile T = tile_of(p, (int)blockIdx.x + i * (int)gridDim.x, G::R, TW);
      const float* xb = p.x + (size_t)T.n * p.Ci * p.H * p.W;
      for (int c = 0; c < p.nch; ++c, ++g) {
        const int s = g & 1, use = g >> 1;
        // f16 (and the tf32 weight-ring tiles) with a box ring: the box of this chunk has a slot of its own and
        // lands ahead of time, so it is read and split into registers before the stage is free (while the
        // MMAs of the two previous chunks still read it); only the stores wait for the stage.
        constexpr bool EARLY = (F16 || G::WR) && G::SEP;
        constexpr int EI = EARLY ? G::ITEMS : 1;
        uint4 hreg[EI], lreg[EI];
        const bool early = EARLY && p.use_tma;
        if (early) {
          if (group_any<NLOAD>(!wait(&raw_full[g & 1], (uint32_t)((g >> 1) & 1)))) {
            stop = true;
            break;
          }
          const float* raw = reinterpret_cast<const float*>(smem + G::RAW_OFF + (g % RING) * G::RAW);
#pragma unroll
          for (int b = 0; b < EI; ++b) {
            const int it = b * NLOAD + tid;
            if (it < 2 * G::NPIX) {
              const int kh = it >= G::NPIX ? 1 : 0;
              const int pix = it - kh * G::NPIX;
              const int br = pix / G::BCOLS, bc = pix - br * G::BCOLS;
              float u[G::CPH];
#pragma unroll
              for (int k = 0; k < G::CPH; ++k) u[k] = raw[((kh * G::CPH + k) * G::BROWS + br) * G::RAW_W + bc + 3];
              if constexpr (F16) {
                range_bad |= split_f16x8(u, p.xscale, hreg[b], lreg[b]);
              } else {
                // tf32 split: hi keeps the top 10 mantissa bits (exact in tf32), lo = v - hi (exact in fp32)
                uint32_t hb[4], lb[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  hb[k] = __float_as_uint(u[k]) & 0xFFFFE000u;
                  lb[k] = __float_as_uint(u[k] - __uint_as_float(hb[k]));
                }
                hreg[b] = make_uint4(hb[0], hb[1], hb[2], hb[3]);
                lreg[b] = make_uint4(lb[0], lb[1], lb[2], lb[3]);
              }
            }
          }
          // the slot is rewritten next by a tensor-map copy: reads ordered before it, then released
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          group_sync<NLOAD>();
          if (tid == 0 && raw_issued < nall && raw_issued == g + G::NRAW) {
            issue_raw(raw_issued, smem + G::RAW_OFF + (raw_issued % RING) * G::RAW);
            ++raw_issued;
          }
        }
        if (group_any<NLOAD>(use > 0 && !wait(&empty[s], (uint32_t)((use - 1) & 1)))) {
          stop = true;
          break;
        }
        unsigned char* st = smem + G::XOFF + s * G::STAGE;
        float4* hi = reinterpret_cast<float4*>(st);
        float4* lo = reinterpret_cast<float4*>(st + G::IN_BYTES);
        if (tid == 0) {
          if (!G::WR && g >= 2) {
            issue_w(g, s);
            ++w_issued;
          }
          if (p.use_tma && !G::SEP) {
            issue_raw(g, reinterpret_cast<unsigned char*>(lo));
            ++raw_issued;
          }
        }
        const int ch0 = c * G::KCH;
        if (early) {
#pragma unroll
          for (int b = 0; b < EI; ++b) {
            const int it = b * NLOAD + tid;
            if (it < 2 * G::NPIX) {
              const int dst = it + (it >= G::NPIX ? G::NPIXA - G::NPIX : 0);  // K halves NPIXA apart
              reinterpret_cast<uint4*>(hi)[dst] = hreg[b];
              reinterpret_cast<uint4*>(lo)[dst] = lreg[b];
            }
          }
        } else if (p.use_tma) {
          if (group_any<NLOAD>(!wait(&raw_full[g & 1], (uint32_t)((g >> 1) & 1)))) {
            stop = true;
            break;
          }
          const float* raw = G::SEP ? reinterpret_cast<const float*>(smem + G::RAW_OFF + (g % RING) * G::RAW)
                                    : reinterpret_cast<const float*>(lo);
          float v[G::ITEMS][G::CPH];
#pragma unroll
          for (int b = 0; b < G::ITEMS; ++b) {
            const int it = b * NLOAD + tid;
            const int kh = it >= G::NPIX ? 1 : 0;
            const int pix = it - kh * G::NPIX;
            const int br = pix / G::BCOLS, bc = pix - br * G::BCOLS;
#pragma unroll
            for (int k = 0; k < G::CPH; ++k)
              v[b][k] = it < 2 * G::NPIX ? raw[((kh * G::CPH + k) * G::BROWS + br) * G::RAW_W + bc + 3] : 0.f;
          }
          // The raw slot is rewritten next by a tensor-map copy (async proxy):
          // each thread orders its generic-proxy reads of the slot before that
          // copy with a proxy fence, then the loader barrier lets thread 0 issue it.
          if (G::SEP) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          group_sync<NLOAD>();  // every raw value is in registers before its slot is reused
          if (G::SEP && tid == 0 && raw_issued < nall && raw_issued == g + G::NRAW) {
            issue_raw(raw_issued, smem + G::RAW_OFF + (raw_issued % RING) * G::RAW);
            ++raw_issued;
          }
#pragma unroll
          for (int b = 0; b < G::ITEMS; ++b) {
            const int it = b * NLOAD + tid;
            if (it < 2 * G::NPIX) {
              const int dst = it + (it >= G::NPIX ? G::NPIXA - G::NPIX : 0);  // K halves NPIXA apart
              if constexpr (F16) {
                uint4 h, l;
                range_bad |= split_f16x8(&v[b][0], p.xscale, h, l);
                reinterpret_cast<uint4*>(hi)[dst] = h;
                reinterpret_cast<uint4*>(lo)[dst] = l;
              } else {
                float4 h;
                h.x = __uint_as_float(__float_as_uint(v[b][0]) & 0xFFFFE000u);
                h.y = __uint_as_float(__float_as_uint(v[b][1]) & 0xFFFFE000u);
                h.z = __uint_as_float(__float_as_uint(v[b][2]) & 0xFFFFE000u);
                h.w = __uint_as_float(__float_as_uint(v[b][3]) & 0xFFFFE000u);
                hi[dst] = h;
                lo[dst] = make_float4(v[b][0] - h.x, v[b][1] - h.y, v[b][2] - h.z, v[b][3] - h.w);
              }
            }
          }
        } else {
          // Items in batches of LBATCH per thread: all global loads of a batch
          // are issued before any is used, so their latencies overlap.
          constexpr int LB = F16 ? LBATCH / 2 : LBATCH;  // f16 items carry 8 values: the same loads in flight
          for (int base = 0; base < 2 * G::NPIX; base += NLOAD * LB) {
            float v[LB][G::CPH];
#pragma unroll
            for (int b = 0; b < LB; ++b) {
              const int it = base + b * NLOAD + tid;
              const int kh = it >= G::NPIX ? 1 : 0;
              const int pix = it - kh * G::NPIX;
              const int br = pix / G::BCOLS, bc = pix - br * G::BCOLS;
              const int r = T.r0 - 1 + br, cc = T.c0 - 1 + bc;
              const bool inside = it < 2 * G::NPIX && (unsigned)r < (unsigned)p.H && (unsigned)cc < (unsigned)p.W;
#pragma unroll
              for (int k = 0; k < G::CPH; ++k) {
                const int ch = ch0 + kh * G::CPH + k;
                v[b][k] = (inside && ch < p.Ci) ? __ldg(xb + ((size_t)ch * p.H + r) * p.W + cc) : 0.f;
              }
            }
#pragma unroll
            for (int b = 0; b < LB; ++b) {
              const int it = base + b * NLOAD + tid;
              if (it < 2 * G::NPIX) {
                const int dst = it + (it >= G::NPIX ? G::NPIXA - G::NPIX : 0);
                if constexpr (F16) {
                  uint4 h, l;
                  range_bad |= split_f16x8(&v[b][0], p.xscale, h, l);
                  reinterpret_cast<uint4*>(hi)[dst] = h;
                  reinterpret_cast<uint4*>(lo)[dst] = l;
                } else {
                  float4 h;
                  h.x = __uint_as_float(__float_as_uint(v[b][0]) & 0xFFFFE000u);
                  h.y = __uint_as_float(__float_as_uint(v[b][1]) & 0xFFFFE000u);
                  h.z = __uint_as_float(__float_as_uint(v[b][2]) & 0xFFFFE000u);
                  h.w = __uint_as_float(__float_as_uint(v[b][3]) & 0xFFFFE000u);
                  hi[dst] = h;
                  lo[dst] = make_float4(v[b][0] - h.x, v[b][1] - h.y, v[b][2] - h.z, v[b][3] - h.w);
                }
              }
            }
          }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive(su32(&full[s]));
      }
    }
    if (F16 && range_bad != 0) atomicOr(p.status, ppc::kStatusF16Range);
    if (tid == 0) {
      // No copy may still be writing shared memory when the CTA exits: after an
      // early stop, wait (bounded) for the last copies of each kind to land.
      // (A stage's barrier may then lack loader arrivals and never complete;
      // the bounded wait outlasts any copy still in flight.)
      for (int gg = raw_issued - 2; gg < raw_issued; ++gg)
        if (gg >= 0)
          for (long k = 0; k < WAIT_LIMIT && !mbar_try(su32(&raw_full[gg & 1]), (uint32_t)((gg >> 1) & 1)); ++k) {
          }
      for (int gg = w_issued - 2; gg < w_issued; ++gg)
        if (gg >= 0)
          for (long k = 0; k < WAIT_LIMIT && !mbar_try(su32(&full[gg & 1]), (uint32_t)((gg >> 1) & 1)); ++k) {
          }
    }
  } else if (warp == MMA_WARP) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int g = 0, wslot = 0;  // chunk count and (WR) the weight-ring slot of the next group
      for (int i = 0; i < nmine && !abort_s; ++i) {
        const int b = i & 1, ub = i >> 1;
        if (ub > 0 && !wait(&acc_empty[b], (uint32_t)((ub - 1) & 1))) break;
        tm_fence_after();
        const uint32_t dbase = tmem + (uint32_t)(b * NCOL);
        bool okc = true;
        for (int c = 0; c < p.nch; ++c, ++g) {
          const int s = g & 1, use = g >> 1;
          if (!wait(&full[s], (uint32_t)(use & 1))) {
            okc = false;
            break;
          }
          tm_fence_after();
          const unsigned char* st = smem + G::XOFF + s * G::STAGE;
          // Descriptors hold address / 16 in their low 14 bits and every operand
          // lies below 256 KB, so moving an operand is one add to the descriptor.
          const uint64_t w0 = smem_desc(su32(smem + s * G::STAGE), G::WLBO);  // without WR
          const uint64_t xh0 = smem_desc(su32(st), G::IN_HALF);
          const uint64_t xl0 = smem_desc(su32(st + G::IN_BYTES), G::IN_HALF);
          int gs[NGRP];  // WR: the chunk's weight groups, consecutive slots of the ring
#pragma unroll
          for (int k = 0; k < NGRP; ++k) {
            gs[k] = wslot;
            if (G::WR) wslot = wslot + 1 == G::WSL ? 0 : wslot + 1;
          }
          const uint32_t acc0 = c == 0 ? 0u : 1u;  // the tile's first chunk overwrites the accumulators
#pragma unroll
          for (int t = 0; t < NTAP; ++t) {
            const int dy = t / 3, dx = t % 3;
            const uint64_t whi = G::WR ? smem_desc(su32(smem + gs[t / TPG] * G::GRP + (t % TPG) * 2 * G::W_TILE), G::WLBO)
                                       : w0 + (uint64_t)(t * 2 * G::W_TILE / 16);
            const uint64_t wlo = whi + (uint64_t)FB;  // lo rows follow the hi rows: FB rows of 16 bytes
#pragma unroll(G::NSEG <= 8 ? G::NSEG : 4)
            for (int rr = 0; rr < G::NSEG; ++rr) {
              const uint64_t off = (uint64_t)((rr * G::RSEG + dy) * G::BCOLS + dx);  // pixels of 16 bytes
              const uint64_t xh = xh0 + off, xl = xl0 + off;
              const uint32_t d = dbase + (uint32_t)(rr * G::SEGC);
              if (F16) {
                // acc1 += w_hi x_hi; acc2 += w_lo x_hi + w_hi x_lo (lo parts scaled by 2^11)
                if (ORI == ORI_FP) {
                  mma_f16(d, whi, xh, G::IDESC, t == 0 ? acc0 : 1u);
                  mma_f16(d + G::ACC2, wlo, xh, G::IDESC, t == 0 ? acc0 : 1u);
                  mma_f16(d + G::ACC2, whi, xl, G::IDESC, 1u);
                } else {
                  mma_f16(d, xh, whi, G::IDESC2, t == 0 ? acc0 : 1u);  // [acc1 | acc2] += x_hi [w_hi | w_lo]
                  mma_f16(d + G::ACC2, xl, whi, G::IDESC, 1u);
                }
              } else if (ORI == ORI_FP) {
                mma_tf32(d, whi, xh, G::IDESC, t == 0 ? acc0 : 1u);
                mma_tf32(d, wlo, xh, G::IDESC, 1u);
                mma_tf32(d, whi, xl, G::IDESC, 1u);
              } else if (G::MRG) {
                mma_tf32(d, xh, whi, G::IDESC2, t == 0 ? acc0 : 1u);
                mma_tf32(d, xl, whi, G::IDESC, 1u);
              } else {
                mma_tf32(d, xh, whi, G::IDESC, t == 0 ? acc0 : 1u);
                mma_tf32(d, xh, wlo, G::IDESC, 1u);
                mma_tf32(d, xl, whi, G::IDESC, 1u);
              }
            }
            if (G::WR && t % TPG == TPG - 1) mma_commit(su32(&wempty[gs[t / TPG]]));  // slot free once these complete
          }
          mma_commit(su32(&empty[s]));
        }
        if (!okc) break;
        mma_commit(su32(&acc_full[b]));
      }
      // every MMA issued by this thread is complete before TMEM is released
      // the next kernel in the stream may start its prologue (it waits for this
      // grid to complete before it reads anything this grid writes)
      asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
      mma_commit(su32(&done_bar));
      wait(&done_bar, 0u);
    }
    __syncwarp();
  } else if (warp == WPROD_WARP) {
    // ------------------------------------------------------------ weight producer (WR)
    // A chunk's weights are NGRP groups of TPG tap tiles, copied into the ring of
    // G::WSL slots.  A group is copied as soon as the MMAs of the group that held
    // its slot before have completed; the chunk's copies arrive (with their bytes)
    // on the stage's full barrier, and those of chunk g go out only after that
    // barrier's previous phase (chunk g - 2) has completed.
    if (G::WR && lane == 0) {
      const int nall = nmine * p.nch;
      int slot = 0, use = 0, issued = 0;  // ring position, its round, groups issued
      bool ok = true;
      for (int gg = 0; gg < nall && ok; ++gg) {
        const int s = gg & 1;
        if (gg >= 2) ok = wait(&full[s], (uint32_t)(((gg - 2) >> 1) & 1));
        const Tile T = tile_of(p, (int)blockIdx.x + (gg / p.nch) * (int)gridDim.x, G::R, TW);
        const unsigned char* src = p.wt + ((size_t)T.fb * p.nch + gg % p.nch) * G::W_BYTES;
        for (int k = 0; k < NGRP && ok; ++k) {
          if (use > 0) ok = wait(&wempty[slot], (uint32_t)((use - 1) & 1));
          if (!ok) break;
          mbar_arrive_expect_tx(su32(&full[s]), G::GRP);
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                  su32(smem + slot * G::GRP)),
              "l"(src + (size_t)k * G::GRP), "r"(G::GRP), "r"(su32(&full[s]))
              : "memory");
          ++issued;
          if (++slot == G::WSL) {
            slot = 0;
            ++use;
          }
        }
      }
      // No copy may still be writing shared memory when the CTA exits: wait
      // (bounded) for the last two chunks' barriers (after a timeout a barrier
      // may lack loader arrivals; the bounded wait outlasts any copy in flight).
      const int last = (issued + NGRP - 1) / NGRP;
      for (int gg = last > 2 ? last - 2 : 0; gg < last; ++gg)
        for (long w = 0; w < WAIT_LIMIT && !mbar_try(su32(&full[gg & 1]), (uint32_t)((gg >> 1) & 1)); ++w) {
        }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;                 // TMEM lane quadrant of this warp
    const int half = (warp - EPI_WARP0) >> 2;  // the two warps of a quadrant split the columns
    const bool pool = p.flags & PP_POOL2;
    for (int i = 0; i < nmine; ++i) {
      const int b = i & 1, ub = i >> 1;
      // the whole warp leaves together: its TMEM loads and shuffles are warp-collective
      if (!__all_sync(0xffffffffu, wait(&acc_full[b], (uint32_t)(ub & 1)))) break;
      tm_fence_after();
      const Tile T = tile_of(p, (int)blockIdx.x + i * (int)gridDim.x, G::R, TW);
      const uint32_t lanebase = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * NCOL);
      if (ORI == ORI_FP) {
        // lane = filter; columns = pixels of row segment rr
        const int jr = T.fb * FB + 32 * q + lane;
        const bool valid = jr < p.Co;
        const int o = valid ? __ldg(p.perm + jr) : 0;
        const float bs = (valid && p.bias) ? __ldg(p.bias + jr) : 0.f;
        const float rs = F16 ? __ldg(p.rscale + jr) : 1.f;  // the layout holds nfb x FB entries
        const int step = pool ? 2 : 1;
        for (int rr = half * step; rr < G::R; rr += 2 * step) {
          const int row = T.r0 + rr;
          for (int cc = 0; cc < TW; cc += 16) {
            float a[16], bb[16];
            tm_ld16(lanebase + (uint32_t)(rr * G::SEGC + cc), a);
            if (pool) tm_ld16(lanebase + (uint32_t)((rr + 1) * G::SEGC + cc), bb);
            if constexpr (F16) {
              float a2[16], bb2[16];
              tm_ld16(lanebase + (uint32_t)(rr * G::SEGC + G::ACC2 + cc), a2);
              if (pool) tm_ld16(lanebase + (uint32_t)((rr + 1) * G::SEGC + G::ACC2 + cc), bb2);
              tm_wait_ld();
#pragma unroll
              for (int k = 0; k < 16; ++k) {
                a[k] = fmaf(a2[k], 0x1p-11f, a[k]) * rs;
                if (pool) bb[k] = fmaf(bb2[k], 0x1p-11f, bb[k]) * rs;
              }
            }
            tm_wait_ld();
            // the TMEM loads above are warp-collective; lanes without an output skip only the stores
            if (valid && row < p.H) {
            const int col = T.c0 + cc;
            const float* sk0 = (p.flags & PP_ADD_SKIP) ? p.skip + (((size_t)T.n * p.Co + o) * p.H + row) * p.W : nullptr;
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              a[k] += bs;
              if (sk0 && col + k < p.W) a[k] += __ldg(sk0 + col + k);
              if (p.flags & PP_RELU) a[k] = fmaxf(a[k], 0.f);
            }
            if (!pool) {
              float* yo = p.y + (((size_t)T.n * p.Co + o) * p.H + row) * p.W;
              if (col + 16 <= p.W && (p.W & 3) == 0) {
#pragma unroll
                for (int k = 0; k < 16; k += 4)
                  *reinterpret_cast<float4*>(yo + col + k) = make_float4(a[k], a[k + 1], a[k + 2], a[k + 3]);
              } else {
#pragma unroll
                for (int k = 0; k < 16; ++k)
                  if (col + k < p.W) yo[col + k] = a[k];
              }
            } else {
              const float* sk1 = sk0 ? sk0 + p.W : nullptr;
#pragma unroll
              for (int k = 0; k < 16; ++k) {
                bb[k] += bs;
                if (sk1 && col + k < p.W) bb[k] += __ldg(sk1 + col + k);
                if (p.flags & PP_RELU) bb[k] = fmaxf(bb[k], 0.f);
              }
              const int Ho = p.H / 2, Wo = p.W / 2;
              float* yo = p.y + (((size_t)T.n * p.Co + o) * Ho + (row >> 1)) * Wo;
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const int pc = (col >> 1) + k;
                if (pc < Wo) yo[pc] = fmaxf(fmaxf(a[2 * k], a[2 * k + 1]), fmaxf(bb[2 * k], bb[2 * k + 1]));
              }
            }
            }
          }
        }
      } else {
        // lane = pixel 32q + lane of row segment rr; columns = filters (this
        // warp: half of them).  The block's filter indices and biases sit in
        // registers spread over the lanes (filter j in lane j % 32 of register
        // j / 32) and are fetched by shuffle; output offsets within an image
        // fit in 32 bits (checked on the host), so an output costs a shuffle,
        // a multiply-add and a store.
        constexpr int NR = FB / 32;
        int pm[NR];
        float bv[NR], rv[NR];
#pragma unroll
        for (int k = 0; k < NR; ++k) {
          const int jr = T.fb * FB + 32 * k + lane;
          pm[k] = jr < p.Co ? __ldg(p.perm + jr) : -1;
          bv[k] = (jr < p.Co && p.bias) ? __ldg(p.bias + jr) : 0.f;
          rv[k] = F16 ? __ldg(p.rscale + jr) : 1.f;  // f16: inverse scale (nfb x FB entries)
        }
        // flattened rows (ORI_PFR): lane j of a segment is row j / TW, column j % TW of it
        const int jl = 32 * q + lane;
        const int rsub = ORI == ORI_PFR ? jl / TW : 0;
        const int col = ORI == ORI_PFR ? jl % TW : T.c0 + jl;
        const int Ho = p.H / 2, Wo = p.W / 2;
        const int HW = p.H * p.W, HWo = Ho * Wo;
        const size_t nco = (size_t)T.n * p.Co;
        float* ybase = p.y + nco * (size_t)(pool ? HWo : HW);
        const float* sbase = (p.flags & PP_ADD_SKIP) ? p.skip + nco * (size_t)HW : nullptr;
        for (int rr = 0; rr < G::NSEG; rr += (pool ? 2 : 1)) {
          const int row = T.r0 + rr * G::RSEG + rsub;
          const bool in0 = row < p.H && col < p.W;
          const int roff = row * p.W + col;
          const int poff = (row >> 1) * Wo + (col >> 1);
#pragma unroll
          for (int jj = half * (FB / 2); jj < (half + 1) * (FB / 2); jj += 16) {
            float a[16], bb[16];
            if constexpr (F16) {
              // (acc1 + 2^-11 acc2) times the filter's inverse scale, one row at a time (fewer live
              // registers); every lane shuffles
              auto combined = [&](int seg, float (&v)[16]) {
                float v2[16];
                tm_ld16(lanebase + (uint32_t)(seg * G::SEGC + jj), v);
                tm_ld16(lanebase + (uint32_t)(seg * G::SEGC + FB + jj), v2);
                tm_wait_ld();
#pragma unroll
                for (int k = 0; k < 16; ++k)
                  v[k] = fmaf(v2[k], 0x1p-11f, v[k]) * __shfl_sync(0xffffffffu, rv[(jj + k) >> 5], (jj + k) & 31);
              };
              combined(rr, a);
              if (pool) combined(rr + 1, bb);
            } else {
            tm_ld16(lanebase + (uint32_t)(rr * G::SEGC + jj), a);
            if (pool) tm_ld16(lanebase + (uint32_t)((rr + 1) * G::SEGC + jj), bb);
            if (G::MRG) {
              float a2[16], bb2[16];
              tm_ld16(lanebase + (uint32_t)(rr * G::SEGC + FB + jj), a2);
              if (pool) tm_ld16(lanebase + (uint32_t)((rr + 1) * G::SEGC + FB + jj), bb2);
              tm_wait_ld();
#pragma unroll
              for (int k = 0; k < 16; ++k) {
                a[k] += a2[k];
                if (pool) bb[k] += bb2[k];
              }
            }
            tm_wait_ld();
            }
            // residual (no pool): the 16 skip values are added in a pass of their
            // own, with no store between the loads, so their latencies overlap.
            // The condition is warp-uniform (kernel arguments): every lane takes
            // part in the shuffles.  Every lane loads (lanes without an output
            // from the tensor's first element) and masks the value, so the 16
            // loads are unconditional and independent.
            if (sbase && !pool) {
#pragma unroll
              for (int k0 = 0; k0 < 16; k0 += 8) {
                float sv[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                  const int o = __shfl_sync(0xffffffffu, pm[(jj + k0 + k) >> 5], (jj + k0 + k) & 31);
                  const bool use = o >= 0 && in0;
                  sv[k] = __ldg(sbase + (use ? o * HW + roff : 0));
                  sv[k] = use ? sv[k] : 0.f;
                }
#pragma unroll
                for (int k = 0; k < 8; ++k) a[k0 + k] += sv[k];
              }
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int j = jj + k;
              const int o = __shfl_sync(0xffffffffu, pm[j >> 5], j & 31);
              const float bs = __shfl_sync(0xffffffffu, bv[j >> 5], j & 31);
              if (o < 0) continue;  // past the last filter: the same for every lane
              float v = a[k] + bs;
              if (sbase && pool && in0) v += __ldg(sbase + o * HW + roff);
              if (p.flags & PP_RELU) v = fmaxf(v, 0.f);
              if (!pool) {
                if (in0) ybase[o * HW + roff] = v;
              } else {
                float u = bb[k] + bs;
                if (sbase && in0) u += __ldg(sbase + o * HW + roff + p.W);
                if (p.flags & PP_RELU) u = fmaxf(u, 0.f);
                const float m = fmaxf(v, u);
                const float m2 = __shfl_down_sync(0xffffffffu, m, 1);
                if (((col & 1) == 0) && in0) ybase[o * HWo + poff] = fmaxf(m, m2);
              }
            }
          }
        }
      }
      tm_fence_before();
      mbar_arrive(su32(&acc_empty[b]));
    }
  }

  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (warp == MMA_WARP)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(2 * NCOL));
}

template <int ORI, int TW, int FB>
cudaError_t set_attr() {
  cudaError_t e = cudaFuncSetAttribute(ppconv_tc_kernel<ORI, TW, FB, false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, Geo<ORI, TW, FB, false>::SMEM_ALLOC);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(ppconv_tc_kernel<ORI, TW, FB, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              Geo<ORI, TW, FB, true>::SMEM_ALLOC);
}

ppc::DeviceOnce g_attr_once;

cudaError_t prepare() {
  return g_attr_once.run([](int) {
    cudaError_t e;
    if ((e = set_attr<ORI_FP, 16, 128>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_FP, 32, 128>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_FP, 64, 128>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_FP, 128, 128>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_PF, 128, 64>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_PF, 128, 128>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_PFR, 16, 64>()) != cudaSuccess) return e;
    if ((e = set_attr<ORI_PFR, 32, 64>()) != cudaSuccess) return e;
    return set_attr<ORI_PFR, 64, 64>();
  });
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
// cuTensorMapEncodeTiled from the driver (null: every launch uses per-thread loads)
std::atomic<EncodeTiledFn> g_encode{nullptr};
ppc::DeviceOnce g_encode_once;

// 4-D map over x viewed as [N][Ci][H][W] (W innermost), box [1][KCH][R+2][TW+8].
template <int ORI, int TW, int FB, bool F16>
bool make_xmap(CUtensorMap* m, const TcParams& p) {
  using G = Geo<ORI, TW, FB, F16>;
  const EncodeTiledFn encode = g_encode.load(std::memory_order_acquire);
  if (!encode) return false;
  const cuuint64_t dims[4] = {(cuuint64_t)p.W, (cuuint64_t)p.H, (cuuint64_t)p.Ci, (cuuint64_t)p.N};
  const cuuint64_t strides[3] = {(cuuint64_t)p.W * 4, (cuuint64_t)p.W * p.H * 4, (cuuint64_t)p.W * p.H * p.Ci * 4};
  const cuuint32_t box[4] = {(cuuint32_t)G::RAW_W, (cuuint32_t)G::BROWS, (cuuint32_t)G::KCH, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float*>(p.x), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int ORI, int TW, int FB, bool F16>
cudaError_t launch_one(const TcParams& p0, cudaStream_t stream, int sms) {
  using G = Geo<ORI, TW, FB, F16>;
  TcParams p = p0;
  if ((p.flags & PP_POOL2) && (G::R & 1)) return cudaErrorInvalidValue;  // pooling reads row pairs of a tile
  p.tiles_x = (p.W + TW - 1) / TW;
  p.tiles_y = (p.H + G::R - 1) / G::R;
  CUtensorMap xmap;
  std::memset(&xmap, 0, sizeof(xmap));
  p.use_tma =
      ((p.W & 3) == 0 && (reinterpret_cast<uintptr_t>(p.x) & 15) == 0 && make_xmap<ORI, TW, FB, F16>(&xmap, p)) ? 1 : 0;
  const int64_t nt = (int64_t)p.tiles_x * p.tiles_y * p.nfb * p.N;
  if (nt > INT32_MAX) return cudaErrorInvalidValue;
  p.ntiles = (int)nt;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)std::min<int64_t>(nt, sms));
  cfg.blockDim = dim3(G::NTHREADS);
  cfg.dynamicSmemBytes = G::SMEM_ALLOC;
  cfg.stream = stream;
  // programmatic dependent launch: the kernel waits (griddepcontrol.wait) for
  // the previous one before touching its inputs and outputs
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, ppconv_tc_kernel<ORI, TW, FB, F16>, p, xmap);
}

template <int ORI, int TW, int FB>
cudaError_t launch(const TcParams& p, cudaStream_t stream, int sms, bool f16) {
  return f16 ? launch_one<ORI, TW, FB, true>(p, stream, sms) : launch_one<ORI, TW, FB, false>(p, stream, sms);
}

}  // namespace

namespace ppc {

pp_status tc_prepare() {
  if (prepare() != cudaSuccess || device_sms() <= 0) return PP_ERR_CUDA;
  // the entry point is process-wide; looked up at the first set-up of each device
  const cudaError_t e = g_encode_once.run([](int) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode.store(reinterpret_cast<EncodeTiledFn>(fn), std::memory_order_release);
    else
      cudaGetLastError();  // without the entry point every launch uses per-thread loads
    return cudaSuccess;
  });
  return e == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

// Dense per-tap weights of every (FB-filter block, 8-channel chunk), split into
// tf32 hi / lo, in the canonical K-major layout of one 2 FB-row tile per tap
// (rows 0 .. FB-1 the hi values, FB .. 2 FB-1 the lo values): element (row r,
// channel k) at byte (k / 4) * (2 FB * 16) + r * 16 + (k % 4) * 4.  The hi or the
// lo rows alone are an FB-row operand with the same K-half stride; all of them
// are the pixel-major kernel's merged operand.  FB = 64 for layers with at most
// 64 filters, else 128.
pp_status tc_build(TcLayout* T, const pp_packed* pk, cudaStream_t stream) {
  const int Co = pk->Co, Ci = pk->Ci;
  const int FB = Co <= 64 ? 64 : 128;
  T->FB = FB;
  T->nfb = (Co + FB - 1) / FB;
  T->nch = (Ci + KC - 1) / KC;
  const size_t wtile = (size_t)FB * KC * 4;
  const size_t wchunk = NTAP * 2 * wtile;
  const size_t total = (size_t)T->nfb * T->nch * wchunk;
  std::vector<float> host(total / 4, 0.f);
  for (int j = 0; j < Co; ++j) {
    const int fb = j / FB, f = j % FB;
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
        const size_t base = ((size_t)fb * T->nch + c) * wchunk + (size_t)t * 2 * wtile;
        // one 2 FB-row tile per tap: rows 0 .. FB-1 hi, FB .. 2 FB-1 lo
        const size_t within = (size_t)(k / 4) * (2 * FB * 16) + (size_t)f * 16 + (size_t)(k % 4) * 4;
        host[(base + within) / 4] = hi;
        host[(base + within + FB * 16) / 4] = lo;
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
  T->state = new (std::nothrow) TcState();
  if (!T->state) {
    cudaFree(d);
    return PP_ERR_OOM;
  }
  T->dmem = d;
  T->dbytes = total + 256;
  T->a = static_cast<const unsigned char*>(d);
  T->status = reinterpret_cast<int*>(static_cast<unsigned char*>(d) + total);
  return PP_OK;
}

// The same layer for the fp16 split (PP_PRECISION_F16X3): per (filter block,
// 16-channel chunk, tap) one tile of 2 FB rows x 16 f16 in the canonical
// K-major layout, element (row r, channel k) at byte (k / 8) * (2 FB * 16) + r *
// 16 + (k % 8) * 2, rows 0 .. FB-1 hi = f16(w s) and FB .. 2 FB-1 lo = f16((w s -
// hi) * 2^11), with s the filter's scale: the power of two that puts its largest
// kept |w| in [2^13, 2^14).  The input is scaled by xs, the largest power of two
// with input_bound * xs <= 2^14, so inputs up to four times the bound stay below
// 65504, the largest fp16 value.  rscale[j] = 1 / (s_j xs) for reordered filter j
// (1 / xs for an empty filter and past Co).  Conversions round to nearest.
pp_status tc_build16(TcLayout* T, const pp_packed* pk, float input_bound, cudaStream_t stream) {
  const int Co = pk->Co, Ci = pk->Ci, FB = T->FB;
  if (!(input_bound > 0.f) || !std::isfinite(input_bound)) input_bound = 16384.f;
  int ex = 0;
  const float m = std::frexp(input_bound, &ex);  // input_bound = m 2^ex, m in [0.5, 1)
  if (m == 0.5f) --ex;                             // ex = ceil(log2(input_bound))
  const int xs_exp = 14 - ex;
  const int nch16 = (Ci + 15) / 16;
  const size_t wtile = (size_t)FB * 16 * 2;
  const size_t wchunk = NTAP * 2 * wtile;
  const size_t wbytes = (size_t)T->nfb * nch16 * wchunk;
  const size_t sbytes = (size_t)T->nfb * FB * 4;
  std::vector<uint16_t> host(wbytes / 2, 0);
  std::vector<float> rs((size_t)T->nfb * FB, std::ldexp(1.f, -xs_exp));
  for (int j = 0; j < Co; ++j) {
    float mx = 0.f;
    for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e)
      for (int q = 0; q < 4; ++q) mx = std::max(mx, std::fabs(pk->kw[(size_t)e * 4 + q]));
    int we = 0;
    if (mx > 0.f) std::frexp(mx, &we);  // mx in [2^(we-1), 2^we)
    const int ws_exp = mx > 0.f ? 14 - we : 0;
    rs[j] = std::ldexp(1.f, -ws_exp - xs_exp);
    const int fb = j / FB, f = j % FB;
    for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e) {
      const int i = pk->kidx[e], c = i / 16, k = i % 16;
      const uint8_t* taps = &pk->taps[4 * pk->kpat[e]];
      for (int q = 0; q < 4; ++q) {
        const float ws = std::ldexp(pk->kw[(size_t)e * 4 + q], ws_exp);  // exact
        const __half h = __float2half_rn(ws);
        const __half l = __float2half_rn((ws - __half2float(h)) * 2048.f);
        const size_t base = ((size_t)fb * nch16 + c) * wchunk + (size_t)taps[q] * 2 * wtile;
        const size_t within = (size_t)(k / 8) * (2 * FB * 16) + (size_t)f * 16 + (size_t)(k % 8) * 2;
        std::memcpy(&host[(base + within) / 2], &h, 2);
        std::memcpy(&host[(base + within + FB * 16) / 2], &l, 2);
      }
    }
  }
  void* d = nullptr;
  if (cudaMalloc(&d, wbytes + sbytes) != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_OOM;
  }
  if (cudaMemcpyAsync(d, host.data(), wbytes, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      cudaMemcpyAsync(static_cast<unsigned char*>(d) + wbytes, rs.data(), sbytes, cudaMemcpyHostToDevice, stream) !=
          cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    cudaFree(d);
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  if (T->dmem16) cudaFree(T->dmem16);
  T->dmem16 = d;
  T->dbytes16 = wbytes + sbytes;
  T->a16 = static_cast<const unsigned char*>(d);
  T->rscale = reinterpret_cast<const float*>(static_cast<unsigned char*>(d) + wbytes);
  T->nch16 = nch16;
  T->xscale = std::ldexp(1.f, xs_exp);
  return PP_OK;
}

// Geometry the launch will use: orientation and tile width for a map width.
void tc_geometry(const TcLayout& T, int W, bool pool, int* ori, int* tw) {
  const bool f16 = T.f16;
  // a pixel-major tile with 128 filters holds one output row (its accumulator
  // row segment is 2 x 128 columns wide), and pooling needs row pairs
  if (T.FB == 64 && !pool && W + 2 <= 64) {
    // narrow map, 64 filters: whole rows flattened into the 128-pixel M side
    *ori = ORI_PFR;
    *tw = W + 2 <= 16 ? 16 : W + 2 <= 32 ? 32 : 64;
  } else if ((T.FB == 64 || W >= 96) && !(T.FB == 128 && pool)) {
    *ori = ORI_PF;
    *tw = 128;
  } else {
    *ori = ORI_FP;
    *tw = W <= 16 ? 16 : W <= 32 ? 32 : W <= 64 ? 64 : 128;
    // f16 filter-major tiles of 128 columns hold one output row (two accumulators per
    // segment): pooling needs row pairs, so wide pooled maps take 64-column tiles
    if (f16 && pool && *tw == 128) *tw = 64;
  }
}

pp_status tc_launch(const TcLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N, int H,
                    int W, int flags, cudaStream_t stream) {
  if ((int64_t)M.Co * H * W >= ((int64_t)1 << 31)) return PP_ERR_UNSUPPORTED;  // 32-bit offsets within an image
  if (tc_prepare() != PP_OK) return PP_ERR_CUDA;
  const bool f16 = T.f16;
  TcParams p;
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
  p.nfb = T.nfb;
  p.FB = T.FB;
  p.flags = flags;
  int ori, tw;
  tc_geometry(T, W, (flags & PP_POOL2) != 0, &ori, &tw);
  const int sms = device_sms();
  cudaError_t e;
  if (ori == ORI_PF)
    e = T.FB == 64 ? launch<ORI_PF, 128, 64>(p, stream, sms, f16) : launch<ORI_PF, 128, 128>(p, stream, sms, f16);
  else if (ori == ORI_PFR)
    e = tw == 16 ? launch<ORI_PFR, 16, 64>(p, stream, sms, f16)
                 : tw == 32 ? launch<ORI_PFR, 32, 64>(p, stream, sms, f16) : launch<ORI_PFR, 64, 64>(p, stream, sms, f16);
  else if (tw == 16)
    e = launch<ORI_FP, 16, 128>(p, stream, sms, f16);
  else if (tw == 32)
    e = launch<ORI_FP, 32, 128>(p, stream, sms, f16);
  else if (tw == 64)
    e = launch<ORI_FP, 64, 128>(p, stream, sms, f16);
  else
    e = launch<ORI_FP, 128, 128>(p, stream, sms, f16);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_CUDA;
  }
  return PP_OK;
}

void tc_free(TcLayout* T) {
  if (T->dmem) cudaFree(T->dmem);
  T->dmem = nullptr;
  if (T->dmem16) cudaFree(T->dmem16);
  T->dmem16 = nullptr;
  T->f16 = false;
  delete T->state;
  T->state = nullptr;
}

pp_status tc_status(const TcLayout& T, int* device_error) {
  int v = 0;
  if (cudaMemcpy(&v, T.status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return PP_ERR_CUDA;
  *device_error = v;
  return PP_OK;
}

}  // namespace ppc

namespace {

// One thread polls an mbarrier that nothing ever completes, with the poll of
// the kernels' bounded waits, `polls` times, and records that it gave up and
// how long the polls took (globaltimer, ns).
__global__ void wait_probe_kernel(long long polls, int* gave_up, long long* ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(su32(&bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    uint64_t t0, t1;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0)::"memory");
    bool done = false;
    for (long long i = 0; i < polls && !done; ++i) done = mbar_try(su32(&bar), 0u);
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t1)::"memory");
    *gave_up = done ? 0 : 1;
    *ns = (long long)(t1 - t0);
  }
}

}  // namespace

extern "C" pp_status pp_wait_probe(long long polls, int* gave_up, long long* elapsed_ns) {
  if (!gave_up || !elapsed_ns || polls < 1 || polls > (1LL << 20)) return PP_ERR_INVALID_ARG;
  void* d = nullptr;
  if (cudaMalloc(&d, 16) != cudaSuccess) {
    cudaGetLastError();
    return PP_ERR_OOM;
  }
  long long* d_ns = static_cast<long long*>(d);
  int* d_gave = reinterpret_cast<int*>(static_cast<unsigned char*>(d) + 8);
  wait_probe_kernel<<<1, 32>>>(polls, d_gave, d_ns);
  long long h[2] = {0, 0};
  const bool ok = cudaGetLastError() == cudaSuccess && cudaMemcpy(h, d, 16, cudaMemcpyDeviceToHost) == cudaSuccess;
  cudaFree(d);
  if (!ok) return PP_ERR_CUDA;
  *elapsed_ns = h[0];
  *gave_up = (int)(h[1] & 0xFFFFFFFF);
  return PP_OK;
}
