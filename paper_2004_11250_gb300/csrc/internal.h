// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <mutex>
#include <vector>

#include "ppconv.h"

// The compact pattern-grouped storage of a layer (Section 3, "Sparse model
// storage" and "Matrix reorder"); field meanings are documented at
// pp_pack_layer in ppconv.h.
struct pp_packed {
  int Co = 0, Ci = 0, P = 0;
  std::vector<uint8_t> taps;   // [P][4]
  std::vector<int32_t> perm;   // [Co]
  std::vector<int32_t> kptr;   // [Co + 1]
  std::vector<int32_t> kidx;   // [nk]
  std::vector<uint8_t> kpat;   // [nk]
  std::vector<float> kw;       // [nk][4]
};

namespace ppc {

// Once-per-device set-up of a launch path (kernel attributes, device queries).
// run(init) calls init(dev) with the current device `dev` until one call
// succeeds; concurrent first calls from several host threads serialise on the
// mutex, and a caller that finds the ready flag set (acquire) sees everything
// the successful init wrote (release).  A failed init is retried next time.
struct DeviceOnce {
  static constexpr int kMaxDevices = 64;
  std::mutex mu;
  std::atomic<bool> ready[kMaxDevices]{};
  template <class F>
  cudaError_t run(F&& init) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (ready[dev].load(std::memory_order_acquire)) return cudaSuccess;
    std::lock_guard<std::mutex> lock(mu);
    if (ready[dev].load(std::memory_order_relaxed)) return cudaSuccess;
    e = init(dev);
    if (e == cudaSuccess) ready[dev].store(true, std::memory_order_release);
    return e;
  }
};

// Number of SMs of the current device (queried once per device).
int device_sms();

// Maximum filter slots handled by one warp of the conv kernel.
constexpr int kSlots = 16;
// Input channels staged in shared memory per pipeline step.
constexpr int kChunk = 16;

// A pattern's taps as a 9-bit mask.
uint16_t tap_mask(const uint8_t* taps4);

// Device-side description shared by every kernel of a layer.
struct LayerMeta {
  int Co = 0, Ci = 0;
  const int* perm = nullptr;    // [Co] original channel of reordered filter j
  const float* bias = nullptr;  // [Co] bias in reordered order, or null
};

// Entry blobs of the tensor-memory kernel (conv_tm.cu).
struct TmLayout {
  int G = 0, nch = 0;
  void* dmem = nullptr;
  size_t dbytes = 0;
  const int* boff = nullptr;
  const uint4* blob = nullptr;
};

// Flat tensor-core kernel geometry chosen by timing (pp_layer_autotune) for one
// shape: rows per tile R and split S, used while (N, H, W, flags) match key.
struct TcState {
  int key[4] = {0, 0, 0, -1};
  int R = 0, S = 0;
};

// Dense per-tap tf32 hi/lo weight tiles of the tensor-core kernels (conv_tc.cu,
// conv_tcf.cu), and, once the layer's precision is PP_PRECISION_F16X3, their
// f16 counterpart.
struct TcLayout {
  int FB = 128, nfb = 0, nch = 0;
  void* dmem = nullptr;
  size_t dbytes = 0;
  const unsigned char* a = nullptr;
  int* status = nullptr;        // device word: bit 0 a timed-out wait, bit 1 an input out of the f16 range
  TcState* state = nullptr;  // owned; see tc_free
  // fp16 split: [nfb][nch16][9][2 FB x 16 f16] tiles (hi rows, then lo rows scaled by 2^11) and, per
  // reordered filter, 1 / (its weight scale x the input scale), a power of two
  bool f16 = false;             // launches run the f16 instantiations
  int nch16 = 0;                // 16-channel chunks
  float xscale = 1.f;           // power of two applied to x before the split
  void* dmem16 = nullptr;
  size_t dbytes16 = 0;
  const unsigned char* a16 = nullptr;
  const float* rscale = nullptr;
};
// Device status bits of a tensor-core layer.
constexpr int kStatusTimeout = 1;
constexpr int kStatusF16Range = 2;

pp_status tc_prepare();
pp_status tc_build(TcLayout* T, const pp_packed* pk, cudaStream_t stream);
pp_status tc_launch(const TcLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N,
                    int H, int W, int flags, cudaStream_t stream);
pp_status tc_status(const TcLayout& T, int* device_error);
// Build the f16 tiles and scales (precision PP_PRECISION_F16X3) for inputs bounded by input_bound.
pp_status tc_build16(TcLayout* T, const pp_packed* pk, float input_bound, cudaStream_t stream);
void tc_free(TcLayout* T);
// Flat variant (maps up to 128 pixels wide, 128-filter blocks); returns
// PP_ERR_UNSUPPORTED for shapes it does not handle.
pp_status tcf_launch(const TcLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N,
                     int H, int W, int flags, cudaStream_t stream);
// The flat kernel's best geometries (rows per tile R, split S) for a shape by
// its cost model, best first; returns how many (up to maxn).
int tcf_plan(const TcLayout& T, int N, int H, int W, int flags, int* R, int* S, int maxn);
// Use geometry (R, S) for launches of this shape (R = 0: back to the model).
void tcf_pin(const TcLayout& T, int N, int H, int W, int flags, int R, int S);
// True when the flat kernel can run geometry (R, S) for this shape.
bool tcf_can_run(const TcLayout& T, int N, int H, int W, int flags, int R, int S);
// The geometry pinned for this shape, or R = S = 0.
void tcf_pinned(const TcLayout& T, int N, int H, int W, int flags, int* R, int* S);

// Direct FMA kernel for layers with few input or few output channels: dense
// [Co][Ci][9] fp32 weights (zeros where pruned) and the bias, original order.
constexpr int kDirectMaxSmall = 16;
struct DirectLayout {
  void* dmem = nullptr;
  const float* w = nullptr;
  const float* bias = nullptr;
  int Co = 0, Ci = 0;
};
bool direct_applicable(int Co, int Ci);
pp_status direct_build(DirectLayout* D, const float* w_dense, const float* bias, int Co, int Ci, cudaStream_t stream);
pp_status direct_launch(const DirectLayout& D, const float* x, float* y, const float* skip, int N, int H, int W,
                        int flags, cudaStream_t stream);
void direct_free(DirectLayout* D);

// True when every pattern of the set is one of the ring patterns (centre plus
// 3 consecutive neighbours); ring_of[p] receives its ring index.
bool tm_supports(const uint8_t* taps, int P, std::vector<int>& ring_of);
pp_status tm_prepare();
pp_status tm_build(TmLayout* T, const pp_packed* pk, const std::vector<int>& ring_of, cudaStream_t stream);
pp_status tm_launch(const TmLayout& T, const LayerMeta& M, const float* x, float* y, const float* skip, int N,
                    int H, int W, int flags, cudaStream_t stream);

}  // namespace ppc
