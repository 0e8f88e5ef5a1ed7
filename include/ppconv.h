/*
 * ppconv.h -- C ABI of a GB300 (sm_103a) library for forward inference of
 * pattern- and connectivity-pruned 3x3 convolution layers.
 *
 * Method: Niu et al., "Towards Real-Time DNN Inference on Mobile Platforms
 * with Model Pruning and Compiler Optimization" (IJCAI-20 demo).
 *   Section 2  connectivity pruning removes whole (output, input) kernels;
 *              pattern pruning keeps certain locations of each kernel: here a
 *              kept kernel keeps 4 of its 9 taps, forming one pattern of a small
 *              caller-given pattern set.
 *   Section 3  "Sparse model storage": zeros and structurally redundant
 *              indices are not stored; "Matrix reorder": filters are reordered
 *              so that similar ones sit together, and the kept kernels of each
 *              filter are compacted; "DSL related optimization": convolution is
 *              fused with its activation to cut data movement.
 *
 * Scope: 3x3 kernels, stride 1, zero padding 1, fp32, NCHW activations.
 * Anything else is rejected with PP_ERR_UNSUPPORTED.
 *
 * Conventions
 *   - Tap index t = 3*ky + kx (ky, kx in 0..2); weights are [Co][Ci][9].
 *   - Every function returns a pp_status (0 = PP_OK) unless noted.  Arguments
 *     are validated on the host before any device work; a call that fails
 *     validation has no effect.
 *   - Handles (pp_packed, pp_layer, pp_dense, pp_net) are opaque, created and
 *     owned by the library, and released with their destroy function
 *     (destroy(NULL) is a no-op).
 *   - Device calls take a CUDA stream as `void*` (a cudaStream_t; NULL = the
 *     legacy default stream), enqueue their work on it and never synchronise
 *     unless stated.  Launch errors are returned by the call; faults that
 *     happen later surface at the caller's next synchronisation.
 *   - Activation, skip and output pointers are caller-owned device memory,
 *     dense NCHW fp32.  Outputs must be 16-byte aligned and inputs at least
 *     4-byte aligned (a 16-byte aligned input with W a multiple of 4 takes the
 *     faster bulk-copy paths); others are rejected with PP_ERR_INVALID_ARG.
 *     An output must not overlap an input.
 *   - A handle may be used from one host thread at a time.
 */
#ifndef PPCONV_H
#define PPCONV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum pp_status_code {
  PP_OK = 0,
  PP_ERR_INVALID_ARG = 1,        /* null pointer, non-positive size, bad flag  */
  PP_ERR_BAD_PATTERN_SET = 2,    /* a pattern is not 4 distinct ascending taps in 0..8, or repeats */
  PP_ERR_TAP_NOT_IN_PATTERN = 3, /* a kept kernel has a nonzero tap outside every pattern */
  PP_ERR_PRUNED_NONZERO = 4,     /* a connectivity-pruned kernel has a nonzero weight */
  PP_ERR_PATTERN_ID_MISMATCH = 5,/* a caller-given pattern id does not cover the kernel's taps */
  PP_ERR_UNSUPPORTED = 6,        /* shape or option outside the library's scope */
  PP_ERR_CUDA = 7,               /* a CUDA runtime call failed */
  PP_ERR_OOM = 8                 /* host or device allocation failed */
};
typedef int pp_status;

/* Epilogue flags of a convolution, applied in this order after the bias:
 * add the skip tensor, ReLU, 2x2 max pool (stride 2, floor). */
#define PP_ADD_SKIP 1
#define PP_RELU 2
#define PP_POOL2 4

/* Static string naming a status code ("PP_OK", ...); never NULL. */
const char* pp_status_string(pp_status status);
/* Library version: major * 10000 + minor * 100 + patch. */
int pp_version(void);

/* ------------------------------------------------------------------------
 * Host packer: compact pattern-grouped storage with filter reorder (Section 3).
 * ------------------------------------------------------------------------ */
typedef struct pp_packed pp_packed;

/*
 * Validate a pruned layer and build its compact form.  Host only, synchronous.
 *   w            [Co][Ci][9] fp32 host weights; zero outside the kept taps
 *   mask         [Co][Ci] host bytes, nonzero = kernel kept (connectivity)
 *   pattern_taps [P][4] host bytes, each row 4 distinct ascending taps in 0..8
 *   P            number of patterns, 1..126, rows pairwise distinct
 *   pattern_ids  [Co][Ci] optional (NULL = infer); for each kept kernel, the
 *                pattern it uses.  Inferred id = lowest pattern containing the
 *                kernel's nonzero taps.
 *   out          receives a new handle on success, untouched on failure
 * Stored form (read with pp_packed_arrays):
 *   perm[Co]     perm[j] = original index of the j-th filter; filters are
 *                sorted by (kept count descending, dominant pattern ascending,
 *                index ascending), the dominant pattern being the most frequent
 *                pattern id among the filter's kept kernels (lowest on ties)
 *   kptr[Co+1]   kept kernels of filter perm[j] are entries kptr[j]..kptr[j+1]-1
 *   kidx[nk]     input channel of each entry
 *   kpat[nk]     pattern id of each entry
 *   kw[nk][4]    weights on the pattern's taps in ascending tap order
 *   Entries of a filter are ordered by (pattern id, input channel).
 * Errors: PP_ERR_INVALID_ARG, PP_ERR_BAD_PATTERN_SET, PP_ERR_PRUNED_NONZERO,
 *   PP_ERR_TAP_NOT_IN_PATTERN, PP_ERR_PATTERN_ID_MISMATCH, PP_ERR_OOM.
 */
pp_status pp_pack_layer(const float* w, const uint8_t* mask, const uint8_t* pattern_taps, int P, int Co, int Ci,
                        const uint8_t* pattern_ids, pp_packed** out);

/* Sizes of a packed layer; any output pointer may be NULL. */
pp_status pp_packed_info(const pp_packed* pk, int64_t* nk, int* Co, int* Ci, int* P);

/* Borrowed read-only views of the stored arrays (valid until destroy); any
 * output pointer may be NULL.  taps is the [P][4] pattern set. */
pp_status pp_packed_arrays(const pp_packed* pk, const int32_t** perm, const int32_t** kptr, const int32_t** kidx,
                           const uint8_t** kpat, const float** kw, const uint8_t** taps);

/* Rebuild the dense weights [Co][Ci][9] and mask [Co][Ci] (host buffers; either
 * may be NULL).  Kept taps come back bit for bit, every other tap as +0.0. */
pp_status pp_unpack_layer(const pp_packed* pk, float* w_out, uint8_t* mask_out);

void pp_packed_destroy(pp_packed* pk);

/* Permute the input channels of a layer's dense description, for packing a
 * layer whose input activation is stored in another channel order (see
 * pp_layer_set_output_order): position c of the result holds original input
 * channel layout[c], i.e. w_out[o][c][t] = w[o][layout[c]][t], and likewise
 * mask_out[o][c] and ids_out[o][c] (each optional: NULL skips it; its source
 * must then be given only if its output is).  Host only; outputs must not
 * overlap inputs.  Errors: PP_ERR_INVALID_ARG (null pointer, Co or Ci < 1,
 * layout not a permutation of 0..Ci-1, an output without its input). */
pp_status pp_permute_input_channels(const float* w, const uint8_t* mask, const uint8_t* pattern_ids, int Co, int Ci,
                                    const int32_t* layout, float* w_out, uint8_t* mask_out, uint8_t* ids_out);

/* Fold an inference batch normalisation that follows the convolution into its
 * weights and bias (Section 3: convolution fused with the layers after it), in
 * place on host arrays before packing: w [Co][Ci][9] becomes w * g[o] and
 * bias [Co] becomes (bias - mean) * g[o] + beta, with g[o] = gamma[o] /
 * sqrt(var[o] + eps) evaluated in double and each result rounded once to fp32.
 * One factor per filter keeps every zero weight zero, so a pattern-pruned and
 * connectivity-pruned layer stays one (same masks, same pattern ids).  bias
 * must be an array of Co (zeros for a convolution without bias).  Host only,
 * synchronous.  Errors: PP_ERR_INVALID_ARG (null pointer, Co or Ci < 1, eps
 * negative or NaN, var[o] + eps not positive). */
pp_status pp_fold_batchnorm(float* w, float* bias, const float* gamma, const float* beta, const float* mean,
                            const float* var, float eps, int Co, int Ci);

/* ------------------------------------------------------------------------
 * Device layer: the pruned convolution on the GPU (Sections 2-3).
 * ------------------------------------------------------------------------ */
typedef struct pp_layer pp_layer;

/*
 * Upload a packed layer to the current CUDA device.  The library allocates
 * and owns the device copy (a few bytes per kept kernel) and derives its
 * kernel-side layout from pk; pk may be destroyed afterwards.
 *   bias   [Co] host fp32 or NULL (no bias)
 *   stream copies are enqueued on it; the call waits for them before returning
 * Errors: PP_ERR_INVALID_ARG, PP_ERR_UNSUPPORTED, PP_ERR_CUDA, PP_ERR_OOM.
 */
pp_status pp_layer_create(const pp_packed* pk, const float* bias, void* stream, pp_layer** out);

/* Co, Ci and the number of device bytes held by the layer (any may be NULL). */
pp_status pp_layer_info(const pp_layer* layer, int* Co, int* Ci, int64_t* device_bytes);

/*
 * y = epilogue(conv(x) + bias): the pruned 3x3 convolution of every image of
 * the batch, fused with the epilogue given by flags (PP_ADD_SKIP, PP_RELU,
 * PP_POOL2, in that order).  Asynchronous on stream.
 *   x     [N][Ci][H][W] device input
 *   y     [N][Co][H][W], or [N][Co][H/2][W/2] with PP_POOL2 (H, W even)
 *   skip  [N][Co][H][W] device tensor added before the ReLU (PP_ADD_SKIP), else NULL
 * Errors: PP_ERR_INVALID_ARG (null pointer, N/H/W < 1, flags, y not 16-byte
 *   or x not 4-byte aligned), PP_ERR_UNSUPPORTED (PP_POOL2 with odd H or W, or
 *   a pattern the kernels do not cover), PP_ERR_CUDA (launch failure).
 */
pp_status pp_conv_forward(const pp_layer* layer, const float* x, float* y, const float* skip, int N, int H, int W,
                          int flags, void* stream);

/*
 * Allocation-free forward through the flat tensor-core kernel
 * (PP_KERNEL_TC_FLAT).  The paper has no counterpart: it is for callers that
 * must not allocate device memory while they run layers (their device memory
 * budget is reserved up front by another allocator, or their loop cannot take
 * the device-wide synchronisation that cudaMalloc / cudaFree may cause).  The
 * flat kernel reduces its cluster-split partial tiles through distributed
 * shared memory, so it needs no workspace; this call runs it whatever kernel
 * the layer has selected and never allocates or frees device memory.
 *   Same arguments, layout, epilogue and fp32 bound as pp_conv_forward.
 *   The first call on a device sets the kernel's launch attributes and should
 *   come before any stream capture.
 * Errors: as pp_conv_forward; PP_ERR_UNSUPPORTED also when the layer cannot
 *   run the flat kernel at this shape (Co <= 64, W > 128).
 */
pp_status pp_conv_forward_noalloc(const pp_layer* layer, const float* x, float* y, const float* skip, int N, int H,
                                  int W, int flags, void* stream);

/*
 * Output channel order of a layer (Section 3 "Matrix reorder", folded into
 * the next layer).  order[o] = the output channel where original filter o is
 * stored (a permutation of 0..Co-1, host array); NULL restores the original
 * order (order[o] = o), the default.  Every kernel and pp_conv_forward_noalloc
 * honour it; a skip tensor (PP_ADD_SKIP) is read at the same channel as the
 * output it is added to.
 * Folding the filter reorder of layer k into layer k + 1: give layer k
 * order[perm_k[j]] = j (filter j of the reordered layer is stored at channel
 * j, so the epilogue writes the filters in the order they are computed), and
 * pack layer k + 1 from weights whose input channels were permuted the same
 * way (pp_permute_input_channels with layout = perm_k).
 * Synchronous on stream (uploads Co indices; layers with a direct-kernel
 * layout also rebuild it).  A CUDA graph captured earlier keeps the direct
 * kernel's old weights: re-capture after calling this (pp_net_use_graph).
 * Errors: PP_ERR_INVALID_ARG (not a permutation), PP_ERR_CUDA, PP_ERR_OOM. */
pp_status pp_layer_set_output_order(pp_layer* layer, const int32_t* order, void* stream);

/*
 * Arithmetic of the tensor-core kernels (PP_KERNEL_TC, PP_KERNEL_TC_FLAT and
 * pp_conv_forward_noalloc); the FMA kernels always compute in fp32.  Both
 * modes meet |gpu - exact| <= 1e-5 * S (S = |bias| + sum |w x| + |skip|) on
 * the inputs their conditions cover.
 *   PP_PRECISION_TF32X3  the default: each operand v = hi + lo with hi its
 *       tf32 truncation; w_hi x_hi + w_lo x_hi + w_hi x_lo accumulated in fp32
 *       (tcgen05 kind::tf32).  Any fp32 input.
 *   PP_PRECISION_F16X3   each operand v = hi + 2^-11 lo with hi = f16(v) and
 *       lo = f16((v - hi) 2^11), rounded to nearest, after exact power-of-two
 *       scaling: per filter for the weights (largest kept |w| into
 *       [2^13, 2^14)), per layer for the input (x_s = x * s_x, s_x the largest
 *       power of two with input_bound * s_x <= 2^14); w_hi x_hi into one fp32
 *       accumulator, w_lo x_hi + w_hi x_lo into a second (tcgen05 kind::f16,
 *       twice the tf32 rate on half the operand bytes), combined as
 *       (acc1 + 2^-11 acc2) / (s_w s_x).  Per product the representation
 *       error is below 3 * 2^-22 of |w x| while |x_s| >= 2^-14; below that
 *       fp16's subnormal spacing adds at most 2^-36 / s_x per unit of |w|, so
 *       the bound holds unless an output's whole receptive field is tiny
 *       (mean |x| below ~1e-6 / s_x) yet not zero.  Inputs must satisfy
 *       |x_s| < 65504, fp16's largest value (|x| < 4 * input_bound at least);
 *       a launch that meets a larger input, or one that is not finite, sets
 *       bit 1 of the layer's device status word and its output is invalid.
 *       input_bound <= 0 means 16384 (s_x = 1).
 * Switching to PP_PRECISION_F16X3 builds the f16 weight layout (half the
 * bytes of the tf32 one) from a host copy of the packed layer, synchronously
 * on stream; a CUDA graph captured before keeps the old arithmetic.
 * Errors: PP_ERR_INVALID_ARG (unknown precision, NaN bound), PP_ERR_UNSUPPORTED
 * (F16X3 on a layer without a tensor-core layout), PP_ERR_CUDA,
 * PP_ERR_OOM. */
#define PP_PRECISION_TF32X3 0
#define PP_PRECISION_F16X3 1
pp_status pp_layer_set_precision(pp_layer* layer, int precision, float input_bound, void* stream);
/* The layer's precision and input scale s_x (1 under PP_PRECISION_TF32X3); either pointer may be NULL. */
pp_status pp_layer_precision(const pp_layer* layer, int* precision, float* input_scale);

/* Which kernel pp_conv_forward runs for a layer.  All compute the same
 * convolution within the documented fp32 bound.
 *   PP_KERNEL_TC        implicit GEMM on the tensor cores over the 9 taps
 *                       (zeros where pruned), 3xTF32 for fp32 accuracy; any
 *                       pattern set; any Ci (channels padded to the
 *                       chunk of 8, or 16 in fp16, with zeros).
 *   PP_KERNEL_TC_FLAT   the same contraction with whole output rows flattened
 *                       into one MMA and, for layers with few output tiles,
 *                       the input channels split over a thread-block cluster
 *                       (partial tiles reduced through distributed shared
 *                       memory); maps at most 128 pixels wide and layers with
 *                       more than 64 filters (other shapes run PP_KERNEL_TC).
 *   PP_KERNEL_TMEM      FP32 FMA over kept taps only, accumulators in tensor
 *                       memory; ring patterns only (the centre tap plus 3
 *                       consecutive of its 8 neighbours).
 *   PP_KERNEL_REGISTER  FP32 FMA over kept taps, accumulators in registers;
 *                       any pattern set.
 *   PP_KERNEL_DIRECT    FP32 FMA over all 9 taps of dense [Co][Ci][9] weights
 *                       (zeros where pruned), one 2 x 2 pixel block and up to
 *                       16 filters per thread; layers with at most 16 input
 *                       or at most 16 output channels (first and last layers).
 * PP_KERNEL_AUTO picks by an estimate of each kernel's time for the layer's
 * density (the direct kernel for Ci <= 4).  Setting a kernel the layer cannot
 * run returns PP_ERR_UNSUPPORTED. */
#define PP_KERNEL_AUTO 0
#define PP_KERNEL_TMEM 1
#define PP_KERNEL_REGISTER 2
#define PP_KERNEL_TC 3
#define PP_KERNEL_TC_FLAT 4
#define PP_KERNEL_DIRECT 5
pp_status pp_layer_set_kernel(pp_layer* layer, int kernel);
/* The kernel that pp_conv_forward will run (one of the PP_KERNEL_ values above, not _AUTO). */
pp_status pp_layer_kernel(const pp_layer* layer, int* kernel);
/* Time the kernels that can run this layer (tensor-core, TMEM and direct
 * kernels where their layouts exist; the register kernel only when none of
 * them can) on zero-filled scratch tensors of the given shape and flags (a few
 * launches each, on stream, synchronous) and keep the fastest for the layer; the flat tensor-core kernel is timed at the
 * best few tile geometries (rows per tile, cluster split) of its cost model and
 * keeps the winning one for launches of this shape.  The kernels differ in speed by layer shape:
 * the tensor-core kernel needs many output tiles to fill the GPU, the FMA
 * kernels split small layers across thread-block clusters.  Allocates and
 * frees scratch device memory; must not be called during stream capture.
 * Errors: PP_ERR_INVALID_ARG, PP_ERR_UNSUPPORTED, PP_ERR_CUDA, PP_ERR_OOM. */
pp_status pp_layer_autotune(pp_layer* layer, int N, int H, int W, int flags, void* stream);

/* Tile geometry of the flat tensor-core kernel (PP_KERNEL_TC_FLAT) for launches
 * of shape (N, H, W, flags): R output rows per tile and a cluster split of the
 * input-channel chunks over S CTAs.  pp_layer_flat_geometry reports the pinned
 * pair (R = S = 0 when none is pinned for that shape: the kernel's cost model
 * then decides).  pp_layer_pin_flat_geometry pins (R, S) for that shape, as
 * pp_layer_autotune does with the pair it measured fastest; R = 0 unpins.  One
 * shape is pinned per layer (a new pin replaces the old).  This lets a tuning
 * result be stored and re-applied without timing again.  Host-only, no device
 * work.  Errors: PP_ERR_INVALID_ARG; PP_ERR_UNSUPPORTED when the layer has no
 * flat-kernel layout (fewer than 65 filters) or the kernel cannot run (R, S)
 * for that shape (R rows of round_up(W + 2, 8) pixels must fit one MMA of at
 * most 256 columns, R even when pooling; S a power of 2 up to 16, at most the
 * number of 8-channel chunks (16-channel in PP_PRECISION_F16X3), with tiles x S
 * within the SM count and the cluster size launchable on this GPU; in
 * PP_PRECISION_F16X3 a tile of more than 128 columns runs single-buffered and
 * not as CTA pairs).  S | PP_FLAT_PAIRED names the same
 * split run by CTA pairs: two filter blocks of a tile share each MMA (M = 256
 * over two SMs, cta_group::2), each SM staging half of the tile's pixels, in
 * clusters of 2 S CTAs (S up to 8; layers with an even number of 128-filter
 * blocks).  Every geometry stays within the error bound; geometries with
 * different splits group the channel sum differently, so their last bits may
 * differ (each is deterministic). */
#define PP_FLAT_PAIRED 256
pp_status pp_layer_flat_geometry(const pp_layer* layer, int N, int H, int W, int flags, int* R, int* S);
pp_status pp_layer_pin_flat_geometry(pp_layer* layer, int N, int H, int W, int flags, int R, int S);

/* Synchronous: *device_error = 0 unless a launch of this layer's tensor-core
 * kernels met an error since the last read, and its output is then invalid:
 * bit 0 (value 1) a bounded wait gave up; bit 1 (value 2) under
 * PP_PRECISION_F16X3 an input was not finite or overflowed fp16 (|x s_x| >=
 * 65520) after the layer's input scale.  The word is cleared by the read. */
pp_status pp_layer_device_status(const pp_layer* layer, int* device_error);

/* Polls of an mbarrier after which a wait in the tensor-core kernels gives up:
 * the kernel then sets the layer's device status word, skips the rest of its
 * work, waits (with the same bound) for its own copies in flight and exits.
 * A poll that finds the phase incomplete suspends the thread for a few
 * microseconds (3.8 us measured on GB300 with pp_wait_probe), so a wait gives
 * up after about a second; the longest wait of a correct launch is below a
 * millisecond. */
#define PP_WAIT_POLLS (1L << 18)

/* Diagnostic for the bound above.  One thread polls an mbarrier that nothing
 * completes, with the kernels' poll instruction, `polls` times (1 .. 2^20),
 * and reports *gave_up = 1 and the elapsed device time in ns; a full wait
 * takes about PP_WAIT_POLLS / polls times as long.  Synchronous, on the legacy
 * default stream; allocates 16 bytes of device memory for the results.
 * Errors: PP_ERR_INVALID_ARG (null pointer, polls out of range), PP_ERR_OOM,
 * PP_ERR_CUDA. */
pp_status pp_wait_probe(long long polls, int* gave_up, long long* elapsed_ns);

/* Peak-rate probes (diagnostics; the paper has no counterpart).  One launch
 * keeps a single execution pipe busy on every SM of the current device and
 * reports its rate, so roofline fractions can be taken against a measured
 * peak instead of a data-sheet figure:
 *   PP_PROBE_FFMA      fp32 fused multiply-add on the CUDA cores (16
 *                      independent chains per thread, 4 CTAs of 256 threads
 *                      per SM), 2 FLOP per multiply-add;
 *   PP_PROBE_MMA_TF32  tcgen05.mma kind::tf32, M = 128, N = 256, K = 8 per
 *                      instruction, one issuing thread per SM, operands in
 *                      shared memory, accumulator in tensor memory;
 *   PP_PROBE_MMA_F16   the same with kind::f16 (f16 operands, fp32
 *                      accumulation), K = 16.
 *   iters   multiply-add groups per thread (FFMA) or MMA instructions per SM,
 *           1 .. 2^24; pick it so the launch takes a few milliseconds
 *   tflops  FLOP of the launch / its duration (CUDA events), in TFLOP/s
 *   sm_mhz  SM clock during the launch: SM cycles over the global timer of
 *           one CTA, in MHz
 *   ms      duration of the launch
 * Synchronous, on the legacy default stream; allocates and frees a small
 * result buffer.  Errors: PP_ERR_INVALID_ARG (null pointer, kind, iters out
 * of range), PP_ERR_OOM, PP_ERR_CUDA (also when an MMA probe's bounded wait
 * for its instructions ran out). */
#define PP_PROBE_FFMA 0
#define PP_PROBE_MMA_TF32 1
#define PP_PROBE_MMA_F16 2
pp_status pp_peak_probe(int kind, long long iters, double* tflops, double* sm_mhz, double* ms);

void pp_layer_destroy(pp_layer* layer);

/* ------------------------------------------------------------------------
 * Dense (unpruned) 3x3 layer, for the end layers of a pruned network.
 * ------------------------------------------------------------------------ */
typedef struct pp_dense pp_dense;

/* w [Co][Ci][9] and bias [Co] (or NULL) are host fp32; copied to the device. */
pp_status pp_dense_create(const float* w, const float* bias, int Co, int Ci, void* stream, pp_dense** out);

/* Same contract as pp_conv_forward, over all 9 taps of every kernel.  Layers
 * with at most 16 input or at most 16 output channels run the direct FMA
 * kernel (PP_KERNEL_DIRECT); others the register-accumulator kernel. */
pp_status pp_dense_forward(const pp_dense* layer, const float* x, float* y, const float* skip, int N, int H, int W,
                           int flags, void* stream);

/* Co and Ci of a dense layer (either may be NULL). */
pp_status pp_dense_info(const pp_dense* layer, int* Co, int* Ci);

void pp_dense_destroy(pp_dense* layer);

/* ------------------------------------------------------------------------
 * Network executor: a chain of convolutions on one stream (Section 3's
 * layer-wise representation, run as a fixed schedule).
 * ------------------------------------------------------------------------ */
typedef struct pp_net pp_net;

/* An empty network for inputs [N][C][H][W]. */
pp_status pp_net_create(int N, int C, int H, int W, pp_net** out);

/*
 * Append one op.  Activation 0 is the network input; op k (0-based) writes
 * activation k + 1.  skip_from = index of an earlier activation added before
 * the ReLU (requires PP_ADD_SKIP in flags and the same shape), or -1.
 * The layer handle is borrowed: it must outlive the network.
 */
pp_status pp_net_add_conv(pp_net* net, const pp_layer* layer, int flags, int skip_from);
pp_status pp_net_add_dense(pp_net* net, const pp_dense* layer, int flags, int skip_from);

/* Plan activation buffers and allocate them on the current device (library
 * owned), then autotune the kernel of every pruned op at its shape
 * (pp_layer_autotune; this changes the kernel choice of the borrowed layers).
 * Must be called once, after the last add and before the first run. */
pp_status pp_net_finalize(pp_net* net);

/* Shape of the network output (any pointer may be NULL). */
pp_status pp_net_output_shape(const pp_net* net, int* N, int* C, int* H, int* W);

/* With enable != 0, pp_net_run captures its launches into a CUDA graph on the
 * first call for a given (x, y, stream) and replays that graph afterwards (one
 * host launch per run).  Needs a non-NULL stream; with the legacy default
 * stream the ops are launched one by one.  Default: off.  A graph keeps the
 * kernels and tile geometries the layers had when it was captured; every call
 * of this function drops the captured graphs, so calling it again after
 * changing a borrowed layer (pp_layer_set_kernel, pins) makes the next run
 * capture the change. */
pp_status pp_net_use_graph(pp_net* net, int enable);

/* Device-resident run: x and y are device buffers of the input and output
 * shapes.  Launches every op on stream; asynchronous. */
pp_status pp_net_run(pp_net* net, const float* x, float* y, void* stream);

/*
 * End-to-end run on host buffers: copies x_host to the device, runs the
 * network and copies the output to y_host, all on stream, and synchronises
 * the stream before returning.  Pinned host memory gives overlap-free DMA at
 * full speed; pageable memory works too.  With graphs enabled, a non-NULL
 * stream and page-locked x_host and y_host, the two copies and the ops are one
 * CUDA graph, captured on the first call for those buffers and stream and
 * replayed afterwards (one host launch per frame).
 */
pp_status pp_net_run_host(pp_net* net, const float* x_host, float* y_host, void* stream);

void pp_net_destroy(pp_net* net);

#ifdef __cplusplus
}
#endif
#endif /* PPCONV_H */
