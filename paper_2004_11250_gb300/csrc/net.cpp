// Network executor: a fixed schedule of fused convolutions on one CUDA stream.
//
// Section 3 of Niu et al. represents a model layer by layer and fuses each
// convolution with its activation; here a network is the list of those fused
// ops.  The executor plans intermediate activation buffers once (liveness-based
// reuse, so a 20-layer stack needs only a few buffers), then every run
// launches the ops back to back on the caller's stream, optionally replayed as
// one captured CUDA graph so the host pays one launch per frame.
#include <cuda_runtime.h>

#include <algorithm>
#include <new>
#include <vector>

#include "internal.h"

namespace {

struct OpDesc {
  const pp_layer* conv = nullptr;
  const pp_dense* dense = nullptr;
  int flags = 0;
  int skip_from = -1;
  int Ci = 0, Co = 0;
  int H = 0, W = 0;    // input spatial size
  int Ho = 0, Wo = 0;  // output spatial size
};

}  // namespace

struct pp_net {
  int N = 0, C = 0, H = 0, W = 0;
  std::vector<OpDesc> ops;
  bool finalized = false;
  std::vector<float*> buffers;    // library-owned intermediate buffers
  std::vector<int> act_buffer;    // activation index -> buffer index (-1: user input/output)
  std::vector<size_t> act_elems;  // elements of each activation
  float* d_in = nullptr;          // staging buffers of pp_net_run_host
  float* d_out = nullptr;
  bool use_graph = false;
  cudaGraphExec_t gexec = nullptr;
  const float* g_x = nullptr;
  float* g_y = nullptr;
  cudaStream_t g_stream = nullptr;
  // pp_net_run_host with pinned buffers: the two copies and the ops in one graph
  cudaGraphExec_t hexec = nullptr;
  const float* h_x = nullptr;
  float* h_y = nullptr;
  cudaStream_t h_stream = nullptr;
};


extern "C" pp_status pp_net_create(int N, int C, int H, int W, pp_net** out) {
  if (!out || N < 1 || C < 1 || H < 1 || W < 1) return PP_ERR_INVALID_ARG;
  pp_net* n = new (std::nothrow) pp_net;
  if (!n) return PP_ERR_OOM;
  n->N = N;
  n->C = C;
  n->H = H;
  n->W = W;
  *out = n;
  return PP_OK;
}

namespace {

pp_status add_op(pp_net* net, OpDesc d, int Co, int Ci) {
  if (net->finalized) return PP_ERR_INVALID_ARG;
  if (d.flags & ~(PP_ADD_SKIP | PP_RELU | PP_POOL2)) return PP_ERR_INVALID_ARG;
  const int k = (int)net->ops.size();
  int C = net->C, H = net->H, W = net->W;
  if (k > 0) {
    C = net->ops.back().Co;
    H = net->ops.back().Ho;
    W = net->ops.back().Wo;
  }
  if (Ci != C) return PP_ERR_INVALID_ARG;
  const bool has_skip = d.flags & PP_ADD_SKIP;
  if (has_skip != (d.skip_from >= 0)) return PP_ERR_INVALID_ARG;
  if (has_skip) {
    if (d.skip_from > k) return PP_ERR_INVALID_ARG;
    // activation a has shape of op a-1's output (or the input for a = 0)
    int sc = net->C, sh = net->H, sw = net->W;
    if (d.skip_from > 0) {
      const OpDesc& s = net->ops[d.skip_from - 1];
      sc = s.Co;
      sh = s.Ho;
      sw = s.Wo;
    }
    if (sc != Co || sh != H || sw != W) return PP_ERR_INVALID_ARG;
  }
  if ((d.flags & PP_POOL2) && ((H & 1) || (W & 1))) return PP_ERR_UNSUPPORTED;
  d.Ci = Ci;
  d.Co = Co;
  d.H = H;
  d.W = W;
  d.Ho = (d.flags & PP_POOL2) ? H / 2 : H;
  d.Wo = (d.flags & PP_POOL2) ? W / 2 : W;
  try {
    net->ops.push_back(d);
  } catch (const std::bad_alloc&) {
    return PP_ERR_OOM;
  }
  return PP_OK;
}

pp_status run_ops(pp_net* net, const float* x, float* y, cudaStream_t stream) {
  const int n = (int)net->ops.size();
  auto act = [&](int a) -> const float* {
    if (a == 0) return x;
    if (a == n) return y;
    return net->buffers[net->act_buffer[a]];
  };
  for (int k = 0; k < n; ++k) {
    const OpDesc& d = net->ops[k];
    float* out = (k + 1 == n) ? y : net->buffers[net->act_buffer[k + 1]];
    const float* skip = d.skip_from >= 0 ? act(d.skip_from) : nullptr;
    pp_status st = d.conv ? pp_conv_forward(d.conv, act(k), out, skip, net->N, d.H, d.W, d.flags, stream)
                          : pp_dense_forward(d.dense, act(k), out, skip, net->N, d.H, d.W, d.flags, stream);
    if (st != PP_OK) return st;
  }
  return PP_OK;
}

}  // namespace

extern "C" pp_status pp_net_add_conv(pp_net* net, const pp_layer* layer, int flags, int skip_from) {
  if (!net || !layer) return PP_ERR_INVALID_ARG;
  int Co = 0, Ci = 0;
  pp_layer_info(layer, &Co, &Ci, nullptr);
  OpDesc d;
  d.conv = layer;
  d.flags = flags;
  d.skip_from = skip_from;
  return add_op(net, d, Co, Ci);
}

extern "C" pp_status pp_net_add_dense(pp_net* net, const pp_dense* layer, int flags, int skip_from) {
  if (!net || !layer) return PP_ERR_INVALID_ARG;
  int Co = 0, Ci = 0;
  pp_dense_info(layer, &Co, &Ci);
  OpDesc d;
  d.dense = layer;
  d.flags = flags;
  d.skip_from = skip_from;
  return add_op(net, d, Co, Ci);
}

extern "C" pp_status pp_net_finalize(pp_net* net) {
  if (!net || net->finalized || net->ops.empty()) return PP_ERR_INVALID_ARG;
  const int n = (int)net->ops.size();
  // Activation a (1..n-1) is written by op a-1 and read by op a and by every
  // op whose skip_from is a.
  std::vector<int> last_use(n + 1, 0);
  for (int a = 0; a <= n; ++a) last_use[a] = a;
  for (int k = 0; k < n; ++k)
    if (net->ops[k].skip_from >= 0) last_use[net->ops[k].skip_from] = std::max(last_use[net->ops[k].skip_from], k);
  net->act_elems.assign(n + 1, 0);
  net->act_elems[0] = (size_t)net->N * net->C * net->H * net->W;
  for (int a = 1; a <= n; ++a) {
    const OpDesc& d = net->ops[a - 1];
    net->act_elems[a] = (size_t)net->N * d.Co * d.Ho * d.Wo;
  }
  // Greedy buffer assignment: a buffer is free for activation a once its
  // previous occupant's last reader ran before op a-1 (the writer of a).
  net->act_buffer.assign(n + 1, -1);
  std::vector<int> occupant;       // per buffer: activation currently held
  std::vector<size_t> buf_elems;   // per buffer: capacity needed
  for (int a = 1; a < n; ++a) {
    int pick = -1;
    for (size_t b = 0; b < occupant.size(); ++b)
      if (last_use[occupant[b]] < a - 1) {
        pick = (int)b;
        break;
      }
    if (pick < 0) {
      pick = (int)occupant.size();
      occupant.push_back(a);
      buf_elems.push_back(0);
    }
    occupant[pick] = a;
    buf_elems[pick] = std::max(buf_elems[pick], net->act_elems[a]);
    net->act_buffer[a] = pick;
  }
  for (size_t b = 0; b < buf_elems.size(); ++b) {
    float* p = nullptr;
    if (cudaMalloc(&p, std::max<size_t>(buf_elems[b], 1) * sizeof(float)) != cudaSuccess) {
      cudaGetLastError();
      for (float* q : net->buffers) cudaFree(q);
      net->buffers.clear();
      return PP_ERR_OOM;
    }
    net->buffers.push_back(p);
  }
  // Pick each pruned op's kernel at the op's own shape.
  for (const OpDesc& d : net->ops) {
    if (!d.conv) continue;
    pp_status st = pp_layer_autotune(const_cast<pp_layer*>(d.conv), net->N, d.H, d.W, d.flags, nullptr);
    if (st != PP_OK) {
      for (float* q : net->buffers) cudaFree(q);
      net->buffers.clear();
      return st;
    }
  }
  net->finalized = true;
  return PP_OK;
}

extern "C" pp_status pp_net_output_shape(const pp_net* net, int* N, int* C, int* H, int* W) {
  if (!net) return PP_ERR_INVALID_ARG;
  int c = net->C, h = net->H, w = net->W;
  if (!net->ops.empty()) {
    c = net->ops.back().Co;
    h = net->ops.back().Ho;
    w = net->ops.back().Wo;
  }
  if (N) *N = net->N;
  if (C) *C = c;
  if (H) *H = h;
  if (W) *W = w;
  return PP_OK;
}

extern "C" pp_status pp_net_use_graph(pp_net* net, int enable) {
  if (!net) return PP_ERR_INVALID_ARG;
  net->use_graph = enable != 0;
  // drop the captured graphs: the next runs capture the layers' current kernels
  if (net->gexec) cudaGraphExecDestroy(net->gexec);
  if (net->hexec) cudaGraphExecDestroy(net->hexec);
  net->gexec = nullptr;
  net->hexec = nullptr;
  return PP_OK;
}

extern "C" pp_status pp_net_run(pp_net* net, const float* x, float* y, void* stream_) {
  if (!net || !x || !y || !net->finalized) return PP_ERR_INVALID_ARG;
  cudaStream_t stream = (cudaStream_t)stream_;
  if (!net->use_graph || stream == nullptr) return run_ops(net, x, y, stream);
  if (!net->gexec || net->g_x != x || net->g_y != y || net->g_stream != stream) {
    if (net->gexec) {
      cudaGraphExecDestroy(net->gexec);
      net->gexec = nullptr;
    }
    cudaGraph_t g = nullptr;
    if (cudaStreamBeginCapture(stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) return PP_ERR_CUDA;
    pp_status st = run_ops(net, x, y, stream);
    cudaError_t ce = cudaStreamEndCapture(stream, &g);
    if (st != PP_OK || ce != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      cudaGetLastError();
      return st != PP_OK ? st : PP_ERR_CUDA;
    }
    ce = cudaGraphInstantiate(&net->gexec, g, 0);
    cudaGraphDestroy(g);
    if (ce != cudaSuccess) {
      net->gexec = nullptr;
      return PP_ERR_CUDA;
    }
    net->g_x = x;
    net->g_y = y;
    net->g_stream = stream;
  }
  return cudaGraphLaunch(net->gexec, stream) == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

namespace {

// True for page-locked host memory (cudaHostAlloc / cudaHostRegister).
bool is_pinned(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeHost;
}

}  // namespace

extern "C" pp_status pp_net_run_host(pp_net* net, const float* x_host, float* y_host, void* stream_) {
  if (!net || !x_host || !y_host || !net->finalized) return PP_ERR_INVALID_ARG;
  cudaStream_t stream = (cudaStream_t)stream_;
  const size_t in_bytes = net->act_elems.front() * sizeof(float);
  const size_t out_bytes = net->act_elems.back() * sizeof(float);
  if (!net->d_in) {
    if (cudaMalloc(&net->d_in, in_bytes) != cudaSuccess || cudaMalloc(&net->d_out, out_bytes) != cudaSuccess) {
      cudaGetLastError();
      cudaFree(net->d_in);
      net->d_in = nullptr;
      return PP_ERR_OOM;
    }
  }
  // With graphs on and page-locked host buffers, the input copy, the ops and
  // the output copy are captured once per (x_host, y_host, stream) and each
  // call is one graph launch; otherwise they are issued one by one.
  if (net->use_graph && stream != nullptr && is_pinned(x_host) && is_pinned(y_host)) {
    if (!net->hexec || net->h_x != x_host || net->h_y != y_host || net->h_stream != stream) {
      if (net->hexec) {
        cudaGraphExecDestroy(net->hexec);
        net->hexec = nullptr;
      }
      cudaGraph_t g = nullptr;
      if (cudaStreamBeginCapture(stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) return PP_ERR_CUDA;
      pp_status st = PP_OK;
      if (cudaMemcpyAsync(net->d_in, x_host, in_bytes, cudaMemcpyHostToDevice, stream) != cudaSuccess)
        st = PP_ERR_CUDA;
      if (st == PP_OK) st = run_ops(net, net->d_in, net->d_out, stream);
      if (st == PP_OK &&
          cudaMemcpyAsync(y_host, net->d_out, out_bytes, cudaMemcpyDeviceToHost, stream) != cudaSuccess)
        st = PP_ERR_CUDA;
      cudaError_t ce = cudaStreamEndCapture(stream, &g);
      if (st != PP_OK || ce != cudaSuccess) {
        if (g) cudaGraphDestroy(g);
        cudaGetLastError();
        return st != PP_OK ? st : PP_ERR_CUDA;
      }
      ce = cudaGraphInstantiate(&net->hexec, g, 0);
      cudaGraphDestroy(g);
      if (ce != cudaSuccess) {
        net->hexec = nullptr;
        return PP_ERR_CUDA;
      }
      net->h_x = x_host;
      net->h_y = y_host;
      net->h_stream = stream;
    }
    if (cudaGraphLaunch(net->hexec, stream) != cudaSuccess) return PP_ERR_CUDA;
    return cudaStreamSynchronize(stream) == cudaSuccess ? PP_OK : PP_ERR_CUDA;
  }
  if (cudaMemcpyAsync(net->d_in, x_host, in_bytes, cudaMemcpyHostToDevice, stream) != cudaSuccess)
    return PP_ERR_CUDA;
  pp_status st = pp_net_run(net, net->d_in, net->d_out, stream_);
  if (st != PP_OK) return st;
  if (cudaMemcpyAsync(y_host, net->d_out, out_bytes, cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    return PP_ERR_CUDA;
  return cudaStreamSynchronize(stream) == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

extern "C" void pp_net_destroy(pp_net* net) {
  if (!net) return;
  if (net->gexec) cudaGraphExecDestroy(net->gexec);
  if (net->hexec) cudaGraphExecDestroy(net->hexec);
  for (float* p : net->buffers) cudaFree(p);
  cudaFree(net->d_in);
  cudaFree(net->d_out);
  delete net;
}
