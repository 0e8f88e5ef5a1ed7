// Host packer: validation, pattern-id inference, compact storage and filter
// reorder of a pattern- and connectivity-pruned 3x3 layer.
//
// Section 2 (Niu et al., IJCAI-20 demo): connectivity pruning removes whole
// kernels; pattern pruning keeps certain locations of each kernel.  Section 3:
// the sparse model is stored without zeros and without the indices the
// structure makes redundant (a kept kernel is a pattern id plus 4 weights), and
// "matrix reorder" sorts filters so that similar ones sit together and then
// compacts each filter's kept kernels.  The exact sort keys are this library's
// reading (documented at pp_pack_layer in ppconv.h): the paper names the goal
// (load balance, regular access) but not the key.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <numeric>

#include "internal.h"

namespace ppc {

uint16_t tap_mask(const uint8_t* taps4) {
  uint16_t m = 0;
  for (int s = 0; s < 4; ++s) m |= uint16_t(1u << taps4[s]);
  return m;
}

}  // namespace ppc

namespace {

pp_status check_pattern_set(const uint8_t* taps, int P) {
  if (P < 1 || P > 126) return PP_ERR_BAD_PATTERN_SET;
  std::vector<uint16_t> seen;
  seen.reserve(P);
  for (int p = 0; p < P; ++p) {
    const uint8_t* t = taps + 4 * p;
    for (int s = 0; s < 4; ++s) {
      if (t[s] > 8) return PP_ERR_BAD_PATTERN_SET;
      if (s && t[s] <= t[s - 1]) return PP_ERR_BAD_PATTERN_SET;
    }
    uint16_t m = ppc::tap_mask(t);
    if (std::find(seen.begin(), seen.end(), m) != seen.end()) return PP_ERR_BAD_PATTERN_SET;
    seen.push_back(m);
  }
  return PP_OK;
}

}  // namespace

extern "C" pp_status pp_pack_layer(const float* w, const uint8_t* mask, const uint8_t* pattern_taps, int P, int Co,
                                   int Ci, const uint8_t* pattern_ids, pp_packed** out) {
  if (!w || !mask || !pattern_taps || !out || Co < 1 || Ci < 1) return PP_ERR_INVALID_ARG;
  if ((int64_t)Co * Ci > (int64_t(1) << 30)) return PP_ERR_UNSUPPORTED;
  pp_status st = check_pattern_set(pattern_taps, P);
  if (st != PP_OK) return st;

  const size_t nker = size_t(Co) * Ci;
  std::vector<uint16_t> pmask(P);
  for (int p = 0; p < P; ++p) pmask[p] = ppc::tap_mask(pattern_taps + 4 * p);

  // Pattern id per kernel: 9-bit support of nonzero taps, matched against the
  // pattern masks (subset test).  -1 marks a pruned kernel.
  std::vector<int16_t> pid(nker, -1);
  for (size_t k = 0; k < nker; ++k) {
    const float* wk = w + k * 9;
    uint16_t support = 0;
    for (int t = 0; t < 9; ++t)
      if (wk[t] != 0.0f) support |= uint16_t(1u << t);
    if (!mask[k]) {
      if (support) return PP_ERR_PRUNED_NONZERO;
      continue;
    }
    if (pattern_ids) {
      int g = pattern_ids[k];
      if (g >= P || (support & ~pmask[g])) return PP_ERR_PATTERN_ID_MISMATCH;
      pid[k] = int16_t(g);
      continue;
    }
    int found = -1;
    for (int p = 0; p < P; ++p)
      if ((support & ~pmask[p]) == 0) {
        found = p;
        break;
      }
    if (found < 0) return PP_ERR_TAP_NOT_IN_PATTERN;
    pid[k] = int16_t(found);
  }

  pp_packed* pk = new (std::nothrow) pp_packed;
  if (!pk) return PP_ERR_OOM;
  try {
    pk->Co = Co;
    pk->Ci = Ci;
    pk->P = P;
    pk->taps.assign(pattern_taps, pattern_taps + 4 * P);

    // Per filter: kept count and pattern histogram -> dominant pattern.
    std::vector<int64_t> cnt(Co, 0);
    std::vector<int> dom(Co, 0);
    std::vector<int64_t> hist(P);
    for (int o = 0; o < Co; ++o) {
      std::fill(hist.begin(), hist.end(), 0);
      for (int i = 0; i < Ci; ++i) {
        int p = pid[size_t(o) * Ci + i];
        if (p >= 0) ++hist[p];
      }
      cnt[o] = std::accumulate(hist.begin(), hist.end(), int64_t(0));
      dom[o] = int(std::max_element(hist.begin(), hist.end()) - hist.begin());  // first maximum
    }
    pk->perm.resize(Co);
    std::iota(pk->perm.begin(), pk->perm.end(), 0);
    std::stable_sort(pk->perm.begin(), pk->perm.end(), [&](int a, int b) {
      if (cnt[a] != cnt[b]) return cnt[a] > cnt[b];
      return dom[a] < dom[b];
    });

    // Compaction: bucket each filter's kept kernels by pattern id; within a
    // bucket the input channels arrive in ascending order.
    int64_t nk = std::accumulate(cnt.begin(), cnt.end(), int64_t(0));
    if (nk > INT32_MAX) {
      delete pk;
      return PP_ERR_UNSUPPORTED;
    }
    pk->kptr.assign(Co + 1, 0);
    pk->kidx.resize(nk);
    pk->kpat.resize(nk);
    pk->kw.resize(size_t(nk) * 4);
    std::vector<int32_t> start(P + 1);
    int64_t base = 0;
    for (int j = 0; j < Co; ++j) {
      const int o = pk->perm[j];
      std::fill(start.begin(), start.end(), 0);
      for (int i = 0; i < Ci; ++i) {
        int p = pid[size_t(o) * Ci + i];
        if (p >= 0) ++start[p + 1];
      }
      for (int p = 0; p < P; ++p) start[p + 1] += start[p];
      for (int i = 0; i < Ci; ++i) {
        const size_t k = size_t(o) * Ci + i;
        int p = pid[k];
        if (p < 0) continue;
        int64_t e = base + start[p]++;
        pk->kidx[e] = i;
        pk->kpat[e] = uint8_t(p);
        const uint8_t* t = pattern_taps + 4 * p;
        for (int s = 0; s < 4; ++s) pk->kw[size_t(e) * 4 + s] = w[k * 9 + t[s]];
      }
      base += cnt[o];
      pk->kptr[j + 1] = int32_t(base);
    }
  } catch (const std::bad_alloc&) {
    delete pk;
    return PP_ERR_OOM;
  }
  *out = pk;
  return PP_OK;
}

extern "C" pp_status pp_packed_info(const pp_packed* pk, int64_t* nk, int* Co, int* Ci, int* P) {
  if (!pk) return PP_ERR_INVALID_ARG;
  if (nk) *nk = int64_t(pk->kidx.size());
  if (Co) *Co = pk->Co;
  if (Ci) *Ci = pk->Ci;
  if (P) *P = pk->P;
  return PP_OK;
}

extern "C" pp_status pp_packed_arrays(const pp_packed* pk, const int32_t** perm, const int32_t** kptr,
                                      const int32_t** kidx, const uint8_t** kpat, const float** kw,
                                      const uint8_t** taps) {
  if (!pk) return PP_ERR_INVALID_ARG;
  if (perm) *perm = pk->perm.data();
  if (kptr) *kptr = pk->kptr.data();
  if (kidx) *kidx = pk->kidx.data();
  if (kpat) *kpat = pk->kpat.data();
  if (kw) *kw = pk->kw.data();
  if (taps) *taps = pk->taps.data();
  return PP_OK;
}

extern "C" pp_status pp_unpack_layer(const pp_packed* pk, float* w_out, uint8_t* mask_out) {
  if (!pk) return PP_ERR_INVALID_ARG;
  const size_t nker = size_t(pk->Co) * pk->Ci;
  if (w_out) std::memset(w_out, 0, nker * 9 * sizeof(float));
  if (mask_out) std::memset(mask_out, 0, nker);
  for (int j = 0; j < pk->Co; ++j) {
    const int o = pk->perm[j];
    for (int32_t e = pk->kptr[j]; e < pk->kptr[j + 1]; ++e) {
      const size_t k = size_t(o) * pk->Ci + pk->kidx[e];
      if (mask_out) mask_out[k] = 1;
      if (w_out) {
        const uint8_t* t = &pk->taps[4 * pk->kpat[e]];
        for (int s = 0; s < 4; ++s) w_out[k * 9 + t[s]] = pk->kw[size_t(e) * 4 + s];
      }
    }
  }
  return PP_OK;
}

extern "C" void pp_packed_destroy(pp_packed* pk) { delete pk; }

extern "C" pp_status pp_fold_batchnorm(float* w, float* bias, const float* gamma, const float* beta,
                                       const float* mean, const float* var, float eps, int Co, int Ci) {
  if (!w || !bias || !gamma || !beta || !mean || !var || Co < 1 || Ci < 1 || !(eps >= 0.f))
    return PP_ERR_INVALID_ARG;
  for (int o = 0; o < Co; ++o)
    if (!(double(var[o]) + eps > 0.0)) return PP_ERR_INVALID_ARG;
  for (int o = 0; o < Co; ++o) {
    // y = gamma (z - mean) / sqrt(var + eps) + beta with z = conv + bias: one scale per filter, so a
    // zero weight stays zero and the layer keeps its patterns and connectivity
    const double scale = double(gamma[o]) / std::sqrt(double(var[o]) + double(eps));
    float* k = w + size_t(o) * Ci * 9;
    for (size_t t = 0; t < size_t(Ci) * 9; ++t) k[t] = float(double(k[t]) * scale);
    bias[o] = float((double(bias[o]) - double(mean[o])) * scale + double(beta[o]));
  }
  return PP_OK;
}

extern "C" pp_status pp_permute_input_channels(const float* w, const uint8_t* mask, const uint8_t* pattern_ids,
                                               int Co, int Ci, const int32_t* layout, float* w_out,
                                               uint8_t* mask_out, uint8_t* ids_out) {
  if (!w || !layout || !w_out || Co < 1 || Ci < 1) return PP_ERR_INVALID_ARG;
  if ((mask_out && !mask) || (ids_out && !pattern_ids)) return PP_ERR_INVALID_ARG;
  std::vector<uint8_t> seen(Ci, 0);
  for (int c = 0; c < Ci; ++c) {
    if (layout[c] < 0 || layout[c] >= Ci || seen[layout[c]]) return PP_ERR_INVALID_ARG;
    seen[layout[c]] = 1;
  }
  // position c of the permuted layer reads original input channel layout[c]
  for (int o = 0; o < Co; ++o)
    for (int c = 0; c < Ci; ++c) {
      const size_t src = size_t(o) * Ci + layout[c], dst = size_t(o) * Ci + c;
      std::memcpy(w_out + dst * 9, w + src * 9, 9 * sizeof(float));
      if (mask_out) mask_out[dst] = mask[src];
      if (ids_out) ids_out[dst] = pattern_ids[src];
    }
  return PP_OK;
}

extern "C" const char* pp_status_string(pp_status s) {
  switch (s) {
    case PP_OK: return "PP_OK";
    case PP_ERR_INVALID_ARG: return "PP_ERR_INVALID_ARG";
    case PP_ERR_BAD_PATTERN_SET: return "PP_ERR_BAD_PATTERN_SET";
    case PP_ERR_TAP_NOT_IN_PATTERN: return "PP_ERR_TAP_NOT_IN_PATTERN";
    case PP_ERR_PRUNED_NONZERO: return "PP_ERR_PRUNED_NONZERO";
    case PP_ERR_PATTERN_ID_MISMATCH: return "PP_ERR_PATTERN_ID_MISMATCH";
    case PP_ERR_UNSUPPORTED: return "PP_ERR_UNSUPPORTED";
    case PP_ERR_CUDA: return "PP_ERR_CUDA";
    case PP_ERR_OOM: return "PP_ERR_OOM";
    default: return "PP_ERR_UNKNOWN";
  }
}

extern "C" int pp_version(void) { return 100; }
