// libfgq C ABI: argument validation, kernel-family dispatch, the device error word and
// status reporting.  Every computation happens in the kernels of the other files.
#include <atomic>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "fgq_internal.h"

namespace fgq {
namespace {

__device__ unsigned int g_error_word;
constexpr int kReadSlots = 64;
__device__ unsigned int g_error_read[kReadSlots];  // the word's value at a read-and-clear, per call
std::atomic<unsigned int> g_read_slot{0};

constexpr int kMaxDevices = 64;
unsigned int* g_err_ptr[kMaxDevices];
std::mutex g_err_mu;
std::atomic<uint64_t> g_launches{0};
// test and benchmark controls (fgq_debug.h), each per host thread
thread_local int t_path = FGQ_PATH_AUTO;
thread_local int t_last_path = FGQ_PATH_AUTO;
thread_local int64_t t_wait_limit_us = -1;
thread_local int t_split_fold = 0;
thread_local int t_last_cuda_error = 0;  // cudaError_t of the last failed launch on this thread
thread_local int t_cta_pairs = 0;        // G = 4 output kernel on CTA pairs (off: single CTAs)
thread_local int t_max_ksplit = 8;       // group ranges a G >= 64 tile may be split into
thread_local int t_last_ksplit = 0;      // ranges of this thread's last G >= 64 tensor-core call

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

bool valid_type(int t) { return t == FGQ_U8 || t == FGQ_S8 || t == FGQ_U4 || t == FGQ_S4; }

bool valid_G(int G) {
  return G == 1 || G == 2 || G == 4 || G == 8 || G == 16 || G == 32 || G == 64 || G == 128;
}

bool is4(int t) { return t == FGQ_U4 || t == FGQ_S4; }

// Fill a Geom for a convolution; returns FGQ_OK or FGQ_ERR_ARG.
fgq_status make_geom(int type, int B, int H, int W, int C, int R, int S, int stride, int pad, int groups,
                     int M, int G, int is_conv, Geom& g) {
  if (!valid_type(type) || B < 0 || H <= 0 || W <= 0 || C <= 0 || R <= 0 || S <= 0 || stride <= 0 ||
      pad < 0 || groups <= 0 || M < 0 || C % groups != 0 || M % groups != 0 || G <= 0)
    return FGQ_ERR_ARG;
  if (is4(type) && (C % 2 != 0)) return FGQ_ERR_ARG;
  g.B = B; g.H = H; g.W = W; g.C = C; g.R = R; g.S = S; g.stride = stride; g.pad = pad; g.groups = groups;
  g.Ho = (H + 2 * pad - R) / stride + 1;
  g.Wo = (W + 2 * pad - S) / stride + 1;
  if (H + 2 * pad < R || W + 2 * pad < S || g.Ho <= 0 || g.Wo <= 0) return FGQ_ERR_ARG;
  g.Cg = C / groups;
  g.Kred = R * S * g.Cg;
  g.G = G;
  g.ng = (g.Kred + G - 1) / G;
  g.Kp = g.ng * G;
  g.wrow = (g.Kp + 15) / 16;
  g.M = M;
  g.Mg = groups ? M / groups : 0;
  g.act_type = type;
  g.is_conv = is_conv;
  g.P = (int64_t)B * g.Ho * g.Wo;
  g.rq_out = nullptr;
  g.rq_scale = nullptr;
  g.rq_signed = 0;
  return FGQ_OK;
}

bool tc_any(const Geom& g) { return g.G == 4 ? tc4_supports(g) : tc_supports(g); }

bool gemv_any(const Geom& g) { return !g.is_conv && gemv_supports((int)g.P, g.Kred, g.G, g.act_type); }

// Fewest filters per conv group for which the automatic choice sends a G = 4 layer to the
// tensor cores (a 64-filter layer fills half of the 128-row tile and still runs at about
// twice the dp4a kernel's rate).
constexpr int T4_MIN_FILTERS = 64;

int choose_path(const Geom& g, bool sums, bool qa) {
  const int forced = t_path;
  if (sums) {
    // the group sums come from the kernel family the output call of this shape would use;
    // the dense and few-row paths form no group sums
    if (forced == FGQ_PATH_GEMV || forced == FGQ_PATH_DENSE) return -1;
    if (forced == FGQ_PATH_SIMT) return FGQ_PATH_SIMT;
    if (forced == FGQ_PATH_TC) return tc_any(g) ? FGQ_PATH_TC : -1;
    if (g.G == 4 && g.Mg < T4_MIN_FILTERS) return FGQ_PATH_SIMT;
    return tc_any(g) ? FGQ_PATH_TC : FGQ_PATH_SIMT;
  }
  if (forced == FGQ_PATH_SIMT) return FGQ_PATH_SIMT;
  if (forced == FGQ_PATH_TC) return tc_any(g) ? FGQ_PATH_TC : -1;
  if (forced == FGQ_PATH_GEMV) return gemv_any(g) ? FGQ_PATH_GEMV : -1;
  // fp32 alphas fold only approximately (split into two fp16 parts): an ablation outside the
  // tolerance guarantee, run only when a test or benchmark asked for it
  if (forced == FGQ_PATH_DENSE) return dense_supports(g) && (qa || t_split_fold) ? FGQ_PATH_DENSE : -1;
  if (gemv_any(g)) return FGQ_PATH_GEMV;  // a few activation rows: stream the weights once
  // fixed-point alphas fold exactly into fp16 weights: one dense tensor-core contraction
  if (qa && dense_supports(g)) return FGQ_PATH_DENSE;
  // automatic choice: the tensor cores where the shape is covered, except G = 4 layers with
  // fewer than T4_MIN_FILTERS filters per conv group, where most rows of the 128-row MMA
  // tile would sit idle and the dp4a kernel is faster
  if (g.G == 4 && g.Mg < T4_MIN_FILTERS) return FGQ_PATH_SIMT;
  return tc_any(g) ? FGQ_PATH_TC : FGQ_PATH_SIMT;
}

// Fixed-point alphas of a contraction call (nullptr: fp32 alphas).
struct QAlpha {
  const uint8_t* aq;
  int bits;
  const float* ascale;
};

fgq_status contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                    const float* act_scale, float* out, int32_t* sums, cudaStream_t s, const QAlpha* qa = nullptr) {
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  const int path = choose_path(g, sums != nullptr, qa != nullptr);
  if (path < 0) return FGQ_ERR_UNSUPPORTED;
  t_last_path = path;
  unsigned int* err = device_error_word();
  if (path == FGQ_PATH_DENSE)
    return launch_dense_contract(act, g, codes, alpha, qa ? qa->aq : nullptr, qa ? qa->bits : 0,
                                 qa ? qa->ascale : nullptr, act_scale, out, err, s);
  if (path == FGQ_PATH_GEMV)
    return launch_gemv(act, g.act_type, (int)g.P, g.Kred, g.M, g.G, codes, alpha, qa ? qa->aq : nullptr,
                       qa ? qa->bits : 0, qa ? qa->ascale : nullptr, act_scale, out, g.rq_out, g.rq_scale,
                       g.rq_signed, s);
  float* a32 = nullptr;  // fixed-point alphas on the fp32-alpha kernels: alpha' = a 2^E, exact
  if (qa) {
    cudaMemPool_t pool = scratch_pool();
    if (!pool || cudaMallocFromPoolAsync(reinterpret_cast<void**>(&a32), sizeof(float) * (size_t)g.M * g.ng, pool, s) !=
                     cudaSuccess)
      return FGQ_ERR_CUDA;
    fgq_status st = launch_dequantize_alpha(qa->aq, qa->bits, g.M, g.ng, qa->ascale, a32, s);
    if (st != FGQ_OK) {
      cudaFreeAsync(a32, s);
      return st;
    }
    alpha = a32;
  }
  fgq_status st;
  if (path == FGQ_PATH_TC)
    st = g.G == 4 ? launch_tc4_contract(act, g, codes, alpha, act_scale, out, sums, err, s)
                  : launch_tc_contract(act, g, codes, alpha, act_scale, out, sums, err, s);
  else
    st = launch_simt_contract(act, g, codes, alpha, 0, act_scale, out, sums, s);
  if (a32 && cudaFreeAsync(a32, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

}  // namespace

cudaMemPool_t scratch_pool() {
  static std::mutex mu;
  static cudaMemPool_t pools[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if (!pools[dev]) {
    cudaMemPoolProps props;
    memset(&props, 0, sizeof props);
    props.allocType = cudaMemAllocationTypePinned;
    props.location.type = cudaMemLocationTypeDevice;
    props.location.id = dev;
    cudaMemPool_t p = nullptr;
    if (cudaMemPoolCreate(&p, &props) != cudaSuccess) return nullptr;
    uint64_t keep = ~0ull;
    cudaMemPoolSetAttribute(p, cudaMemPoolAttrReleaseThreshold, &keep);
    pools[dev] = p;
  }
  return pools[dev];
}

unsigned int* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_err_mu);
  if (!g_err_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
    g_err_ptr[dev] = static_cast<unsigned int*>(p);
  }
  return g_err_ptr[dev];
}

fgq_status after_launch() {
  g_launches.fetch_add(1);
  const cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) return FGQ_OK;
  t_last_cuda_error = (int)e;
  return FGQ_ERR_CUDA;
}

fgq_status after_launch(cudaError_t launch_result) {
  const fgq_status st = after_launch();
  if (launch_result == cudaSuccess) return st;
  t_last_cuda_error = (int)launch_result;
  return FGQ_ERR_CUDA;
}

int64_t debug_wait_limit_us() { return t_wait_limit_us; }

bool debug_cta_pairs() { return t_cta_pairs != 0; }

int debug_max_ksplit() { return t_max_ksplit; }

void note_ksplit(int k) { t_last_ksplit = k; }

namespace {

// Reads and clears the error word in one atomic step, so that an error a kernel on another
// stream records concurrently is either returned now or kept for the next read.
__global__ void error_read_clear_kernel(unsigned int slot) { g_error_read[slot] = atomicExch(&g_error_word, 0u); }

}  // namespace

}  // namespace fgq

namespace fgq {
namespace {

// Byte offsets of the regions of fgq_conv2d_host's workspace (each 256-byte aligned).
struct HostLayout {
  size_t w, x, codes, alpha, q, scale, qws, out, total, qws_bytes;
};

size_t up256(size_t v) { return (v + 255) & ~size_t(255); }

HostLayout host_layout(const Geom& g) {
  HostLayout L;
  const size_t n = (size_t)g.B * g.H * g.W * g.C;
  const bool w8 = g.G == 0;
  size_t o = 0;
  L.w = o;     o = up256(o + sizeof(float) * (size_t)g.M * g.Kred);
  L.x = o;     o = up256(o + sizeof(float) * n);
  L.codes = o; o = up256(o + (w8 ? (size_t)g.M * g.Kred : sizeof(uint32_t) * (size_t)g.M * g.wrow));
  L.alpha = o; o = up256(o + sizeof(float) * (size_t)g.M * (w8 ? 1 : g.ng));
  L.q = o;     o = up256(o + (is4(g.act_type) ? (n + 1) / 2 : n));
  L.scale = o; o = up256(o + sizeof(float));
  L.qws_bytes = quantize_workspace_bytes(n);
  L.qws = o;   o = up256(o + L.qws_bytes);
  L.out = o;   o = up256(o + sizeof(float) * (size_t)g.P * g.M);
  L.total = o;
  return L;
}

// Geometry of a host call (G == 0: the 8-bit-weight layer, 8-bit activations only).
fgq_status host_geom(fgq_act_type type, int B, int H, int W, int C, int R, int S, int stride, int pad, int groups,
                     int M, int G, Geom& g) {
  if (G != 0 && !valid_G(G)) return FGQ_ERR_ARG;
  if (G == 0 && type != FGQ_U8 && type != FGQ_S8) return FGQ_ERR_ARG;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G == 0 ? 1 : G, 1, g);
  if (st != FGQ_OK) return st;
  if (G == 0) {  // dense 8-bit weights: no groups
    g.G = 0;
    g.ng = 1;
    g.Kp = g.Kred;
    g.wrow = 0;
  }
  return FGQ_OK;
}

}  // namespace
}  // namespace fgq

using namespace fgq;

extern "C" {

int fgq_version(void) { return 1; }

const char* fgq_status_string(fgq_status s) {
  switch (s) {
    case FGQ_OK: return "FGQ_OK";
    case FGQ_ERR_ARG: return "FGQ_ERR_ARG: invalid argument";
    case FGQ_ERR_ALIGN: return "FGQ_ERR_ALIGN: misaligned pointer";
    case FGQ_ERR_UNSUPPORTED: return "FGQ_ERR_UNSUPPORTED: unsupported shape or path";
    case FGQ_ERR_NONFINITE: return "FGQ_ERR_NONFINITE: NaN or Inf in input";
    case FGQ_ERR_TIMEOUT: return "FGQ_ERR_TIMEOUT: a bounded wait ran out";
    case FGQ_ERR_CUDA: return "FGQ_ERR_CUDA: CUDA error";
  }
  return "unknown fgq_status";
}

int64_t fgq_codes_words_per_row(int Kred, int G) {
  if (Kred < 0 || !valid_G(G)) return 0;
  const int64_t ng = ((int64_t)Kred + G - 1) / G;
  return (ng * G + 15) / 16;
}

int64_t fgq_num_groups(int Kred, int G) {
  if (Kred < 0 || !valid_G(G)) return 0;
  return ((int64_t)Kred + G - 1) / G;
}

fgq_status fgq_ternarize(const float* w, int M, int Kred, int G, uint32_t* codes, float* alpha,
                         cudaStream_t stream) {
  if (M < 0 || Kred < 0 || !valid_G(G)) return FGQ_ERR_ARG;
  if ((int64_t)M * Kred == 0) return FGQ_OK;
  if (!w || !codes || !alpha) return FGQ_ERR_ARG;
  if (!aligned(w, 4) || !aligned(codes, 4) || !aligned(alpha, 4)) return FGQ_ERR_ALIGN;
  if ((int64_t)Kred + G > INT32_MAX) return FGQ_ERR_ARG;
  return launch_ternarize(w, M, Kred, G, codes, alpha, device_error_word(), stream);
}

fgq_status fgq_ternarize_batch(int n, const float* const* w, const int* M, const int* Kred, int G,
                               uint32_t* const* codes, float* const* alpha, cudaStream_t stream) {
  if (n < 0 || n > FGQ_TERNARIZE_BATCH_MAX || !valid_G(G)) return FGQ_ERR_ARG;
  if (n == 0) return FGQ_OK;
  if (!w || !M || !Kred || !codes || !alpha) return FGQ_ERR_ARG;
  for (int i = 0; i < n; ++i) {
    if (M[i] < 0 || Kred[i] < 0 || (int64_t)Kred[i] + G > INT32_MAX) return FGQ_ERR_ARG;
    if ((int64_t)M[i] * Kred[i] == 0) continue;
    if (!w[i] || !codes[i] || !alpha[i]) return FGQ_ERR_ARG;
    if (!aligned(w[i], 4) || !aligned(codes[i], 4) || !aligned(alpha[i], 4)) return FGQ_ERR_ALIGN;
  }
  return launch_ternarize_batch(n, w, M, Kred, G, codes, alpha, device_error_word(), stream);
}

size_t fgq_ternarize_threshold_workspace_bytes(void) { return threshold_workspace_bytes(); }

fgq_status fgq_ternarize_threshold(const float* w, int M, int Kred, int G, int rule, int per_layer, uint32_t* codes,
                                   float* alpha, void* workspace, size_t workspace_bytes, double* delta_out,
                                   cudaStream_t stream) {
  if (M < 0 || Kred < 0 || !valid_G(G) || (rule != FGQ_RULE_EXP && rule != FGQ_RULE_GAUSS)) return FGQ_ERR_ARG;
  if ((int64_t)M * Kred == 0) return FGQ_OK;
  if (!w || !codes || !alpha) return FGQ_ERR_ARG;
  if (!aligned(w, 4) || !aligned(codes, 4) || !aligned(alpha, 4)) return FGQ_ERR_ALIGN;
  if ((int64_t)Kred + G > INT32_MAX) return FGQ_ERR_ARG;
  if (per_layer) {
    if (!workspace || workspace_bytes < threshold_workspace_bytes()) return FGQ_ERR_ARG;
    if (!aligned(workspace, 16) || (delta_out && !aligned(delta_out, 8))) return FGQ_ERR_ALIGN;
  }
  return launch_ternarize_threshold(w, M, Kred, G, rule, per_layer ? 1 : 0, codes, alpha, workspace,
                                    per_layer ? delta_out : nullptr, device_error_word(), stream);
}

fgq_status fgq_ternary_error(const float* w, int M, int Kred, int G, const uint32_t* codes, const float* alpha,
                             double* err, cudaStream_t stream) {
  if (M < 0 || Kred < 0 || !valid_G(G)) return FGQ_ERR_ARG;
  if ((int64_t)M * Kred == 0) return FGQ_OK;
  if (!w || !codes || !alpha || !err) return FGQ_ERR_ARG;
  if (!aligned(w, 4) || !aligned(codes, 4) || !aligned(alpha, 4) || !aligned(err, 8)) return FGQ_ERR_ALIGN;
  if ((int64_t)Kred + G > INT32_MAX) return FGQ_ERR_ARG;
  return launch_ternary_error(w, M, Kred, G, codes, alpha, err, stream);
}

size_t fgq_quantize_act_workspace_bytes(size_t n) { return quantize_workspace_bytes(n); }

fgq_status fgq_quantize_act(const float* x, size_t n, fgq_act_type type, float scale_in, void* q,
                            float* scale_out, void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  if (!valid_type(type)) return FGQ_ERR_ARG;
  int E = 0;
  const bool derive = !(scale_in > 0.0f);
  if (!derive) {  // the given scale must be a power of two 2^E (subnormal ones included)
    uint32_t b;
    memcpy(&b, &scale_in, sizeof b);
    const uint32_t ex = b >> 23, man = b & 0x7fffffu;
    if (ex == 255) return FGQ_ERR_ARG;
    if (ex > 0) {
      if (man != 0) return FGQ_ERR_ARG;
      E = (int)ex - 127;
    } else {
      if (man & (man - 1)) return FGQ_ERR_ARG;
      E = -149 + (31 - __builtin_clz(man));
    }
  }
  if (n == 0) return FGQ_OK;  // nothing is written
  if (!x || !q || (derive && (!scale_out || !workspace))) return FGQ_ERR_ARG;
  if (!aligned(x, 16) || !aligned(q, 16) || (scale_out && !aligned(scale_out, 4))) return FGQ_ERR_ALIGN;
  if (derive) {
    if (!aligned(workspace, 4)) return FGQ_ERR_ALIGN;
    if (workspace_bytes < quantize_workspace_bytes(n)) return FGQ_ERR_ARG;
  }
  return launch_quantize(x, n, type, E, derive, q, scale_out, static_cast<uint32_t*>(workspace),
                         device_error_word(), stream);
}

size_t fgq_quantize_act_batch_workspace_bytes(int n) {
  return n < 0 || n > FGQ_QUANTIZE_BATCH_MAX ? 0 : quantize_batch_workspace_bytes(n);
}

fgq_status fgq_quantize_act_batch(int n, const float* const* x, const size_t* nelem, const fgq_act_type* type,
                                  void* const* q, float* const* scale_out, void* workspace, size_t workspace_bytes,
                                  cudaStream_t stream) {
  if (n < 0 || n > FGQ_QUANTIZE_BATCH_MAX) return FGQ_ERR_ARG;
  if (n == 0) return FGQ_OK;
  if (!x || !nelem || !type || !q || !scale_out) return FGQ_ERR_ARG;
  if (!workspace || workspace_bytes < quantize_batch_workspace_bytes(n)) return FGQ_ERR_ARG;
  if (!aligned(workspace, 4)) return FGQ_ERR_ALIGN;
  int types[FGQ_QUANTIZE_BATCH_MAX];
  for (int i = 0; i < n; ++i) {
    if (!valid_type(type[i])) return FGQ_ERR_ARG;
    types[i] = type[i];
    if (nelem[i] == 0) continue;
    if (!x[i] || !q[i] || !scale_out[i]) return FGQ_ERR_ARG;
    if (!aligned(x[i], 16) || !aligned(q[i], 16) || !aligned(scale_out[i], 4)) return FGQ_ERR_ALIGN;
  }
  return launch_quantize_batch(n, x, nelem, types, q, scale_out, static_cast<unsigned int*>(workspace),
                               device_error_word(), stream);
}

fgq_status fgq_quantize_weights_w8(const float* w, int M, int Kred, int8_t* wq, float* wscale,
                                   cudaStream_t stream) {
  if (M < 0 || Kred < 0) return FGQ_ERR_ARG;
  if ((int64_t)M * Kred == 0) return FGQ_OK;
  if (!w || !wq || !wscale) return FGQ_ERR_ARG;
  if (!aligned(w, 4) || !aligned(wscale, 4)) return FGQ_ERR_ALIGN;
  return launch_quantize_weights_w8(w, M, Kred, wq, wscale, device_error_word(), stream);
}

fgq_status fgq_gemm(const void* q, fgq_act_type type, const float* act_scale, int P, int Kred,
                    const uint32_t* codes, const float* alpha, int M, int G, float* y, cudaStream_t stream) {
  if (!valid_G(G) || P < 0 || Kred <= 0 || M < 0) return FGQ_ERR_ARG;
  if (is4(type) && Kred % 2) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, P, 1, 1, Kred, 1, 1, 1, 0, 1, M, G, 0, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!q || !act_scale || !codes || !alpha || !y) return FGQ_ERR_ARG;
  if (!aligned(q, 16) || !aligned(codes, 16) || !aligned(alpha, 16) || !aligned(y, 16) || !aligned(act_scale, 4))
    return FGQ_ERR_ALIGN;
  return contract(q, g, codes, alpha, act_scale, y, nullptr, stream);
}

fgq_status fgq_conv2d(const void* act, fgq_act_type type, const float* act_scale, int B, int H, int W, int C,
                      int R, int S, int stride, int pad, int groups, const uint32_t* codes, const float* alpha,
                      int M, int G, float* out, cudaStream_t stream) {
  if (!valid_G(G)) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G, 1, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!act || !act_scale || !codes || !alpha || !out) return FGQ_ERR_ARG;
  if (!aligned(act, 16) || !aligned(codes, 16) || !aligned(alpha, 16) || !aligned(out, 16) ||
      !aligned(act_scale, 4))
    return FGQ_ERR_ALIGN;
  return contract(act, g, codes, alpha, act_scale, out, nullptr, stream);
}

fgq_status fgq_gemm_rq(const void* q, fgq_act_type type, const float* act_scale, int P, int Kred,
                       const uint32_t* codes, const float* alpha, int M, int G, fgq_act_type out_type,
                       const float* out_scale, void* out_q, cudaStream_t stream) {
  if (!valid_G(G) || P < 0 || Kred <= 0 || M < 0 || (out_type != FGQ_U8 && out_type != FGQ_S8)) return FGQ_ERR_ARG;
  if (is4(type) && Kred % 2) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, P, 1, 1, Kred, 1, 1, 1, 0, 1, M, G, 0, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!q || !act_scale || !codes || !alpha || !out_scale || !out_q) return FGQ_ERR_ARG;
  if (!aligned(q, 16) || !aligned(codes, 16) || !aligned(alpha, 16) || !aligned(out_q, 4) ||
      !aligned(act_scale, 4) || !aligned(out_scale, 4))
    return FGQ_ERR_ALIGN;
  g.rq_out = static_cast<uint8_t*>(out_q);
  g.rq_scale = out_scale;
  g.rq_signed = out_type == FGQ_S8;
  return contract(q, g, codes, alpha, act_scale, nullptr, nullptr, stream);
}

fgq_status fgq_conv2d_rq(const void* act, fgq_act_type type, const float* act_scale, int B, int H, int W, int C,
                         int R, int S, int stride, int pad, int groups, const uint32_t* codes, const float* alpha,
                         int M, int G, fgq_act_type out_type, const float* out_scale, void* out_q,
                         cudaStream_t stream) {
  if (!valid_G(G) || (out_type != FGQ_U8 && out_type != FGQ_S8)) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G, 1, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!act || !act_scale || !codes || !alpha || !out_scale || !out_q) return FGQ_ERR_ARG;
  if (!aligned(act, 16) || !aligned(codes, 16) || !aligned(alpha, 16) || !aligned(out_q, 4) ||
      !aligned(act_scale, 4) || !aligned(out_scale, 4))
    return FGQ_ERR_ALIGN;
  g.rq_out = static_cast<uint8_t*>(out_q);
  g.rq_scale = out_scale;
  g.rq_signed = out_type == FGQ_S8;
  return contract(act, g, codes, alpha, act_scale, nullptr, nullptr, stream);
}

fgq_status fgq_quantize_alpha(const float* alpha, int M, int ng, int bits, uint8_t* aq, float* ascale,
                              cudaStream_t stream) {
  if (M < 0 || ng < 0 || (bits != 8 && bits != 4)) return FGQ_ERR_ARG;
  if ((int64_t)M * ng == 0) return FGQ_OK;
  if (!alpha || !aq || !ascale) return FGQ_ERR_ARG;
  if (!aligned(alpha, 4) || !aligned(ascale, 4)) return FGQ_ERR_ALIGN;
  return launch_quantize_alpha(alpha, M, ng, bits, aq, ascale, device_error_word(), stream);
}

fgq_status fgq_gemm_qa(const void* q, fgq_act_type type, const float* act_scale, int P, int Kred,
                       const uint32_t* codes, const uint8_t* aq, int abits, const float* ascale, int M, int G,
                       float* y, cudaStream_t stream) {
  if (!valid_G(G) || P < 0 || Kred <= 0 || M < 0 || (abits != 8 && abits != 4)) return FGQ_ERR_ARG;
  if (is4(type) && Kred % 2) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, P, 1, 1, Kred, 1, 1, 1, 0, 1, M, G, 0, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!q || !act_scale || !codes || !aq || !ascale || !y) return FGQ_ERR_ARG;
  if (!aligned(q, 16) || !aligned(codes, 16) || !aligned(y, 16) || !aligned(act_scale, 4) || !aligned(ascale, 4))
    return FGQ_ERR_ALIGN;
  const QAlpha qa{aq, abits, ascale};
  return contract(q, g, codes, nullptr, act_scale, y, nullptr, stream, &qa);
}

fgq_status fgq_conv2d_qa(const void* act, fgq_act_type type, const float* act_scale, int B, int H, int W, int C,
                         int R, int S, int stride, int pad, int groups, const uint32_t* codes, const uint8_t* aq,
                         int abits, const float* ascale, int M, int G, float* out, cudaStream_t stream) {
  if (!valid_G(G) || (abits != 8 && abits != 4)) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G, 1, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!act || !act_scale || !codes || !aq || !ascale || !out) return FGQ_ERR_ARG;
  if (!aligned(act, 16) || !aligned(codes, 16) || !aligned(out, 16) || !aligned(act_scale, 4) ||
      !aligned(ascale, 4))
    return FGQ_ERR_ALIGN;
  const QAlpha qa{aq, abits, ascale};
  return contract(act, g, codes, nullptr, act_scale, out, nullptr, stream, &qa);
}

fgq_status fgq_conv2d_w8(const void* act, fgq_act_type type, const float* act_scale, int B, int H, int W, int C,
                         int R, int S, int stride, int pad, int groups, const int8_t* wq, const float* wscale,
                         int M, float* out, cudaStream_t stream) {
  Geom g;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, 4, 1, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!act || !act_scale || !wq || !wscale || !out) return FGQ_ERR_ARG;
  if (!aligned(act, 16) || !aligned(wscale, 4) || !aligned(out, 16) || !aligned(act_scale, 4))
    return FGQ_ERR_ALIGN;
  if (t_path != FGQ_PATH_SIMT && dense_w8_supports(g)) {
    t_last_path = FGQ_PATH_DENSE;
    return launch_dense_w8(act, g, wq, wscale, act_scale, out, device_error_word(), stream);
  }
  t_last_path = FGQ_PATH_SIMT;
  return launch_simt_contract(act, g, wq, wscale, 1, act_scale, out, nullptr, stream);
}

fgq_status fgq_conv2d_w8_rq(const void* act, fgq_act_type type, const float* act_scale, int B, int H, int W, int C,
                            int R, int S, int stride, int pad, int groups, const int8_t* wq, const float* wscale,
                            int M, fgq_act_type out_type, const float* out_scale, void* out_q, cudaStream_t stream) {
  if (out_type != FGQ_U8 && out_type != FGQ_S8) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, 4, 1, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!act || !act_scale || !wq || !wscale || !out_scale || !out_q) return FGQ_ERR_ARG;
  if (!aligned(act, 16) || !aligned(wscale, 4) || !aligned(out_q, 4) || !aligned(act_scale, 4) ||
      !aligned(out_scale, 4))
    return FGQ_ERR_ALIGN;
  g.rq_out = static_cast<uint8_t*>(out_q);
  g.rq_scale = out_scale;
  g.rq_signed = out_type == FGQ_S8;
  if (t_path != FGQ_PATH_SIMT && dense_w8_supports(g)) {
    t_last_path = FGQ_PATH_DENSE;
    return launch_dense_w8(act, g, wq, wscale, act_scale, nullptr, device_error_word(), stream);
  }
  t_last_path = FGQ_PATH_SIMT;
  return launch_simt_contract(act, g, wq, wscale, 1, act_scale, nullptr, nullptr, stream);
}

fgq_status fgq_maxpool_u8(const uint8_t* in, int B, int H, int W, int C, int R, int stride, int pad, uint8_t* out,
                          cudaStream_t stream) {
  if (B < 0 || H <= 0 || W <= 0 || C <= 0 || C % 4 || R <= 0 || stride <= 0 || pad < 0 || pad >= R ||
      H + 2 * pad < R || W + 2 * pad < R)
    return FGQ_ERR_ARG;
  if (B == 0) return FGQ_OK;
  if (!in || !out) return FGQ_ERR_ARG;
  if (!aligned(in, 4) || !aligned(out, 4)) return FGQ_ERR_ALIGN;
  return launch_maxpool_u8(in, B, H, W, C, R, stride, pad, out, stream);
}

fgq_status fgq_add_codes(const void* a, fgq_act_type a_type, const float* a_scale, const void* b,
                         fgq_act_type b_type, const float* b_scale, size_t n, float* out, fgq_act_type out_type,
                         const float* out_scale, void* out_q, cudaStream_t stream) {
  auto is8 = [](int t) { return t == FGQ_U8 || t == FGQ_S8; };
  if (!is8(a_type) || !is8(b_type) || (!out && !is8(out_type))) return FGQ_ERR_ARG;
  if (n == 0) return FGQ_OK;
  if (!a || !b || !a_scale || !b_scale || (!out && (!out_q || !out_scale))) return FGQ_ERR_ARG;
  if (!aligned(a_scale, 4) || !aligned(b_scale, 4) || (out && !aligned(out, 4)) ||
      (!out && !aligned(out_scale, 4)))
    return FGQ_ERR_ALIGN;
  return launch_add_codes(static_cast<const uint8_t*>(a), a_type == FGQ_S8, a_scale, static_cast<const uint8_t*>(b),
                          b_type == FGQ_S8, b_scale, (int64_t)n, out, out ? nullptr : static_cast<uint8_t*>(out_q),
                          out_scale, out_type == FGQ_S8, stream);
}

fgq_status fgq_group_sums(const void* q, fgq_act_type type, int P, int Kred, const uint32_t* codes, int M, int G,
                          int32_t* s, cudaStream_t stream) {
  if (!valid_G(G) || P < 0 || Kred <= 0 || M < 0) return FGQ_ERR_ARG;
  if (is4(type) && Kred % 2) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, P, 1, 1, Kred, 1, 1, 1, 0, 1, M, G, 0, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!q || !codes || !s) return FGQ_ERR_ARG;
  if (!aligned(q, 16) || !aligned(codes, 16) || !aligned(s, 4)) return FGQ_ERR_ALIGN;
  return contract(q, g, codes, nullptr, nullptr, nullptr, s, stream);
}

fgq_status fgq_conv2d_group_sums(const void* act, fgq_act_type type, int B, int H, int W, int C, int R, int S,
                                 int stride, int pad, int groups, const uint32_t* codes, int M, int G, int32_t* s,
                                 cudaStream_t stream) {
  if (!valid_G(G)) return FGQ_ERR_ARG;
  Geom g;
  fgq_status st = make_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G, 1, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!act || !codes || !s) return FGQ_ERR_ARG;
  if (!aligned(act, 16) || !aligned(codes, 16) || !aligned(s, 4)) return FGQ_ERR_ALIGN;
  return contract(act, g, codes, nullptr, nullptr, nullptr, s, stream);
}

size_t fgq_conv2d_host_workspace_bytes(fgq_act_type type, int B, int H, int W, int C, int R, int S, int stride,
                                       int pad, int groups, int M, int G) {
  Geom g;
  if (host_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G, g) != FGQ_OK) return 0;
  return host_layout(g).total;
}

fgq_status fgq_conv2d_host(const float* h_w, const float* h_x, fgq_act_type type, int B, int H, int W, int C, int R,
                           int S, int stride, int pad, int groups, int M, int G, float* h_out, void* workspace,
                           size_t workspace_bytes, cudaStream_t stream) {
  Geom g;
  fgq_status st = host_geom(type, B, H, W, C, R, S, stride, pad, groups, M, G, g);
  if (st != FGQ_OK) return st;
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  if (!h_w || !h_x || !h_out || !workspace) return FGQ_ERR_ARG;
  if (!aligned(workspace, 256)) return FGQ_ERR_ALIGN;
  const HostLayout L = host_layout(g);
  if (workspace_bytes < L.total) return FGQ_ERR_ARG;
  uint8_t* base = static_cast<uint8_t*>(workspace);
  float* w = reinterpret_cast<float*>(base + L.w);
  float* x = reinterpret_cast<float*>(base + L.x);
  float* alpha = reinterpret_cast<float*>(base + L.alpha);
  float* scale = reinterpret_cast<float*>(base + L.scale);
  float* out = reinterpret_cast<float*>(base + L.out);
  const size_t n = (size_t)g.B * g.H * g.W * g.C;
  // one copy per input buffer, in order on the stream
  if (cudaMemcpyAsync(w, h_w, sizeof(float) * (size_t)g.M * g.Kred, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      cudaMemcpyAsync(x, h_x, sizeof(float) * n, cudaMemcpyHostToDevice, stream) != cudaSuccess)
    return FGQ_ERR_CUDA;
  if (G == 0)
    st = fgq_quantize_weights_w8(w, g.M, g.Kred, reinterpret_cast<int8_t*>(base + L.codes), alpha, stream);
  else
    st = fgq_ternarize(w, g.M, g.Kred, G, reinterpret_cast<uint32_t*>(base + L.codes), alpha, stream);
  if (st != FGQ_OK) return st;
  st = fgq_quantize_act(x, n, type, 0.0f, base + L.q, scale, base + L.qws, L.qws_bytes, stream);
  if (st != FGQ_OK) return st;
  if (G == 0)
    st = fgq_conv2d_w8(base + L.q, type, scale, B, H, W, C, R, S, stride, pad, groups,
                       reinterpret_cast<const int8_t*>(base + L.codes), alpha, M, out, stream);
  else
    st = fgq_conv2d(base + L.q, type, scale, B, H, W, C, R, S, stride, pad, groups,
                    reinterpret_cast<const uint32_t*>(base + L.codes), alpha, M, G, out, stream);
  if (st != FGQ_OK) return st;
  if (cudaMemcpyAsync(h_out, out, sizeof(float) * (size_t)g.P * g.M, cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    return FGQ_ERR_CUDA;
  return FGQ_OK;
}

fgq_status fgq_stream_status(cudaStream_t stream) {
  if (!device_error_word()) return FGQ_ERR_CUDA;
  // a slot of its own for each concurrent call (up to kReadSlots of them)
  const unsigned int slot = g_read_slot.fetch_add(1u) % kReadSlots;
  error_read_clear_kernel<<<1, 1, 0, stream>>>(slot);
  if (cudaGetLastError() != cudaSuccess) return FGQ_ERR_CUDA;
  unsigned int v = 0;
  if (cudaMemcpyFromSymbolAsync(&v, g_error_read, sizeof v, sizeof v * slot, cudaMemcpyDeviceToHost, stream) !=
          cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess)
    return FGQ_ERR_CUDA;
  return (fgq_status)v;
}

int fgq_set_path(int path) {
  if (path != FGQ_PATH_AUTO && path != FGQ_PATH_SIMT && path != FGQ_PATH_TC && path != FGQ_PATH_GEMV &&
      path != FGQ_PATH_DENSE)
    return -1;
  const int prev = t_path;
  t_path = path;
  return prev;
}

int64_t fgq_debug_set_wait_limit_us(int64_t us) {
  const int64_t prev = t_wait_limit_us;
  t_wait_limit_us = us < 0 ? -1 : us;
  return prev;
}

int fgq_debug_allow_split_fold(int allow) {
  const int prev = t_split_fold;
  t_split_fold = allow ? 1 : 0;
  return prev;
}

int fgq_debug_cta_pairs(int on) {
  const int prev = t_cta_pairs;
  t_cta_pairs = on ? 1 : 0;
  return prev;
}

int fgq_debug_max_ksplit(int k) {
  const int prev = t_max_ksplit;
  t_max_ksplit = k < 1 ? 1 : (k > 8 ? 8 : k);
  return prev;
}

int fgq_debug_last_ksplit(void) { return t_last_ksplit; }

int fgq_debug_last_cuda_error(char* name, size_t len) {
  const int e = t_last_cuda_error;
  t_last_cuda_error = 0;
  if (name && len > 0) {
    const char* n = e ? cudaGetErrorName((cudaError_t)e) : "";
    size_t i = 0;
    for (; n[i] && i + 1 < len; ++i) name[i] = n[i];
    name[i] = 0;
  }
  return e;
}

int fgq_last_path(void) { return t_last_path; }

uint64_t fgq_launch_count(void) { return g_launches.load(); }

fgq_status fgq_selftest_wait_timeout(uint32_t max_iterations, cudaStream_t stream) {
  return launch_wait_timeout_selftest(max_iterations, device_error_word(), stream);
}

}  // extern "C"
