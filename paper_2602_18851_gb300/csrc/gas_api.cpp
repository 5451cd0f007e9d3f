// C ABI of the library (include/gas.h): argument checks, workspace, TMA descriptor
// cache and the launch sequences of the two power-iteration back ends.

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "../../include/gas.h"
#include "gas_internal.h"

using gas::Shape;

struct gas_ctx {
  Shape s{};
  int device = 0;
  int num_sms = 0;
  int method = GAS_METHOD_AUTO;
  int seq_len = 1024;
  double eta_fp8 = 0.8;
  double alpha_override = 0.0;
  std::string err;
  int last_launches = 0;
  cudaStream_t last_stream = nullptr;
  std::vector<const char*> launch_names;  // kernels of the last call, in order
  std::vector<cudaEvent_t> events;        // optional timing brackets (caller-owned)

  // workspace (one allocation)
  void* ws = nullptr;
  size_t ws_bytes = 0;
  unsigned* status = nullptr;
  float* zp = nullptr;    // [L][nq][nch][dh]
  float* n2p = nullptr;   // [L][nq][nch]
  float* tp = nullptr;    // [L][nq][nch][dh]
  float* s2p = nullptr;   // [L][nq][nch]
  float* zr = nullptr;    // [L][nq][dh]  chunk sums of the streaming passes
  float* n2r = nullptr;   // [L][nq]
  float* tr = nullptr;    // [L][nq][dh]
  float* s2r = nullptr;   // [L][nq]
  uint16_t* vhl = nullptr;
  float* gq = nullptr;
  float* gk = nullptr;
  float* z0 = nullptr;
  float* ybuf = nullptr;
  CUtensorMap* dmaps = nullptr;  // [2L + 1]: q maps, k maps, v map
  unsigned* flags = nullptr;     // [L][tiles_k] key-tile flags of the fused kernel
  unsigned* vflags = nullptr;    // [L][tiles_k] v-norm flags of the fused kernel
  float* vn2 = nullptr;          // [L][nq] ||v||^2 of the start vectors (fused kernel)
  unsigned* layer_cnt = nullptr;  // [L] finished heads per layer of the fused kernel
  unsigned* done_cnt = nullptr;   // finished CTAs of the fused kernel
  unsigned long long* layer_max = nullptr;  // [L] epoch-tagged sigma maxima of the fused kernel
  float* lz = nullptr;           // whole-layer path: z_kv [L][n_kv*d_h]
  float* lu = nullptr;           //                   u'   [L][d]
  float* ly = nullptr;           //                   y    [L][n_q*d_h]
  float* lv = nullptr;           //                   v'   [L][d]
  unsigned* epoch = nullptr;     // device word: flag value of the fused Gram launches

  // host copies of the encoded descriptors and the pointers they were built for
  std::vector<CUtensorMap> hmaps;
  std::vector<const void*> map_q, map_k;
  bool maps_valid = false;
};

namespace {

thread_local std::string g_create_err;

gas_status fail(gas_ctx* h, gas_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  if (h) h->err = buf;
  else g_create_err = buf;
  return st;
}

gas_status cuda_fail(gas_ctx* h, cudaError_t e, const char* what) {
  return fail(h, GAS_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int round_up16(int x) { return (x + 15) / 16 * 16; }

// Resolved once per process (a function-local static: thread-safe initialisation).
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() -> PFN_cuTensorMapEncodeTiled_v12000 {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return nullptr;
  }();
  return fn;
}

// 2D bf16 map: inner dim `cols` (elements, contiguous), outer `rows`, box 64 x box_rows,
// 128-byte swizzle (the canonical K-major layout the tcgen05 descriptors expect).
bool encode_2d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 2D fp32 map of the start vectors [rows][d] (row-major): box 64 columns x box_rows rows,
// no swizzle (the fused Gram kernel's converter warps read the rows as loaded).
bool encode_vrows(CUtensorMap* m, const void* base, uint64_t d, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {d, rows};
  cuuint64_t strides[1] = {d * 4};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 3D bf16 map of one weight matrix: (column c, row i inside a head, head j) at
// base + j * hs + i * ld + c; box 64 columns x d_h rows x hpt heads (128 / tile head
// width), so a box fills the top d_h * hpt rows of one 128-row tile in the canonical
// K-major SW128 layout whatever the strides (all 128 rows unless d_h is 80 or 96).
bool encode_weights(CUtensorMap* m, const void* base, uint64_t d, uint32_t dh, uint64_t heads, uint64_t ld,
                    uint64_t hs, uint32_t hpt) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {d, dh, heads};
  cuuint64_t strides[2] = {ld * 2, hs * 2};
  cuuint32_t box[3] = {64, dh, hpt};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 2D bf16 map of a Conv1D weight matrix: element (row r, column c) at base + c * ld + r;
// box 64 rows x 64 columns (the rows are the contiguous, swizzled dimension).
bool encode_cols(CUtensorMap* m, const void* base, uint64_t rows, uint64_t d, uint64_t ld) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {rows, d};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

float scale_constant(const gas_ctx* h, double alpha, double r_max) {
  return static_cast<float>(alpha * (static_cast<double>(h->s.d) / std::sqrt(static_cast<double>(h->s.dh))) /
                            (h->eta_fp8 * r_max));
}

double h_fn(double g) { return g - 1.0 - std::log(g); }

gas_status check_weights(gas_ctx* h, const void* const* wq, const void* const* wk) {
  if (!wq || !wk) return fail(h, GAS_ERR_INVALID_ARG, "wq/wk pointer arrays must not be NULL");
  for (int l = 0; l < h->s.L; ++l) {
    if (!wq[l] || !wk[l]) return fail(h, GAS_ERR_INVALID_ARG, "layer %d: NULL weight pointer", l);
    if (!aligned16(wq[l]) || !aligned16(wk[l]))
      return fail(h, GAS_ERR_INVALID_ARG, "layer %d: weight pointers must be 16-byte aligned", l);
  }
  return GAS_OK;
}

gas_status ensure_maps(gas_ctx* h, const void* const* wq, const void* const* wk, cudaStream_t st) {
  const int L = h->s.L;
  bool same = h->maps_valid;
  for (int l = 0; same && l < L; ++l) same = (h->map_q[l] == wq[l] && h->map_k[l] == wk[l]);
  if (same) return GAS_OK;
  for (int l = 0; l < L; ++l) {
    const Shape& sh = h->s;
    const bool ok =
        sh.cols ? encode_cols(&h->hmaps[l], wq[l], static_cast<uint64_t>(sh.nq) * sh.dh, sh.d, sh.ldq) &&
                      encode_cols(&h->hmaps[L + l], wk[l], static_cast<uint64_t>(sh.nkv) * sh.dh, sh.d, sh.ldk)
                : encode_weights(&h->hmaps[l], wq[l], sh.d, sh.dh, sh.nq, sh.ldq, sh.hsq, sh.dh == 64 ? 2 : 1) &&
                      encode_weights(&h->hmaps[L + l], wk[l], sh.d, sh.dh, sh.nkv, sh.ldk, sh.hsk, sh.dh == 64 ? 2 : 1);
    if (!ok)
      return fail(h, GAS_ERR_CUDA, "cuTensorMapEncodeTiled failed for layer %d", l);
    h->map_q[l] = wq[l];
    h->map_k[l] = wk[l];
  }
  // The previous descriptors may still be read by work queued on `st`; the upload is
  // stream-ordered before the kernels that read it (pageable source: staged at call).
  cudaError_t e = cudaStreamSynchronize(st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->dmaps, h->hmaps.data(), sizeof(CUtensorMap) * (2 * L + 1), cudaMemcpyHostToDevice,
                        st);
  if (e != cudaSuccess) {
    h->maps_valid = false;
    return cuda_fail(h, e, "uploading TMA descriptors");
  }
  h->maps_valid = true;
  return GAS_OK;
}

void fill_table(const gas_ctx* h, gas::LayerTable& tab, const void* const* wq, const void* const* wk) {
  for (int l = 0; l < h->s.L; ++l) {
    tab.q[l] = static_cast<const uint16_t*>(wq[l]);
    tab.k[l] = static_cast<const uint16_t*>(wk[l]);
  }
}

// Every kernel launch of a call goes through here: records its name and, when the
// caller installed timing events, brackets it with them on the same stream.
template <typename F>
cudaError_t launch(gas_ctx* h, const char* name, cudaStream_t st, F&& fn) {
  const size_t i = h->launch_names.size();
  const bool timed = 2 * i + 1 < h->events.size();
  if (timed) cudaEventRecord(h->events[2 * i], st);
  cudaError_t e = fn();
  if (timed) cudaEventRecord(h->events[2 * i + 1], st);
  h->launch_names.push_back(name);
  return e;
}

// ---------------- streaming back end ----------------
gas_status run_stream(gas_ctx* h, const gas::LayerTable& tab, int iters, const float* v_in, float* v_out,
                      float* sigma, float* s_out, float scale_c, cudaStream_t st) {
  const Shape& s = h->s;
  int launches = 0;
  gas::StreamArgs a{};
  a.s = s;
  // K0: z = B_g v_in, ||v_in||^2
  a.mode = gas::kPassK0;
  a.out = h->zp;
  a.out2 = h->n2p;
  a.outr = h->zr;
  a.outr2 = h->n2r;
  a.status = h->status;
  a.v_in = v_in;
  a.s_zero = s_out;
  cudaError_t e = launch(h, "stream_pass_k0", st, [&] { return gas::launch_stream_pass(tab, a, st); });
  ++launches;
  if (e == cudaSuccess) {
    e = launch(h, "stream_reduce", st, [&] { return gas::launch_stream_reduce(a, st); });
    ++launches;
  }
  for (int it = 0; it < iters && e == cudaSuccess; ++it) {
    gas::StreamArgs q{};
    q.s = s;
    q.mode = gas::kPassQ;
    q.in_scaled = 1;
    q.in = h->zr;
    q.in2 = h->n2r;
    q.out = h->tp;
    q.out2 = h->s2p;
    q.outr = h->tr;
    q.outr2 = h->s2r;
    q.status = h->status;
    e = launch(h, "stream_pass_q", st, [&] { return gas::launch_stream_pass(tab, q, st); });
    ++launches;
    if (e == cudaSuccess) {
      e = launch(h, "stream_reduce", st, [&] { return gas::launch_stream_reduce(q, st); });
      ++launches;
    }
    if (e != cudaSuccess) break;
    const bool last = (it == iters - 1);
    if (last && v_out == nullptr) break;
    gas::StreamArgs k{};
    k.s = s;
    k.mode = last ? gas::kPassKOut : gas::kPassK;
    k.in_scaled = 1;
    k.in = h->tr;
    k.in2 = h->s2r;
    k.out = h->zp;
    k.out2 = h->n2p;
    k.outr = h->zr;
    k.outr2 = h->n2r;
    k.status = h->status;
    k.v_out = v_out;
    e = launch(h, last ? "stream_pass_kout" : "stream_pass_k", st,
               [&] { return gas::launch_stream_pass(tab, k, st); });
    ++launches;
    if (e == cudaSuccess) {
      e = launch(h, "stream_reduce", st, [&] { return gas::launch_stream_reduce(k, st); });
      ++launches;
    }
  }
  if (e == cudaSuccess) {
    gas::FinalizeArgs f{};
    f.s = s;
    f.s2 = h->s2r;
    f.n2 = h->n2r;
    f.v_out = v_out;
    f.sigma = sigma;
    f.scale_out = s_out;
    f.scale_c = scale_c;
    f.status = h->status;
    e = launch(h, "finalize", st, [&] { return gas::launch_finalize(f, st); });
    ++launches;
  }
  h->last_launches = launches;
  if (e != cudaSuccess) return cuda_fail(h, e, "streaming pass launch");
  return GAS_OK;
}

// ---------------- Gram back end ----------------
gas_status run_gram(gas_ctx* h, const void* const* wq, const void* const* wk, const gas::LayerTable& tab,
                    int iters, const float* v_in, float* v_out, float* sigma, float* s_out, float scale_c,
                    bool fused, cudaStream_t st) {
  // the tensor-core kernels see the tile head width (rows past the model's d_h are zero)
  Shape s = h->s;
  s.dh = s.rows == 64 ? 64 : 128;
  gas_status gs = ensure_maps(h, wq, wk, st);
  if (gs != GAS_OK) return gs;
  int launches = 0;
  cudaError_t e = cudaSuccess;
  gas::GramArgs g{};
  if (fused) {
    // the fused kernel reads the fp32 v rows itself, writes the per-layer scales without a
    // cleared accumulator and advances its flag epoch: it is the first launch of the call
    if (!encode_vrows(&g.map_vf, v_in, static_cast<uint64_t>(s.d), static_cast<uint64_t>(s.L) * s.nq,
                      static_cast<uint32_t>(s.nz / 2)))
      return fail(h, GAS_ERR_CUDA, "cuTensorMapEncodeTiled failed for v_in");
  } else {
    gas::PrepArgs p{};
    p.s = s;
    p.v_in = v_in;
    p.vhl = h->vhl;
    p.s_zero = s_out;
    p.epoch = h->epoch;
    e = launch(h, "prep_v", st, [&] { return gas::launch_prep_v(p, st); });
    ++launches;
  }
  if (e == cudaSuccess) {
    g.s = s;
    g.maps_q = h->dmaps;
    g.maps_k = h->dmaps + s.L;
    g.map_v = h->dmaps + 2 * s.L;
    g.gq = h->gq;
    g.gk = h->gk;
    g.z0 = h->z0;
    g.status = h->status;
    if (fused) {
      g.flags = h->flags;
      g.vflags = h->vflags;
      g.vn2 = h->vn2;
      g.epoch = h->epoch;
      g.layer_cnt = h->layer_cnt;
      g.layer_max = h->layer_max;
      g.done_cnt = h->done_cnt;
      g.iters = iters;
      g.ybuf = h->ybuf;
      g.sigma = sigma;
      g.scale_out = s_out;
      g.scale_c = scale_c;
    }
    e = launch(h, fused ? "gram_fused" : "gram", st, [&] { return gas::launch_gram(g, h->num_sms, fused, st); });
    ++launches;
  }
  if (e == cudaSuccess && !fused) {
    gas::IterArgs it{};
    it.s = s;
    it.iters = iters;
    it.gq = h->gq;
    it.gk = h->gk;
    it.z0 = h->z0;
    it.ybuf = h->ybuf;
    it.sigma = sigma;
    it.scale_out = s_out;
    it.scale_c = scale_c;
    it.status = h->status;
    e = launch(h, "iterate", st, [&] { return gas::launch_iterate(it, st); });
    ++launches;
  }
  if (e == cudaSuccess && v_out != nullptr) {
    gas::WbArgs w{};
    w.s = s;
    w.maps_k = h->dmaps + s.L;
    w.ybuf = h->ybuf;
    w.v_out = v_out;
    w.status = h->status;
    e = launch(h, "writeback", st, [&] { return gas::launch_writeback(w, h->num_sms, st); });
    ++launches;
  }
  h->last_launches = launches;
  if (e != cudaSuccess) return cuda_fail(h, e, "Gram path launch");
  return GAS_OK;
}

gas_status spectral_impl(gas_ctx* h, const void* const* wq, const void* const* wk, int iters, const float* v_in,
                         float* v_out, float* sigma, float* s_out, float scale_c, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (iters < 1) return fail(h, GAS_ERR_INVALID_ARG, "iters must be >= 1 (got %d)", iters);
  gas_status gs = check_weights(h, wq, wk);
  if (gs != GAS_OK) return gs;
  if (!v_in || !sigma) return fail(h, GAS_ERR_INVALID_ARG, "v_in and sigma must not be NULL");
  if (!aligned16(v_in) || (v_out && !aligned16(v_out)))
    return fail(h, GAS_ERR_INVALID_ARG, "v_in / v_out must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSetDevice(h->device);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
  h->last_stream = st;
  h->launch_names.clear();
  gas::LayerTable tab;
  std::memset(&tab, 0, sizeof(tab));
  fill_table(h, tab, wq, wk);
  // Conv1D tiles are read as 64-row boxes of whole heads: d_h 64 or 128 only
  const bool tc_ok = h->s.tc && !h->s.f32 && (!h->s.cols || h->s.dh == 64 || h->s.dh == 128);
  const int method = h->method == GAS_METHOD_AUTO ? (tc_ok ? GAS_METHOD_FUSED : GAS_METHOD_STREAM) : h->method;
  if (method != GAS_METHOD_STREAM && !tc_ok)
    return fail(h, GAS_ERR_UNSUPPORTED, "the tensor-core back ends need d_h 64, 80, 96 or 128, 16-bit weights, "
                                        "and d_h 64 or 128 in the Conv1D layout (use GAS_METHOD_STREAM or AUTO)");
  if (method == GAS_METHOD_STREAM && h->s.f32 && h->s.dh > 128)
    return fail(h, GAS_ERR_UNSUPPORTED, "fp32 weights are supported up to d_h 128");
  if (method == GAS_METHOD_STREAM && h->s.cols)
    return fail(h, GAS_ERR_UNSUPPORTED, "the streaming back end reads the nn.Linear layout only (use fused or gram)");
  if (method == GAS_METHOD_STREAM) return run_stream(h, tab, iters, v_in, v_out, sigma, s_out, scale_c, st);
  return run_gram(h, wq, wk, tab, iters, v_in, v_out, sigma, s_out, scale_c, method == GAS_METHOD_FUSED, st);
}

// Whole-layer sigma (Algorithms 2-3 over all heads of a layer): 4 streaming kernels per
// iteration, then sigma = ||u'||, v_out = v'/||v'|| and the layer scale.
gas_status run_layer(gas_ctx* h, const gas::LayerTable& tab, int iters, const float* v_in, float* v_out,
                     float* sigma, float* s_out, float scale_c, cudaStream_t st) {
  const Shape& s = h->s;
  const size_t Rq = static_cast<size_t>(s.nq) * s.dh, Rk = static_cast<size_t>(s.nkv) * s.dh;
  int launches = 0;
  cudaError_t e = cudaSuccess;
  for (int it = 0; it < iters && e == cudaSuccess; ++it) {
    gas::LayerArgs a{};
    a.s = s;
    a.which = 0;  // z_kv = W^K^T (v/||v||)
    a.src = it == 0 ? v_in : h->lv;
    a.out = h->lz;
    a.out_stride = Rk;
    e = launch(h, "layer_rowdot_k", st, [&] { return gas::launch_layer_rowdot(tab, a, st); });
    ++launches;
    if (e != cudaSuccess) break;
    a.which = 1;  // u' = W^Q RepeatBlocks(z_kv)
    a.src = h->lz;
    a.src_stride = Rk;
    a.out = h->lu;
    a.out_stride = s.d;
    e = launch(h, "layer_coldot_q", st, [&] { return gas::launch_layer_coldot(tab, a, st); });
    ++launches;
    if (e != cudaSuccess || (it == iters - 1 && v_out == nullptr)) break;
    a.which = 1;  // y = W^Q^T (u'/||u'||)
    a.src = h->lu;
    a.out = h->ly;
    a.out_stride = Rq;
    e = launch(h, "layer_rowdot_q", st, [&] { return gas::launch_layer_rowdot(tab, a, st); });
    ++launches;
    if (e != cudaSuccess) break;
    a.which = 0;  // v' = W^K SumGroups(y)
    a.src = h->ly;
    a.src_stride = Rq;
    a.out = h->lv;
    a.out_stride = s.d;
    e = launch(h, "layer_coldot_k", st, [&] { return gas::launch_layer_coldot(tab, a, st); });
    ++launches;
  }
  if (e == cudaSuccess) {
    gas::LayerArgs f{};
    f.s = s;
    f.src = h->lu;
    f.vsrc = h->lv;
    f.v_out = v_out;
    f.sigma = sigma;
    f.scale_out = s_out;
    f.scale_c = scale_c;
    f.status = h->status;
    e = launch(h, "layer_finalize", st, [&] { return gas::launch_layer_finalize(f, st); });
    ++launches;
  }
  h->last_launches = launches;
  if (e != cudaSuccess) return cuda_fail(h, e, "whole-layer launch");
  return GAS_OK;
}

gas_status resolve(gas_ctx* h, double gamma, double delta_star, double r_max, double* g_out, double* a_out) {
  if (!(delta_star > 0.0)) return fail(h, GAS_ERR_INVALID_ARG, "delta_star must be > 0");
  if (!(r_max > 0.0)) return fail(h, GAS_ERR_INVALID_ARG, "r_max must be > 0");
  if (gamma > 0.0 && gamma <= 1.0) return fail(h, GAS_ERR_INVALID_ARG, "gamma must exceed 1 (got %g)", gamma);
  const long long N = static_cast<long long>(h->s.L) * h->s.nq;
  double g = gamma > 0.0 ? gamma : gas_gamma_min(h->s.dh, N, h->seq_len, delta_star);
  if (!std::isfinite(g)) return fail(h, GAS_ERR_INVALID_ARG, "could not solve for gamma");
  double a = h->alpha_override > 0.0 ? h->alpha_override
                                     : gas_alpha_min(g, h->s.d, h->s.dh, N, h->seq_len, delta_star);
  *g_out = g;
  *a_out = a;
  return GAS_OK;
}

}  // namespace

void gas::set_global_error(const char* msg) { g_create_err = msg; }

extern "C" {

gas_status gas_create(int layers, int d, int n_q, int n_kv, int d_h, gas_handle* out) {
  if (!out) return fail(nullptr, GAS_ERR_INVALID_ARG, "out must not be NULL");
  *out = nullptr;
  if (layers < 1 || d < 1 || n_q < 1 || n_kv < 1 || d_h < 1)
    return fail(nullptr, GAS_ERR_INVALID_ARG, "sizes must be positive");
  if (layers > gas::kMaxLayers)
    return fail(nullptr, GAS_ERR_UNSUPPORTED, "at most %d layers per handle", gas::kMaxLayers);
  if (d % 8 != 0 || d < 8) return fail(nullptr, GAS_ERR_UNSUPPORTED, "d must be a multiple of 8 (got %d)", d);
  if (n_q % n_kv != 0) return fail(nullptr, GAS_ERR_UNSUPPORTED, "n_q (%d) must be a multiple of n_kv (%d)", n_q, n_kv);
  if (d_h != 64 && d_h != 80 && d_h != 96 && d_h != 128 && d_h != 256)
    return fail(nullptr, GAS_ERR_UNSUPPORTED, "d_h must be 64, 80, 96, 128 or 256 (got %d)", d_h);
  const int G = n_q / n_kv;
  // d_h 64 / 128: whole heads fill 128-row tiles; d_h 80 / 96: one head per 128-row tile,
  // the rows past d_h zero.  These run on the tensor-core back ends; d_h 256 runs on the
  // streaming back end only.
  const bool tc = d_h == 64 || d_h == 80 || d_h == 96 || d_h == 128;
  const int dh_t = d_h == 64 ? 64 : 128;  // head width of a tensor-core tile
  const int gpt = tc ? 128 / dh_t : 1;
  const int nz = round_up16(2 * G * gpt);
  if (tc && nz > 128)
    return fail(nullptr, GAS_ERR_UNSUPPORTED, "group size %d too large for d_h %d (max %d)", G, d_h, 64 / gpt);
  int nz_t = nz <= 16 ? 16 : nz <= 32 ? 32 : nz <= 64 ? 64 : 128;

  gas_ctx* h = new (std::nothrow) gas_ctx();
  if (!h) return fail(nullptr, GAS_ERR_ALLOC, "host allocation failed");
  Shape& s = h->s;
  s.L = layers; s.d = d; s.nq = n_q; s.nkv = n_kv; s.dh = d_h; s.G = G;
  s.nch = (d + gas::kStreamChunk - 1) / gas::kStreamChunk;
  s.tiles_q = (n_q * dh_t + 127) / 128;
  s.tiles_k = (n_kv * dh_t + 127) / 128;
  s.nkc = (d + 63) / 64;
  s.nz = nz_t;
  s.ldq = s.ldk = d;
  s.hsq = s.hsk = static_cast<long long>(d_h) * d;
  s.f16 = 0;
  s.cols = 0;
  s.f32 = 0;
  s.tc = tc ? 1 : 0;
  s.rows = d_h;

  cudaError_t e = cudaGetDevice(&h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  int cc_major = 0, smem_optin = 0;
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
  if (e != cudaSuccess) {
    gas_status st = cuda_fail(nullptr, e, "device query");
    delete h;
    return st;
  }
  if (cc_major != 10 || (tc && static_cast<size_t>(smem_optin) < gas::gram_smem_bytes(s.nz))) {
    delete h;
    return fail(nullptr, GAS_ERR_UNSUPPORTED, "needs an sm_10x GPU with >= %zu B shared memory per block",
                gas::gram_smem_bytes(s.nz));
  }

  const size_t L = layers, NQ = n_q, DH = d_h, NCH = s.nch;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t o_status = take(256);  // status word, then the epoch word at +128
  const size_t o_zp = take(L * NQ * NCH * DH * 4);
  const size_t o_n2p = take(L * NQ * NCH * 4);
  const size_t o_tp = take(L * NQ * NCH * DH * 4);
  const size_t o_s2p = take(L * NQ * NCH * 4);
  const size_t o_zr = take(L * NQ * DH * 4);
  const size_t o_n2r = take(L * NQ * 4);
  const size_t o_tr = take(L * NQ * DH * 4);
  const size_t o_s2r = take(L * NQ * 4);
  const size_t o_vhl = take(L * s.tiles_k * static_cast<size_t>(s.nz) * d * 2);
  const size_t o_gq = take(L * s.tiles_q * 16384ull * 4);
  const size_t o_gk = take(L * s.tiles_k * 16384ull * 4);
  const size_t o_z0 = take(L * NQ * 2 * static_cast<size_t>(dh_t) * 4);
  const size_t o_y = take(L * NQ * static_cast<size_t>(dh_t) * 4);
  const size_t o_maps = take((2 * L + 1) * sizeof(CUtensorMap));
  const size_t o_flags = take(L * s.tiles_k * sizeof(unsigned));
  const size_t o_vflags = take(L * s.tiles_k * sizeof(unsigned));
  const size_t o_vn2 = take(L * NQ * 4);
  const size_t o_lcnt = take((L + 1) * sizeof(unsigned));
  const size_t o_lmax = take(L * sizeof(unsigned long long));
  const size_t o_lz = take(L * static_cast<size_t>(n_kv) * d_h * 4);
  const size_t o_lu = take(L * static_cast<size_t>(d) * 4);
  const size_t o_ly = take(L * static_cast<size_t>(n_q) * d_h * 4);
  const size_t o_lv = take(L * static_cast<size_t>(d) * 4);
  h->ws_bytes = off;
  e = cudaMalloc(&h->ws, h->ws_bytes);
  if (e != cudaSuccess) {
    delete h;
    return fail(nullptr, GAS_ERR_ALLOC, "cudaMalloc(%zu) failed: %s", off, cudaGetErrorString(e));
  }
  e = cudaMemset(h->ws, 0, h->ws_bytes);
  char* b = static_cast<char*>(h->ws);
  h->status = reinterpret_cast<unsigned*>(b + o_status);
  h->epoch = reinterpret_cast<unsigned*>(b + o_status + 128);
  if (e == cudaSuccess) {  // flag epochs start at 1: a cleared flag (0) never reads as published
    const unsigned one = 1u;
    e = cudaMemcpy(h->epoch, &one, sizeof(one), cudaMemcpyHostToDevice);
  }
  h->zp = reinterpret_cast<float*>(b + o_zp);
  h->n2p = reinterpret_cast<float*>(b + o_n2p);
  h->tp = reinterpret_cast<float*>(b + o_tp);
  h->s2p = reinterpret_cast<float*>(b + o_s2p);
  h->zr = reinterpret_cast<float*>(b + o_zr);
  h->n2r = reinterpret_cast<float*>(b + o_n2r);
  h->tr = reinterpret_cast<float*>(b + o_tr);
  h->s2r = reinterpret_cast<float*>(b + o_s2r);
  h->vhl = reinterpret_cast<uint16_t*>(b + o_vhl);
  h->gq = reinterpret_cast<float*>(b + o_gq);
  h->gk = reinterpret_cast<float*>(b + o_gk);
  h->z0 = reinterpret_cast<float*>(b + o_z0);
  h->ybuf = reinterpret_cast<float*>(b + o_y);
  h->dmaps = reinterpret_cast<CUtensorMap*>(b + o_maps);
  h->flags = reinterpret_cast<unsigned*>(b + o_flags);
  h->vflags = reinterpret_cast<unsigned*>(b + o_vflags);
  h->vn2 = reinterpret_cast<float*>(b + o_vn2);
  h->layer_cnt = reinterpret_cast<unsigned*>(b + o_lcnt);
  h->done_cnt = h->layer_cnt + L;
  h->layer_max = reinterpret_cast<unsigned long long*>(b + o_lmax);
  h->lz = reinterpret_cast<float*>(b + o_lz);
  h->lu = reinterpret_cast<float*>(b + o_lu);
  h->ly = reinterpret_cast<float*>(b + o_ly);
  h->lv = reinterpret_cast<float*>(b + o_lv);
  h->hmaps.assign(2 * L + 1, CUtensorMap{});
  h->map_q.assign(L, nullptr);
  h->map_k.assign(L, nullptr);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    gas_status st = cuda_fail(nullptr, e, "workspace init");
    cudaFree(h->ws);
    delete h;
    return st;
  }
  if (!encode_2d(&h->hmaps[2 * L], h->vhl, d, L * s.tiles_k * static_cast<uint64_t>(s.nz), s.nz)) {
    cudaFree(h->ws);
    delete h;
    return fail(nullptr, GAS_ERR_CUDA, "cuTensorMapEncodeTiled failed for the vector operand");
  }
  *out = h;
  return GAS_OK;
}

gas_status gas_destroy(gas_handle h) {
  if (!h) return GAS_OK;
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  if (h->ws) cudaFree(h->ws);
  delete h;
  return GAS_OK;
}

size_t gas_workspace_bytes(gas_handle h) { return h ? h->ws_bytes : 0; }

gas_status gas_set_calibration(gas_handle h, int seq_len, double eta_fp8, double alpha_override) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (seq_len < 1) return fail(h, GAS_ERR_INVALID_ARG, "seq_len must be >= 1");
  if (!(eta_fp8 > 0.0 && eta_fp8 <= 1.0)) return fail(h, GAS_ERR_INVALID_ARG, "eta_fp8 must be in (0, 1]");
  h->seq_len = seq_len;
  h->eta_fp8 = eta_fp8;
  h->alpha_override = alpha_override > 0.0 ? alpha_override : 0.0;
  return GAS_OK;
}

gas_status gas_set_method(gas_handle h, int method) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (method != GAS_METHOD_AUTO && method != GAS_METHOD_STREAM && method != GAS_METHOD_GRAM &&
      method != GAS_METHOD_FUSED)
    return fail(h, GAS_ERR_INVALID_ARG, "unknown method %d", method);
  h->method = method;
  return GAS_OK;
}

gas_status gas_set_weight_layout(gas_handle h, int layout, long long ld_q, long long ld_k, long long hs_q,
                                 long long hs_k) {
  if (!h) return GAS_ERR_INVALID_ARG;
  const Shape& s = h->s;
  long long lq, lk, hq, hk;
  if (layout == GAS_LAYOUT_ROWS) {
    lq = ld_q ? ld_q : s.d;
    lk = ld_k ? ld_k : s.d;
    hq = hs_q ? hs_q : lq * s.dh;
    hk = hs_k ? hs_k : lk * s.dh;
    if (lq < s.d || lk < s.d)
      return fail(h, GAS_ERR_INVALID_ARG, "row strides must be >= d (%d), got %lld and %lld", s.d, lq, lk);
    if (hq < lq * s.dh || hk < lk * s.dh)
      return fail(h, GAS_ERR_INVALID_ARG, "head strides must be >= d_h * row stride (heads must not overlap)");
  } else if (layout == GAS_LAYOUT_COLS) {
    const long long rq = static_cast<long long>(s.nq) * s.dh, rk = static_cast<long long>(s.nkv) * s.dh;
    lq = ld_q ? ld_q : rq;
    lk = ld_k ? ld_k : rk;
    if (lq < rq || lk < rk)
      return fail(h, GAS_ERR_INVALID_ARG, "Conv1D strides must be >= the matrix's row count (%lld, %lld)", rq, rk);
    if ((hs_q && hs_q != s.dh) || (hs_k && hs_k != s.dh))
      return fail(h, GAS_ERR_INVALID_ARG, "Conv1D heads are contiguous: head strides must be 0 or d_h");
    hq = hk = s.dh;
  } else {
    return fail(h, GAS_ERR_UNSUPPORTED, "unknown weight layout %d", layout);
  }
  if (lq % 8 || lk % 8 || hq % 8 || hk % 8)
    return fail(h, GAS_ERR_INVALID_ARG, "row and head strides must be multiples of 8 elements (16 bytes)");
  if ((lq >> 37) || (lk >> 37) || (hq >> 37) || (hk >> 37))
    return fail(h, GAS_ERR_INVALID_ARG, "strides too large");
  h->s.cols = layout == GAS_LAYOUT_COLS ? 1 : 0;
  h->s.ldq = lq;
  h->s.ldk = lk;
  h->s.hsq = hq;
  h->s.hsk = hk;
  h->maps_valid = false;  // descriptors are rebuilt at the next call
  return GAS_OK;
}

gas_status gas_set_weight_dtype(gas_handle h, int dtype) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (dtype != GAS_DTYPE_BF16 && dtype != GAS_DTYPE_F16 && dtype != GAS_DTYPE_F32)
    return fail(h, GAS_ERR_INVALID_ARG, "unknown weight dtype %d", dtype);
  h->s.f16 = dtype == GAS_DTYPE_F16 ? 1 : 0;
  h->s.f32 = dtype == GAS_DTYPE_F32 ? 1 : 0;
  return GAS_OK;
}

gas_status gas_spectral_norms(gas_handle h, const void* const* wq, const void* const* wk, int iters,
                              const float* v_in, float* v_out, float* sigma, void* stream) {
  return spectral_impl(h, wq, wk, iters, v_in, v_out, sigma, nullptr, 0.0f, stream);
}

gas_status gas_scales(gas_handle h, const float* sigma, double gamma, double delta_star, double r_max, float* s,
                      void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (!sigma || !s) return fail(h, GAS_ERR_INVALID_ARG, "sigma and s must not be NULL");
  double g, a;
  gas_status gs = resolve(h, gamma, delta_star, r_max, &g, &a);
  if (gs != GAS_OK) return gs;
  cudaError_t e = cudaSetDevice(h->device);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
  gas::ScalesArgs sa{h->s.L, h->s.nq, sigma, s, scale_constant(h, a, r_max)};
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  h->launch_names.clear();
  e = launch(h, "scales", st, [&] { return gas::launch_scales(sa, st); });
  h->last_launches = 1;
  if (e != cudaSuccess) return cuda_fail(h, e, "scales launch");
  return GAS_OK;
}

gas_status gas_refresh(gas_handle h, const void* const* wq, const void* const* wk, int iters, const float* v_in,
                       float* v_out, float* sigma, double gamma, double delta_star, double r_max, float* s,
                       void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (!s) return fail(h, GAS_ERR_INVALID_ARG, "s must not be NULL");
  double g, a;
  gas_status gs = resolve(h, gamma, delta_star, r_max, &g, &a);
  if (gs != GAS_OK) return gs;
  return spectral_impl(h, wq, wk, iters, v_in, v_out, sigma, s, scale_constant(h, a, r_max), stream);
}

gas_status gas_layer_refresh(gas_handle h, const void* const* wq, const void* const* wk, int iters,
                             const float* v_in, float* v_out, float* sigma, double gamma, double delta_star,
                             double r_max, float* s, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (iters < 1) return fail(h, GAS_ERR_INVALID_ARG, "iters must be >= 1 (got %d)", iters);
  gas_status gs = check_weights(h, wq, wk);
  if (gs != GAS_OK) return gs;
  if (!v_in || !sigma) return fail(h, GAS_ERR_INVALID_ARG, "v_in and sigma must not be NULL");
  if (!aligned16(v_in) || (v_out && !aligned16(v_out)))
    return fail(h, GAS_ERR_INVALID_ARG, "v_in / v_out must be 16-byte aligned");
  if (h->s.cols)
    return fail(h, GAS_ERR_UNSUPPORTED, "the whole-layer path reads the nn.Linear layout only");
  if (static_cast<size_t>(h->s.d + 8) * 4 > 227 * 1024 ||
      static_cast<size_t>(h->s.nq * h->s.dh + 2048) * 4 > 227 * 1024)
    return fail(h, GAS_ERR_UNSUPPORTED, "whole-layer path keeps a d- or n_q*d_h-vector in shared memory");
  float c = 0.0f;
  if (s) {
    double g, a;
    gs = resolve(h, gamma, delta_star, r_max, &g, &a);
    if (gs != GAS_OK) return gs;
    c = scale_constant(h, a, r_max);
  }
  cudaError_t e = cudaSetDevice(h->device);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  h->last_stream = st;
  h->launch_names.clear();
  gas::LayerTable tab;
  std::memset(&tab, 0, sizeof(tab));
  fill_table(h, tab, wq, wk);
  return run_layer(h, tab, iters, v_in, v_out, sigma, s, c, st);
}

double gas_gamma_min(int d_h, long long n_heads_total, int seq_len, double delta_star) {
  if (d_h < 1 || n_heads_total < 1 || seq_len < 1 || !(delta_star > 0.0)) return NAN;
  const double rhs = (2.0 / d_h) * std::log(2.0 * static_cast<double>(n_heads_total) * seq_len / delta_star);
  if (!(rhs > 0.0)) return 1.0;
  // h(g) = g - 1 - ln g is increasing on (1, inf): bracket, then bisect.
  double lo = 1.0, hi = 2.0;
  while (h_fn(hi) < rhs) hi *= 2.0;
  for (int i = 0; i < 200 && hi - lo > 1e-13 * hi; ++i) {
    const double mid = 0.5 * (lo + hi);
    if (h_fn(mid) >= rhs) hi = mid;
    else lo = mid;
  }
  return hi;
}

double gas_alpha_min(double gamma, int d, int d_h, long long n_heads_total, int seq_len, double delta_star) {
  if (!(gamma >= 1.0) || d < 1 || d_h < 1 || n_heads_total < 1 || seq_len < 1 || !(delta_star > 0.0)) return NAN;
  const double lg = std::log(4.0 * static_cast<double>(n_heads_total) * seq_len * static_cast<double>(seq_len) /
                             delta_star);
  return std::sqrt(2.0 * gamma * d_h) / d * std::sqrt(lg > 0.0 ? lg : 0.0);
}

gas_status gas_resolve_calibration(gas_handle h, double gamma, double delta_star, double* gamma_out,
                                   double* alpha_out) {
  if (!h || !gamma_out || !alpha_out) return GAS_ERR_INVALID_ARG;
  return resolve(h, gamma, delta_star, 448.0, gamma_out, alpha_out);
}

const char* gas_last_error(gas_handle h) { return h ? h->err.c_str() : g_create_err.c_str(); }

const char* gas_status_string(gas_status s) {
  switch (s) {
    case GAS_OK: return "GAS_OK";
    case GAS_ERR_INVALID_ARG: return "GAS_ERR_INVALID_ARG";
    case GAS_ERR_UNSUPPORTED: return "GAS_ERR_UNSUPPORTED";
    case GAS_ERR_CUDA: return "GAS_ERR_CUDA";
    case GAS_ERR_ALLOC: return "GAS_ERR_ALLOC";
    case GAS_ERR_DEVICE_TIMEOUT: return "GAS_ERR_DEVICE_TIMEOUT";
  }
  return "GAS_ERR_UNKNOWN";
}

gas_status gas_get_device_status(gas_handle h, int* code, int clear) {
  if (!h || !code) return GAS_ERR_INVALID_ARG;
  cudaError_t e = cudaSetDevice(h->device);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  unsigned v = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&v, h->status, sizeof(v), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && clear) e = cudaMemset(h->status, 0, sizeof(unsigned));
  if (e != cudaSuccess) return cuda_fail(h, e, "reading device status");
  *code = static_cast<int>(v);
  if (v & GAS_DEV_WAIT_TIMEOUT) return fail(h, GAS_ERR_DEVICE_TIMEOUT, "a device-side bounded wait ran out");
  return GAS_OK;
}

gas_status gas_selftest_wait_timeout(gas_handle h, int which, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (which != 0 && which != 1) return fail(h, GAS_ERR_INVALID_ARG, "which must be 0 or 1 (got %d)", which);
  cudaError_t e = cudaSetDevice(h->device);
  if (e == cudaSuccess) e = gas::launch_wait_selftest(h->status, which, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "self-test launch");
  return GAS_OK;
}

int gas_last_launch_count(gas_handle h) { return h ? h->last_launches : 0; }

gas_status gas_set_launch_events(gas_handle h, void* const* events, int n_events) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (n_events < 0 || (n_events & 1)) return fail(h, GAS_ERR_INVALID_ARG, "n_events must be even and >= 0");
  h->events.clear();
  if (events)
    for (int i = 0; i < n_events; ++i) h->events.push_back(static_cast<cudaEvent_t>(events[i]));
  return GAS_OK;
}

const char* gas_last_launch_name(gas_handle h, int i) {
  if (!h || i < 0 || static_cast<size_t>(i) >= h->launch_names.size()) return "";
  return h->launch_names[i];
}

}  // extern "C"
