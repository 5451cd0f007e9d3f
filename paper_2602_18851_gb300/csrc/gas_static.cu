// Allocation-free spectral norms: gas_spectral_norms_static (include/gas.h).
//
// Some callers of this library cannot allocate device memory at all: code that runs
// under another framework's memory manager (which owns every byte of HBM and hands
// out nothing extra), code on a latency-critical path where the implicit device
// synchronisation of cudaMalloc / cudaFree is not allowed, and small plugins that
// have no place to keep a handle (and its workspace) alive between calls.  For them
// this entry point runs the streaming power iteration (the same kernels as
// GAS_METHOD_STREAM) with its scratch in one file-scope device array instead of a
// handle's workspace.  The caller still passes every input and output buffer.
//
// The array is part of the library's device image: every GPU that loads the library
// holds kStaticScratchBytes for it until the process exits.  All calls share it, so
// calls whose kernels overlap on the GPU (two streams, two host threads) race on it.

#include <cstdio>
#include <cstring>

#include "../../include/gas.h"
#include "gas_device.cuh"

namespace gas {
namespace {

constexpr size_t kStaticScratchBytes = GAS_STATIC_SCRATCH_BYTES;

// Host code must not use this name as a device address (see static_scratch_ptr).
__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// Device address of the scratch array in the current context.  It is looked up on every
// call: the address belongs to the context that loaded the library's device code, so a
// cached value would go stale after cudaDeviceReset or under another context.  After the
// first call on a device (which also loads the device code) the lookup is a table search.
cudaError_t static_scratch_ptr(void** out) { return cudaGetSymbolAddress(out, g_static_scratch); }

// Bytes of scratch one call needs (0 for sizes that are not positive).
// Layout: z and t partials [L][n_q][nch][d_h], their squared-norm partials [L][n_q][nch]
// and the chunk sums of both ([L][n_q][d_h] and [L][n_q]), each region 256-byte aligned.
struct StaticLayout {
  size_t vec, nrm, rvec, rnrm, total;
};
StaticLayout static_layout(int layers, int d, int n_q, int d_h) {
  StaticLayout o{};
  if (layers < 1 || d < 1 || n_q < 1 || d_h < 1) return o;
  const size_t nch = (static_cast<size_t>(d) + kStreamChunk - 1) / kStreamChunk;
  o.vec = static_cast<size_t>(layers) * n_q * nch * d_h * sizeof(float);
  o.nrm = static_cast<size_t>(layers) * n_q * nch * sizeof(float);
  o.rvec = static_cast<size_t>(layers) * n_q * d_h * sizeof(float);
  o.rnrm = static_cast<size_t>(layers) * n_q * sizeof(float);
  o.total = 2 * align256(o.vec) + 2 * align256(o.nrm) + 2 * align256(o.rvec) + 2 * align256(o.rnrm);
  return o;
}

}  // namespace
}  // namespace gas

namespace {
// Errors are reported like gas_create's: gas_last_error(NULL) returns the message.
gas_status static_fail(gas_status st, const char* msg) {
  gas::set_global_error(msg);
  return st;
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

extern "C" gas_status gas_spectral_norms_static(int layers, int d, int n_q, int n_kv, int d_h,
                                                const void* const* wq, const void* const* wk, int iters,
                                                const float* v_in, float* v_out, float* sigma, void* stream) {
  char buf[256];
  if (layers < 1 || d < 8 || n_q < 1 || n_kv < 1 || iters < 1)
    return static_fail(GAS_ERR_INVALID_ARG, "gas_spectral_norms_static: sizes and iters must be positive");
  if (layers > gas::kMaxLayers || d % 8 != 0 || n_q % n_kv != 0 || (d_h != 64 && d_h != 128))
    return static_fail(GAS_ERR_UNSUPPORTED,
                       "gas_spectral_norms_static: needs layers <= 512, d % 8 == 0, n_q % n_kv == 0, d_h 64/128");
  if (!wq || !wk || !v_in || !sigma)
    return static_fail(GAS_ERR_INVALID_ARG, "gas_spectral_norms_static: NULL argument");
  if (!al16(v_in) || (v_out && !al16(v_out)))
    return static_fail(GAS_ERR_INVALID_ARG, "gas_spectral_norms_static: vectors must be 16-byte aligned");
  for (int l = 0; l < layers; ++l)
    if (!wq[l] || !wk[l] || !al16(wq[l]) || !al16(wk[l]))
      return static_fail(GAS_ERR_INVALID_ARG, "gas_spectral_norms_static: NULL or misaligned weight pointer");

  gas::Shape s{};
  s.L = layers; s.d = d; s.nq = n_q; s.nkv = n_kv; s.dh = d_h; s.G = n_q / n_kv;
  s.nch = (d + gas::kStreamChunk - 1) / gas::kStreamChunk;
  s.ldq = s.ldk = d;
  s.hsq = s.hsk = static_cast<long long>(d_h) * d;
  s.f16 = 0;
  s.f32 = 0;
  s.tc = 1;
  const gas::StaticLayout lay = gas::static_layout(layers, d, n_q, d_h);
  const size_t vec = lay.vec, nrm = lay.nrm, rvec = lay.rvec, rnrm = lay.rnrm, need = lay.total;
  if (need > gas::kStaticScratchBytes) {
    snprintf(buf, sizeof(buf),
             "gas_spectral_norms_static: this shape needs %zu bytes of scratch, the static array holds %zu",
             need, gas::kStaticScratchBytes);
    return static_fail(GAS_ERR_UNSUPPORTED, buf);
  }
  void* base = nullptr;
  cudaError_t e = gas::static_scratch_ptr(&base);
  if (e != cudaSuccess) {
    snprintf(buf, sizeof(buf), "gas_spectral_norms_static: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
    return static_fail(GAS_ERR_CUDA, buf);
  }
  char* b = static_cast<char*>(base);
  float* zp = reinterpret_cast<float*>(b);
  float* tp = reinterpret_cast<float*>(b + gas::align256(vec));
  float* n2p = reinterpret_cast<float*>(b + 2 * gas::align256(vec));
  float* s2p = reinterpret_cast<float*>(b + 2 * gas::align256(vec) + gas::align256(nrm));
  char* r = b + 2 * gas::align256(vec) + 2 * gas::align256(nrm);
  float* zr = reinterpret_cast<float*>(r);
  float* tr = reinterpret_cast<float*>(r + gas::align256(rvec));
  float* n2r = reinterpret_cast<float*>(r + 2 * gas::align256(rvec));
  float* s2r = reinterpret_cast<float*>(r + 2 * gas::align256(rvec) + gas::align256(rnrm));
  // Every scratch value a pass reads was written earlier in the same call (each pass and
  // its chunk reduction cover all heads, chunks and rows), so nothing carries over from
  // an earlier call and nothing has to be cleared.
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  gas::LayerTable tab;
  std::memset(&tab, 0, sizeof(tab));
  for (int l = 0; l < layers; ++l) {
    tab.q[l] = static_cast<const uint16_t*>(wq[l]);
    tab.k[l] = static_cast<const uint16_t*>(wk[l]);
  }
  gas::StreamArgs a{};
  a.s = s;
  a.mode = gas::kPassK0;
  a.out = zp;
  a.out2 = n2p;
  a.outr = zr;
  a.outr2 = n2r;
  a.v_in = v_in;
  e = gas::launch_stream_pass(tab, a, st);
  if (e == cudaSuccess) e = gas::launch_stream_reduce(a, st);
  for (int it = 0; it < iters && e == cudaSuccess; ++it) {
    gas::StreamArgs q{};
    q.s = s;
    q.mode = gas::kPassQ;
    q.in_scaled = 1;
    q.in = zr;
    q.in2 = n2r;
    q.out = tp;
    q.out2 = s2p;
    q.outr = tr;
    q.outr2 = s2r;
    e = gas::launch_stream_pass(tab, q, st);
    if (e == cudaSuccess) e = gas::launch_stream_reduce(q, st);
    const bool last = (it == iters - 1);
    if (e != cudaSuccess || (last && v_out == nullptr)) break;
    gas::StreamArgs k{};
    k.s = s;
    k.mode = last ? gas::kPassKOut : gas::kPassK;
    k.in_scaled = 1;
    k.in = tr;
    k.in2 = s2r;
    k.out = zp;
    k.out2 = n2p;
    k.outr = zr;
    k.outr2 = n2r;
    k.v_out = v_out;
    e = gas::launch_stream_pass(tab, k, st);
    if (e == cudaSuccess) e = gas::launch_stream_reduce(k, st);
  }
  if (e == cudaSuccess) {
    gas::FinalizeArgs f{};
    f.s = s;
    f.s2 = s2r;
    f.n2 = n2r;
    f.v_out = v_out;
    f.sigma = sigma;
    e = gas::launch_finalize(f, st);
  }
  if (e != cudaSuccess) {
    snprintf(buf, sizeof(buf), "gas_spectral_norms_static: launch failed: %s", cudaGetErrorString(e));
    return static_fail(GAS_ERR_CUDA, buf);
  }
  return GAS_OK;
}

extern "C" size_t gas_static_scratch_bytes(int layers, int d, int n_q, int d_h) {
  return gas::static_layout(layers, d, n_q, d_h).total;
}
