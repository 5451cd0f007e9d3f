// Internal declarations shared by the host API (gas_api.cpp) and the kernels.
// Nothing here is part of the public C ABI (include/gas.h).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#ifndef GAS_DEV_NONFINITE_SIGMA
#define GAS_DEV_NONFINITE_SIGMA 0x1
#define GAS_DEV_WAIT_TIMEOUT 0x2
#endif

namespace gas {

constexpr int kMaxLayers = 512;             // per-layer pointer table carried as a kernel parameter
constexpr int kStreamChunk = 256;           // columns of d per streaming CTA
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // bounded device waits: 2 s

// Per-layer base pointers of the bf16 weight blocks, passed by value.
struct LayerTable {
  const uint16_t* q[kMaxLayers];
  const uint16_t* k[kMaxLayers];
};

// Shape of one handle.
struct Shape {
  int L, d, nq, nkv, dh, G;
  int nch;        // ceil(d / kStreamChunk)
  int tiles_q;    // ceil(nq * dh / 128)
  int tiles_k;    // ceil(nkv * dh / 128)
  int nkc;        // ceil(d / 64)
  int nz;         // z-accumulator columns of a K tile (multiple of 16)
  long long ldq;  // elements between consecutive rows of one head of Wq[l] (>= d)
  long long ldk;  // elements between consecutive rows of one key group of Wk[l] (>= d)
  long long hsq;  // elements between the first rows of consecutive query heads (>= d_h * ldq)
  long long hsk;  // elements between the first rows of consecutive key groups (>= d_h * ldk)
  int f16;        // weights (and the MMA operands) are binary16 instead of bf16
  int cols;       // GPT-2 Conv1D layout: element (row r, column c) at w[c * ld + r]
  int f32;        // fp32 weights (CUDA-core back ends only)
  int tc;         // d_h in {64, 80, 96, 128}: the tensor-core back ends apply
  int rows;       // weight rows per head as stored (the model's d_h).  The tensor-core
                  // kernels get a shape whose dh is the tile head width (64, or 128 for
                  // d_h 80 / 96 / 128); a head's rows past `rows` read as zero in the tile
};

// Element offset of row r (head r / d_h, row r % d_h inside it) of a weight matrix.
__host__ __device__ inline long long weight_row_offset(int r, int dh, long long ld, long long hs) {
  return static_cast<long long>(r / dh) * hs + static_cast<long long>(r % dh) * ld;
}

// ---- streaming matvec-chain passes (Algorithm 2 applied literally) ---------------
// One pass streams one weight matrix X (a head's A_h or a group's B_g, d_h x d) in
// column chunks.  For every vector that uses X it forms p = X^T x over the chunk
// (and ||p||^2), then either q = X p (partial over the chunk) or writes p out.  A short
// reduction kernel then sums the chunk partials (in chunk order) into one d_h-vector and
// one squared norm per head, which the next pass reads.
enum StreamMode : int {
  kPassQ = 0,      // X = A_h, x = z / ||v'|| (K results); out: t = A_h u', ||u'||^2
  kPassK = 1,      // X = B_g, x = t / ||u'|| = y (Q results, G heads); out: z = B_g v', ||v'||^2
  kPassK0 = 2,     // X = B_g, p = v_in chunk (G heads); out: z = B_g v, ||v||^2
  kPassKOut = 3,   // X = B_g, x = y (G heads); writes p (= v') to v_out, ||v'||^2
};

struct StreamArgs {
  Shape s;
  int mode;
  int in_scaled;      // 1: x = in / sqrt(in2); 0: x = in
  const float* in;    // [L][nq][dh] input vector of every head (modes Q, K, KOut)
  const float* in2;   // [L][nq]     its squared norm
  float* out;         // [L][nq][nch][dh] q partials                 (modes Q, K, K0)
  float* out2;        // [L][nq][nch]     ||p||^2 partials            (all modes)
  float* outr;        // [L][nq][dh]      q summed over the chunks    (modes Q, K, K0)
  float* outr2;       // [L][nq]          ||p||^2 summed over the chunks (all modes)
  const float* v_in;  // [L][nq][d]                                   (mode K0)
  float* v_out;       // [L][nq][d]                                   (mode KOut)
  float* s_zero;      // mode K0: per-layer scale slots zeroed for the fused epilogue
  unsigned* status;   // device status word (may be null)
  long long pf_dist;  // streaming pass: CTAs ahead whose tile is prefetched into L2 (0: none)
};

struct FinalizeArgs {
  Shape s;
  const float* s2;    // [L][nq] ||u'||^2 of the last Q pass
  const float* n2;    // [L][nq] ||v'||^2 of the last K pass (or null)
  float* v_out;       // [L][nq][d] raw v' (normalised in place) or null
  float* sigma;       // [L][nq]
  float* scale_out;   // [L] fused scale (atomic max) or null
  float scale_c;      // alpha * d / sqrt(d_h) / (eta * r_max)
  unsigned* status;
};

// ---- Gram path --------------------------------------------------------------------
struct PrepArgs {
  Shape s;
  const float* v_in;   // [L][nq][d]
  uint16_t* vhl;       // [L][tiles_k][nz][d] bf16 hi/lo rows of v / ||v||
  float* s_zero;       // [L] or null
  unsigned* epoch;     // flag value of the next fused Gram launch (advanced here)
};

struct GramArgs {
  Shape s;
  // fused variant: fp32 v rows [L*nq][d], box 64 columns x nz/2 rows, no swizzle; a
  // kernel parameter (re-encoded on the host for every call, no device upload)
  CUtensorMap map_vf;
  const CUtensorMap* maps_q;  // [L] tensor maps over Wq[l] ([nq*dh, d], box 64 x 128)
  const CUtensorMap* maps_k;  // [L]
  const CUtensorMap* map_v;   // unfused: one map over vhl ([L*tiles_k*nz, d], box 64 x nz)
  float* gq;                  // [L][tiles_q][128][128] (unfused only)
  float* gk;                  // [L][tiles_k][128][128]
  float* z0;                  // [L][nq][2][dh] hi and lo halves of B_g v/||v|| (unfused)
                              // or of B_g v (fused)
  unsigned* status;
  // fused variant: k iterations in the epilogue, straight from tensor memory
  unsigned* flags;            // [L][tiles_k] key-tile publication flags (== epoch when ready)
  unsigned* epoch;            // this launch's flag value (never 0); the fused kernel's last CTA
                              // advances it, so that a replayed CUDA graph gets a new one
  unsigned* layer_cnt;        // [L] finished heads per layer (fused scales), cleared at the end
  unsigned long long* layer_max;  // [L] epoch-tagged maximum sigma bits per layer
  unsigned* done_cnt;         // finished CTAs
  float* vn2;                 // [L][nq] ||v||^2 summed by the converter warps
  unsigned* vflags;           // [L][tiles_k] v-norm flags (== epoch when vn2 of the tile is ready)
  int iters;
  float* ybuf;                // [L][nq][dh]
  float* sigma;               // [L][nq]
  float* scale_out;           // [L] or null
  float scale_c;
};

// Tensor-core write-back v_out = B_g^T (y / ||v'||) for every head.
struct WbArgs {
  Shape s;
  const CUtensorMap* maps_k;  // [L] (box 64 x 128, as for the Gram pass)
  const float* ybuf;          // [L][nq][dh]
  float* v_out;               // [L][nq][d]
  unsigned* status;
};

struct IterArgs {
  Shape s;
  int iters;
  const float* gq;
  const float* gk;
  const float* z0;
  float* ybuf;        // [L][nq][dh]  y / ||v'|| of the last iteration (write-back input)
  float* sigma;       // [L][nq]
  float* scale_out;   // [L] fused scale (atomic max) or null
  float scale_c;
  unsigned* status;
};

// Whole-layer power iteration (Algorithms 2-3 with M = W^Q W^K_exp^T over all heads).
struct LayerArgs {
  Shape s;
  int which;              // 0: key matrix Wk, 1: query matrix Wq
  const float* src;       // input vector per layer
  size_t src_stride;      // floats between layers of src (coldot)
  float* out;
  size_t out_stride;
  const float* vsrc;      // finalize: v' of the last iteration
  float* v_out;           // finalize: [L][d] or null
  float* sigma;           // finalize: [L]
  float* scale_out;       // finalize: [L] or null
  float scale_c;
  unsigned* status;
};

struct ScalesArgs {
  int L, nq;
  const float* sigma;
  float* s;
  float scale_c;
};

// Raise a kernel's opt-in dynamic shared-memory limit on the current device, once per
// device (bit `device` of `done`; devices past 63 set it on every call).
inline cudaError_t set_smem_per_device(const void* kernel, int bytes, unsigned long long& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = dev < 64 ? 1ull << dev : 0ull;
  // `done` is a per-kernel static shared by every thread of the process: atomic accesses
  if (bit != 0ull && (__atomic_load_n(&done, __ATOMIC_RELAXED) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) __atomic_fetch_or(&done, bit, __ATOMIC_RELAXED);
  return e;
}

// Launchers (return cudaGetLastError() of the launch).
cudaError_t launch_stream_pass(const LayerTable& tab, const StreamArgs& a, cudaStream_t st);
cudaError_t launch_stream_reduce(const StreamArgs& a, cudaStream_t st);  // chunk sums of a pass
cudaError_t launch_finalize(const FinalizeArgs& a, cudaStream_t st);
cudaError_t launch_scales(const ScalesArgs& a, cudaStream_t st);
cudaError_t launch_prep_v(const PrepArgs& a, cudaStream_t st);
cudaError_t launch_gram(const GramArgs& a, int num_sms, bool fused, cudaStream_t st);
cudaError_t launch_iterate(const IterArgs& a, cudaStream_t st);
cudaError_t launch_writeback(const WbArgs& a, int num_sms, cudaStream_t st);
cudaError_t launch_layer_rowdot(const LayerTable& tab, const LayerArgs& a, cudaStream_t st);
cudaError_t launch_layer_coldot(const LayerTable& tab, const LayerArgs& a, cudaStream_t st);
cudaError_t launch_layer_finalize(const LayerArgs& a, cudaStream_t st);
cudaError_t launch_wait_selftest(unsigned* status, int which, cudaStream_t st);
void set_global_error(const char* msg);  // message returned by gas_last_error(NULL)
size_t gram_smem_bytes(int nz);

}  // namespace gas
