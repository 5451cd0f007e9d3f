// Gram back end: the same power iteration as Algorithm 2, moved into R^{d_h}.
//
// For head h with A = A_h = (W^Q_h)^T and B = B_g = (W^K_g)^T (both d_h x d), a unit v
// and z = B v, one iteration of Algorithm 2 is, exactly,
//   u' = A^T z,  ||u'||^2 = z^T (A A^T) z,  y = A u = (A A^T) z / ||u'||,
//   v' = B^T y,  ||v'||^2 = y^T (B B^T) y,  z_next = B v = (B B^T) y / ||v'||.
// So with the d_h x d_h Gram matrices G_Q = A A^T and G_K = B B^T the k iterations need
// no further weight traffic: one pass over every A_h and B_g (tensor cores), k
// iterations on 128 x 128 matrices (CUDA cores), and one more pass over B_g for the
// write-back v_out = B^T y / ||v'||.
//
//   prep_v_kernel   (unfused) v / ||v|| split into bf16 hi + lo rows, the tensor-core
//                   operand for z0
//   gram_kernel     persistent, warp-specialised: TMA -> smem ring -> tcgen05.mma into
//                   TMEM; G = X X^T for every 128-row weight tile and, on key tiles,
//                   Z = X [v_hi; v_lo]^T (z0 = B v in ~16-bit-mantissa precision).  The
//                   fused variant loads the fp32 v rows with the key tiles and splits
//                   them into the hi / lo operand inside the ring (two converter warps),
//                   which also sum ||v||^2 per head; its epilogue runs the k iterations
//   iterate_kernel  (unfused) k iterations per head in R^{d_h} from G_Q, G_K, z0; sigma,
//                   y/||v'||, fused per-layer scale (Eq. 15)
// The write-back v_out = B^T y / ||v'|| is its own tensor-core kernel (gas_writeback.cu),
// launched as a programmatic dependent of this one: every CTA here signals it once its
// prologue is done, so the write-back's CTAs can set up and prefetch W^K on the SMs this
// launch leaves.  The key tiles of the last layers are read with an L2 evict-last policy,
// because the write-back starts with those layers.

#include "gas_device.cuh"

namespace gas {

namespace {

// Warp 0: TMA producer; warp 1: MMA issuer (+ TMEM allocation); then the epilogue
// (4 warps for the Gram-only kernel, 8 for the fused one: two threads per row); the
// fused kernel ends with 2 converter warps (fp32 v rows -> bf16 hi / lo MMA operand).
// Twelve warps hold the same 168 registers per thread as ten (three warps per scheduler).
template <bool FUSED>
struct GramWarps {
  static constexpr int kEpiWarps = FUSED ? 8 : 4;
  static constexpr int kConvWarps = FUSED ? 2 : 0;
  static constexpr int kThreads = 64 + 32 * (kEpiWarps + kConvWarps);
};
constexpr uint32_t kTileBytes = 128u * 64u * 2u;  // one 128-row x 64-column bf16 box
constexpr int kSmemBudget = 232448;               // 227 KB opt-in dynamic shared memory
constexpr int kSmemReserve = 22528;               // alignment slack, barriers, epilogue scratch

// A ring stage holds BPS consecutive 64-column chunks of a tile: BPS weight boxes, the
// BPS matching v operand boxes (NZ rows of bf16 hi / lo, key tiles only) and, in the
// fused kernel, the BPS fp32 v boxes they are converted from (NZ/2 rows x 64 floats).
// Two chunks per stage halve the per-byte count of barrier waits, commits and copy
// issues on the producer and MMA threads.
template <int NZ, int BPS, bool FUSED>
struct GramCfg {
  static constexpr uint32_t kVBytes = static_cast<uint32_t>(NZ) * 64u * 2u;
  static constexpr uint32_t kFBytes = FUSED ? static_cast<uint32_t>(NZ / 2) * 64u * 4u : 0u;
  static constexpr uint32_t kStageBytes = BPS * (kTileBytes + kVBytes + kFBytes);
  static constexpr int kStages = (kSmemBudget - kSmemReserve) / static_cast<int>(kStageBytes);
  static constexpr size_t kSmem = static_cast<size_t>(kStages) * kStageBytes + kSmemReserve;
  // Tensor-memory accumulators (G: 128 columns, z: NZ columns each) cycled over tiles:
  // three when they fit in the 512 columns, so a query tile's epilogue may run its
  // iterations for two mainloops before the MMA warp needs its accumulator back.
  static constexpr int kAcc = (3 * (128 + NZ) <= 512) ? 3 : 2;
  static_assert(kStages >= 3, "ring too shallow");
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
};

// ---- v / ||v|| as hi + lo rows of the weights' 16-bit format -----------------------
// Row layout of one key tile's operand (nz rows): group gi of the tile owns rows
// gi*2G .. gi*2G+2G-1; head j of the group has its hi part at gi*2G + j and its lo
// part at gi*2G + G + j.  Padding rows stay zero (cleared at handle creation).
__global__ void __launch_bounds__(256) prep_v_kernel(const __grid_constant__ PrepArgs a) {
  const Shape& s = a.s;
  const size_t hidx = blockIdx.x;
  const int l = static_cast<int>(hidx / s.nq), h = static_cast<int>(hidx % s.nq);
  const int g = h / s.G, j = h % s.G;
  const int tk = (g * s.dh) / 128, gi = ((g * s.dh) % 128) / s.dh;
  const float* v = a.v_in + hidx * s.d;
  __shared__ float wsum[8];
  float n2 = 0.0f;
  for (int c = threadIdx.x * 4; c < s.d; c += blockDim.x * 4) {
    const float4 x = *reinterpret_cast<const float4*>(v + c);
    n2 = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, fmaf(x.w, x.w, n2))));
  }
  n2 = warp_sum(n2);
  if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = n2;
  __syncthreads();
  float tot = 0.0f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += wsum[w];
  const float inv = safe_inv_sqrt(tot);
  const size_t base = (static_cast<size_t>(l) * s.tiles_k + tk) * s.nz;
  uint16_t* hi_row = a.vhl + (base + gi * 2 * s.G + j) * s.d;
  uint16_t* lo_row = a.vhl + (base + gi * 2 * s.G + s.G + j) * s.d;
  for (int c = threadIdx.x * 8; c < s.d; c += blockDim.x * 8) {
    const float4 x0 = *reinterpret_cast<const float4*>(v + c);
    const float4 x1 = *reinterpret_cast<const float4*>(v + c + 4);
    const float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
    uint32_t hb[8], lb[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) split_hilo(xv[e] * inv, s.f16 != 0, hb[e], lb[e]);
    *reinterpret_cast<uint4*>(hi_row + c) =
        make_uint4(hb[0] | (hb[1] << 16), hb[2] | (hb[3] << 16), hb[4] | (hb[5] << 16), hb[6] | (hb[7] << 16));
    *reinterpret_cast<uint4*>(lo_row + c) =
        make_uint4(lb[0] | (lb[1] << 16), lb[2] | (lb[3] << 16), lb[4] | (lb[5] << 16), lb[6] | (lb[7] << 16));
  }
  if (a.s_zero != nullptr && h == 0 && threadIdx.x == 0) a.s_zero[l] = 0.0f;
  if (hidx == 0 && threadIdx.x == 0 && a.epoch != nullptr) {
    const unsigned e = *a.epoch + 1u;
    *a.epoch = e == 0u ? 1u : e;
  }
}

// ---- tcgen05 Gram kernel -------------------------------------------------------------
struct TileRef {
  int layer, is_k, idx;
};

// Tile order: the key tiles of the first D layers, then for every layer l the key tiles
// of layer l + D (while there is such a layer) followed by the query tiles of layer l.
// D layers of key tiles span at least one wave of the grid, so every query tile's key
// tile comes at least one wave earlier in the order (and earlier in its own CTA's list):
// its G_K and z0 are normally published by the time the query tile's epilogue starts,
// and every flag wait targets a smaller tile index, so the waits form no cycle.  Between
// the first and last D layers key tiles, whose epilogue is short, alternate with query
// tiles, whose epilogue runs the iterations: on MHA shapes (as many key tiles as query
// tiles) this halves the epilogue's load there.  D = L puts every key tile first.
__device__ __forceinline__ int lead_layers(const Shape& s, int grid) {
  const int d = (grid + s.tiles_k - 1) / s.tiles_k;
  return d < s.L ? d : s.L;
}

__device__ __forceinline__ TileRef decode_tile(const Shape& s, int D, int t) {
  TileRef r;
  const int tk = s.tiles_k, tq = s.tiles_q;
  const int P = D * tk;
  if (t < P) {
    r.is_k = 1;
    r.layer = t / tk;
    r.idx = t - r.layer * tk;
    return r;
  }
  int u = t - P;
  const int nf = s.L - D;  // layers whose block also carries the key tiles of layer l + D
  const int fb = nf * (tk + tq);
  if (u < fb) {
    const int l = u / (tk + tq), q = u - l * (tk + tq);
    r.is_k = q < tk;
    r.layer = r.is_k ? l + D : l;
    r.idx = r.is_k ? q : q - tk;
  } else {
    u -= fb;
    r.is_k = 0;
    r.layer = nf + u / tq;
    r.idx = u - (r.layer - nf) * tq;
  }
  return r;
}

// Shared scratch of the fused epilogue.  `stage` carries one TMEM lane quarter (32 rows)
// of a query tile's G_Q at a time from the row-per-thread layout tcgen05.ld produces to
// the block layout of the iteration; xs / ts hold the current x and t' of each head
// slot (two heads per tile when d_h = 64).
// Layout of a 4-float chunk q of a 128-float row inside a "plane" array: chunks that the
// lanes of a half-warp read together (same plane, consecutive q / 2 ... see plane_off)
// are contiguous, so 128-bit shared loads and stores are free of bank conflicts.
struct EpiSmem {
  float stage[2][32][68];  // [plane][row][16 chunks x 4 floats + 4 pad]
  float xs[2][2][64];      // [slot][plane][64]: x in the same plane layout
  float ts[2][2][64];
  int ok[2];
};

// Column col (of a d_h-wide row) -> offset inside [plane][16 chunks][4] when each thread
// owns cpt consecutive columns (cpt = 8: two planes, cpt = 4: one plane).
template <int CPT>
__device__ __forceinline__ int plane_off(int col, int row_stride) {
  const int p = (CPT == 8) ? ((col >> 2) & 1) : 0;
  const int slot = col / CPT;
  return p * 32 * row_stride + slot * 4 + (col & 3);
}

// The same layout for a single d_h-vector: [plane][16 chunks x 4].
template <int CPT>
__device__ __forceinline__ int vec_off(int col) {
  const int p = (CPT == 8) ? ((col >> 2) & 1) : 0;
  return p * 64 + (col / CPT) * 4 + (col & 3);
}

// Sum over the 16 lanes of a half-warp of 8 values per lane: on return v[0] holds the
// total of value number `idx` (3 halving exchange steps plus one butterfly step).
__device__ __forceinline__ float halfwarp_transpose_reduce8(float (&v)[8], int lane, int& idx) {
  int base = 0;
#pragma unroll
  for (int n = 8, off = 8; n > 1; n >>= 1, off >>= 1) {
    const int h = n >> 1;
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int k = 0; k < h; ++k) {
      const float send = up ? v[k] : v[k + h];
      const float keep = up ? v[k + h] : v[k];
      v[k] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, off);
    }
    if (up) base += h;
  }
  v[0] += __shfl_xor_sync(0xFFFFFFFFu, v[0], 1);
  idx = base;
  return v[0];
}

// Sum over the 16 lanes of a half-warp (all lanes get the total).
__device__ __forceinline__ float halfwarp_sum(float v) {
#pragma unroll
  for (int off = 1; off < 16; off <<= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, off);
  return v;
}

// k power iterations for the head(s) of one query tile, in R^{d_h}, run by the 8
// epilogue warps.  Block layout: inside a head, warp w owns rows 16w + 8*(lane/16) .. +8
// and lane % 16 owns d_h/16 consecutive columns, for both G_Q (copied once out of the
// tile's tensor-memory accumulator, which is then handed back to the MMA warp) and G_K
// (published by the key tile).  A matvec is 8 x d_h/16 FMAs per thread plus an 8-value
// half-warp reduction; each thread reads only its own d_h/16 entries of the vector.
// With x = c z (c a known scalar, c = 1 for z0) one iteration of Algorithm 2 is
//   t' = G_Q x,  S1 = x.t' = c^2 sigma^2,  y = t' / sqrt(S1),
//   w  = G_K y,  S2 = y.w = ||v'||^2,       x <- w,  c <- sqrt(S2),
// two barriers per iteration.
template <int DH>
__device__ __forceinline__ void fused_iterate(const GramArgs& a, int layer, int idx, uint32_t tacc, int q,
                                              int half, int ew, int lane, EpiSmem* ep, volatile int* abort,
                                              uint32_t acce_bar, unsigned epoch) {
  constexpr int HPT = 128 / DH;   // heads per 128-row tile
  constexpr int NTH = 256 / HPT;  // threads per head
  constexpr int NWH = NTH / 32;   // warps per head
  constexpr int CPT = DH / 16;    // columns per thread
  constexpr int HALF = DH / 2;    // accumulator columns each loader thread copies
  const Shape& s = a.s;
  // (1) copy this thread's TMEM row (its head block, its half of the columns) to registers
  const int trow = q * 32 + lane;                 // tile row = TMEM lane
  const int lslot = trow / DH;                    // head slot of that row
  float rowv[HALF];
  {
    const uint32_t ta = tacc + static_cast<uint32_t>(lslot * DH + half * HALF);
#pragma unroll
    for (int c0 = 0; c0 < HALF; c0 += 32) {
      uint32_t v[32];
      tmem_ld32(ta + c0, v);
#pragma unroll
      for (int e = 0; e < 32; ++e) rowv[c0 + e] = __uint_as_float(v[e]);
    }
    tmem_ld_wait();
  }
  tc_fence_before();
  mbar_arrive(acce_bar);  // G_Q is in registers: the accumulator is free for the next tile
  // (2) re-distribute G_Q into the block layout, one lane quarter at a time
  const int hs = ew / NWH, ewh = ew % NWH;
  const int rs = lane >> 4, cg = lane & 15;
  const int rb = 16 * ewh + 8 * rs;               // first of my 8 rows inside the head block
  const int cb = CPT * cg;                        // first of my columns
  const int myq = (hs * DH + rb) >> 5;            // lane quarter holding my rows
  float gq[8][CPT];
  float* stage = &ep->stage[0][0][0];
#pragma unroll 1
  for (int qq = 0; qq < 4; ++qq) {
    if (q == qq) {
#pragma unroll
      for (int c = 0; c < HALF; c += 4)
        *reinterpret_cast<float4*>(stage + lane * 68 + plane_off<CPT>(half * HALF + c, 68)) =
            make_float4(rowv[c], rowv[c + 1], rowv[c + 2], rowv[c + 3]);
    }
    named_bar_sync(5, 256);
    if (myq == qq) {
      const int r0 = hs * DH + rb - 32 * qq;
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int k = 0; k < CPT; k += 4) {
          const float4 g4 = *reinterpret_cast<const float4*>(stage + (r0 + i) * 68 + plane_off<CPT>(cb + k, 68));
          gq[i][k] = g4.x; gq[i][k + 1] = g4.y; gq[i][k + 2] = g4.z; gq[i][k + 3] = g4.w;
        }
    }
    named_bar_sync(5, 256);
  }
  const int head = idx * HPT + hs;
  if (head >= s.nq) return;  // whole head groups: a ragged last tile has an empty slot
  // (3) wait for the key tile, then G_K (block layout) and z0
  const int bar = 1 + hs;
  const int th = ewh * 32 + lane;                 // thread index inside the head group
  const int g = head / s.G;
  const int tk = (g * DH) / 128, og = (g * DH) % 128;
  const unsigned* flag = a.flags + layer * s.tiles_k + tk;
  const unsigned* vflag = a.vflags + layer * s.tiles_k + tk;
  if (th == 0)
    ep->ok[hs] = (wait_flag(flag, epoch, abort, a.status) && wait_flag(vflag, epoch, abort, a.status)) ? 1 : 0;
  named_bar_sync(bar, NTH);
  if (!ep->ok[hs]) return;
  (void)ld_acquire_u32(flag);
  (void)ld_acquire_u32(vflag);
  // G_K is stored transposed: element (j, i) holds G_K[i][j]; rows rb.. are contiguous.
  const float* GK = a.gk + static_cast<size_t>(layer * s.tiles_k + tk) * 16384u + og * 128 + og;
  float gk[8][CPT];
#pragma unroll
  for (int k = 0; k < CPT; ++k) {
    const float4 a0 = __ldcg(reinterpret_cast<const float4*>(GK + (cb + k) * 128 + rb));
    const float4 a1 = __ldcg(reinterpret_cast<const float4*>(GK + (cb + k) * 128 + rb + 4));
    gk[0][k] = a0.x; gk[1][k] = a0.y; gk[2][k] = a0.z; gk[3][k] = a0.w;
    gk[4][k] = a1.x; gk[5][k] = a1.y; gk[6][k] = a1.z; gk[7][k] = a1.w;
  }
  const size_t hidx = static_cast<size_t>(layer) * s.nq + head;
  // x and t' live in the plane layout (row stride 0: one "row" per slot).
  float* xs = &ep->xs[hs][0][0];
  float* ts = &ep->ts[hs][0][0];
  if (th < DH) {  // z0 = B v from the unnormalised v rows: x = z0 / ||v|| (0 for a zero v)
    const float inv = safe_inv_sqrt(__ldcg(a.vn2 + hidx));
    xs[vec_off<CPT>(th)] = (__ldcg(a.z0 + (hidx * 2) * DH + th) + __ldcg(a.z0 + (hidx * 2 + 1) * DH + th)) * inv;
  }
  named_bar_sync(bar, NTH);
  const bool writer = (lane & 1) == 0;  // one of the two lanes holding a row total
  // Each half-warp holds all d_h columns of x (and, after the middle barrier, of t'), so
  // the dot products S1 = x.t' and S2 = y.w are half-warp sums that overlap the next
  // matvec.  Inside the loop any normalising factor works as long as S2 and the tracked
  // scale use the same one: rsqrt(S1) is used, and sigma = sqrt(S1) / sqrt(S2 of the
  // previous iteration) is formed once, with IEEE operations, after the loop.
  float c2 = 1.0f, c2_prev = 1.0f, s1_last = 0.0f, inv1 = 0.0f, y = 0.0f;
  float tv[CPT];
#pragma unroll
  for (int k = 0; k < CPT; ++k) tv[k] = 0.0f;
  int ridx = 0;
  for (int it = 0; it < a.iters; ++it) {
    float xv[CPT];
#pragma unroll
    for (int k = 0; k < CPT; k += 4) {
      const float4 x4 = *reinterpret_cast<const float4*>(xs + vec_off<CPT>(cb + k));
      xv[k] = x4.x; xv[k + 1] = x4.y; xv[k + 2] = x4.z; xv[k + 3] = x4.w;
    }
    if (it > 0) {  // S2 of the previous iteration: y.w = inv1 * t'.w, w being this x
      float q = 0.0f;
#pragma unroll
      for (int k = 0; k < CPT; ++k) q = fmaf(tv[k], xv[k], q);
      const float s2 = halfwarp_sum(q) * inv1;
      c2 = s2 < 0.0f ? 0.0f : s2;  // rounding can dip below 0; NaN must survive
    }
    // t' = G_Q x
    float part[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float acc0 = 0.0f;
#pragma unroll
      for (int k = 0; k < CPT; ++k) acc0 = fmaf(gq[i][k], xv[k], acc0);
      part[i] = acc0;
    }
    const float tp = halfwarp_transpose_reduce8(part, lane, ridx);
    const int row = rb + ridx;
    if (writer) ts[vec_off<CPT>(row)] = tp;
    named_bar_sync(bar, NTH);
    // S1 = x.t';  w = G_K y with y = t' / sqrt(S1);  next x = w
#pragma unroll
    for (int k = 0; k < CPT; k += 4) {
      const float4 t4 = *reinterpret_cast<const float4*>(ts + vec_off<CPT>(cb + k));
      tv[k] = t4.x; tv[k + 1] = t4.y; tv[k + 2] = t4.z; tv[k + 3] = t4.w;
    }
    float q1 = 0.0f;
#pragma unroll
    for (int k = 0; k < CPT; ++k) q1 = fmaf(xv[k], tv[k], q1);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float acc0 = 0.0f;
#pragma unroll
      for (int k = 0; k < CPT; ++k) acc0 = fmaf(gk[i][k], tv[k], acc0);
      part[i] = acc0;
    }
    float s1 = halfwarp_sum(q1);
    s1 = s1 < 0.0f ? 0.0f : s1;
    inv1 = s1 == 0.0f ? 0.0f : rsqrtf(s1);  // zero guard that lets a NaN through
    s1_last = s1;
    c2_prev = c2;
    const float wrow = halfwarp_transpose_reduce8(part, lane, ridx) * inv1;
    y = tp * inv1;
    if (writer) xs[vec_off<CPT>(row)] = wrow;
    named_bar_sync(bar, NTH);
  }
  // ||v'||^2 of the last iteration (for y / ||v'||), and sigma = ||M v_{k-1}||
  float n = 0.0f;
  if (a.iters > 0) {
    float q = 0.0f;
#pragma unroll
    for (int k = 0; k < CPT; k += 4) {
      const float4 x4 = *reinterpret_cast<const float4*>(xs + vec_off<CPT>(cb + k));
      q = fmaf(tv[k], x4.x, fmaf(tv[k + 1], x4.y, fmaf(tv[k + 2], x4.z, fmaf(tv[k + 3], x4.w, q))));
    }
    const float s2 = halfwarp_sum(q) * inv1;
    n = sqrtf(s2 < 0.0f ? 0.0f : s2);
  }
  const float sigma = c2_prev == 0.0f ? 0.0f : sqrtf(s1_last) / sqrtf(c2_prev);
  if (writer && a.iters > 0) a.ybuf[hidx * DH + rb + ridx] = n == 0.0f ? 0.0f : y / n;
  if (th == 0) {
    a.sigma[hidx] = sigma;
    if (!isfinite(sigma)) set_status(a.status, GAS_DEV_NONFINITE_SIGMA);
    if (a.scale_out != nullptr) {
      // s_l = c * max_h sigma_{l,h} (Eq. 15): every head folds its sigma into an
      // epoch-tagged maximum (epoch << 32 | bits; a word left by an earlier launch always
      // loses, and on the bit patterns of non-negative floats a NaN wins), then the
      // layer's last head writes the scale
      const float w = sigma == 0.0f ? 0.0f : sigma;  // no -0.0
      atomicMax(a.layer_max + layer, (static_cast<unsigned long long>(epoch) << 32) | __float_as_uint(w));
      __threadfence();
      if (atomicAdd(a.layer_cnt + layer, 1u) == static_cast<unsigned>(s.nq) - 1u) {
        __threadfence();
        const unsigned long long m = __ldcg(a.layer_max + layer);
        a.scale_out[layer] = a.scale_c * __uint_as_float(static_cast<unsigned>(m));
      }
    }
  }
}

// Chunks per ring stage: two when the v operand is narrow (at most 32 rows).
template <int NZ, bool GENERIC>
struct GramBps {
  static constexpr int value = NZ <= 32 ? 2 : 1;
};

// GENERIC: binary16 weights or the Conv1D layout, chosen at run time; the default
// instantiation (bf16, nn.Linear rows) has both folded away.
template <int NZ, int DH, bool FUSED, bool GENERIC>
__global__ void __launch_bounds__(GramWarps<FUSED>::kThreads, 1) gram_kernel(const __grid_constant__ GramArgs a) {
  constexpr int NE = 32 * GramWarps<FUSED>::kEpiWarps;  // epilogue threads
  constexpr int BPS = GramBps<NZ, GENERIC>::value;
  using Cfg = GramCfg<NZ, BPS, FUSED>;
  constexpr uint32_t kVOff = BPS * kTileBytes;                   // stage offset of the v operand boxes
  constexpr uint32_t kFOff = BPS * (kTileBytes + Cfg::kVBytes);  // ... of the fp32 v boxes (fused)
  constexpr int S = Cfg::kStages;
  constexpr uint32_t SB = Cfg::kStageBytes;
  static_assert(1023 + (4 * S + 2 * Cfg::kAcc + 1) * 8 + 64 + 127 + sizeof(EpiSmem) <= kSmemReserve,
                "alignment slack, barriers and epilogue scratch must fit in the reserve");
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment by pointer arithmetic on the shared array itself, so that the
  // compiler keeps every derived pointer in the shared address space.
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S * SB);
  uint64_t* full = bars;
  uint64_t* empty = bars + S;
  uint64_t* conv = bars + 2 * S;   // fused key stages: the v operand is converted
  uint64_t* vfull = bars + 3 * S;  // fused key stages: the fp32 v boxes have landed
  constexpr int NA = Cfg::kAcc;
  uint64_t* accf = bars + 4 * S;
  uint64_t* acce = accf + NA;
  uint64_t* done = acce + NA;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t ep_off = ((smem_u32(done) + 64u + 127u) & ~127u) - smem_u32(smem);
  EpiSmem* ep = reinterpret_cast<EpiSmem*>(smem + ep_off);
  volatile int no_abort_flag = 0;

  const Shape& s = a.s;
  const bool cols = GENERIC && s.cols != 0;
  const bool f16 = GENERIC && s.f16 != 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
      mbar_init(smem_u32(&conv[i]), 32 * GramWarps<FUSED>::kConvWarps + (FUSED ? 0 : 1));
      mbar_init(smem_u32(&vfull[i]), 1);
    }
    for (int i = 0; i < NA; ++i) {
      mbar_init(smem_u32(&accf[i]), 1);
      mbar_init(smem_u32(&acce[i]), NE);
    }
    mbar_init(smem_u32(done), 1);
    *abort = 0;
    fence_mbar_init();
  }
  // Bytes one weight box brings: 128 rows, or d_h of them when a d_h 80 / 96 head sits in
  // a 128-row tile; the rows below stay zero (written once here, never by TMA).
  const uint32_t wbox = cols ? kTileBytes : static_cast<uint32_t>((128 / DH) * s.rows) * 128u;
  if (wbox < kTileBytes) {
    for (int st = 0; st < S; ++st)
      for (int b = 0; b < BPS; ++b)
        for (uint32_t o = wbox + threadIdx.x * 16u; o < kTileBytes; o += blockDim.x * 16u)
          *reinterpret_cast<uint4*>(smem + st * SB + b * kTileBytes + o) = make_uint4(0, 0, 0, 0);
  }
  if (FUSED) {
    // v operand rows that no head uses (padding of NZ) must read as zero in every stage
    for (int st = 0; st < S; ++st)
      for (uint32_t o = threadIdx.x * 16u; o < BPS * Cfg::kVBytes; o += blockDim.x * 16u)
        *reinterpret_cast<uint4*>(smem + st * SB + kVOff + o) = make_uint4(0, 0, 0, 0);
  }
  fence_proxy_async_smem();
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // The write-back launched after this kernel may start its prologue and its first W^K
  // copies on the SMs this launch leaves; it waits for the whole launch before it reads y.
  griddep_launch_dependents();
  const uint32_t tmem = *tmem_slot;
  const int T = s.L * (s.tiles_k + s.tiles_q);
  const int D = lead_layers(s, gridDim.x);
  // Fused key stages: the conv[] and vfull[] barriers of stage st complete one phase per
  // key-tile use of st; bit st of a role's kpar holds the parity of its next such phase.

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_first();
      // The key tiles of the last layers stay in L2 (evict_last) for the write-back, which
      // walks the layers from the last one down: about 48 MB of them.
      const uint64_t pol_k = l2_policy_evict_last();
      const long long kbytes = static_cast<long long>(s.tiles_k) * 128 * s.d * 2;
      const int keep0 = s.L - static_cast<int>(max(1LL, (48LL << 20) / kbytes));
      uint32_t issued = 0, kpar = 0u, kmask = 0u;  // kmask bit st: the latest use of st was a key stage
      bool ok = true;
      for (int t = blockIdx.x; t < T && ok; t += gridDim.x) {
        const TileRef tr = decode_tile(s, D, t);
        const CUtensorMap* map = tr.is_k ? &a.maps_k[tr.layer] : &a.maps_q[tr.layer];
        const int row0 = tr.idx * 128;
        const int vrow0 = (tr.layer * s.tiles_k + tr.idx) * NZ;
        for (int kc = 0; kc < s.nkc; kc += BPS) {
          const uint32_t st = issued % S, ph = (issued / S) & 1u;
          if (!mbar_wait(smem_u32(&empty[st]), ph ^ 1u, abort, a.status)) { ok = false; break; }
          const uint32_t sx = smem_u32(smem + st * SB);
          const uint32_t fb = smem_u32(&full[st]);
          const int nb = min(BPS, s.nkc - kc);  // a ragged last stage holds fewer chunks
          const uint32_t vfb = smem_u32(&vfull[st]);
          if (FUSED) {
            mbar_arrive_expect_tx(fb, static_cast<uint32_t>(nb) * wbox);
            if (tr.is_k) mbar_arrive_expect_tx(vfb, static_cast<uint32_t>(nb) * Cfg::kFBytes);
          } else {
            mbar_arrive_expect_tx(fb, static_cast<uint32_t>(nb) * (tr.is_k ? wbox + Cfg::kVBytes : wbox));
          }
#pragma unroll
          for (int b = 0; b < BPS; ++b) {
            if (b >= nb) break;
            const uint32_t bx = sx + b * kTileBytes;
            if (cols) {  // out-features contiguous: two 64-row halves of the tile, MN-major
              tma_load_2d(bx, map, fb, row0, (kc + b) * 64, pol);
              tma_load_2d(bx + kTileBytes / 2, map, fb, row0 + 64, (kc + b) * 64, pol);
            } else {
              tma_load_3d(bx, map, fb, (kc + b) * 64, 0, row0 / DH,  // 128/d_h heads of d_h rows
                          tr.is_k && tr.layer >= keep0 ? pol_k : pol);
            }
            if (tr.is_k) {
              if (FUSED)  // fp32 rows of the tile's heads: layer * nq + first head of the tile
                tma_load_2d(sx + kFOff + b * Cfg::kFBytes, &a.map_vf, vfb, (kc + b) * 64,
                            tr.layer * s.nq + tr.idx * (128 / DH) * s.G, pol);
              else
                tma_load_2d(sx + kVOff + b * Cfg::kVBytes, a.map_v, fb, (kc + b) * 64, vrow0, pol);
            }
          }
          if (FUSED) {
            kmask = tr.is_k ? (kmask | (1u << st)) : (kmask & ~(1u << st));
            if (tr.is_k) kpar ^= 1u << st;
          }
          ++issued;
        }
      }
      // Every copy still in flight targets this CTA's shared memory: wait for them to land
      // (the latest use of each stage; fp32 v boxes of key stages land on vfull[]).
      const uint32_t first = issued > static_cast<uint32_t>(S) ? issued - S : 0u;
      for (uint32_t i = first; i < issued; ++i) {
        const uint32_t st = i % S;
        mbar_wait(smem_u32(&full[st]), (i / S) & 1u, &no_abort_flag, a.status);
        if (FUSED && ((kmask >> st) & 1u))
          mbar_wait(smem_u32(&vfull[st]), ((kpar >> st) & 1u) ^ 1u, &no_abort_flag, a.status);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (one thread) ----------------
    if (lane == 0) {
      // Conv1D weights arrive MN-major (A and B of G = X X^T, A of Z = X V^T).
      const uint32_t idG = idesc_f32acc(128, 128, f16) | (cols ? (1u << 15) | (1u << 16) : 0u);
      const uint32_t idZ = idesc_f32acc(128, NZ, f16) | (cols ? (1u << 15) : 0u);
      uint32_t consumed = 0, tc = 0, kpar = 0u;
      bool ok = true;
      for (int t = blockIdx.x; t < T && ok; t += gridDim.x) {
        const TileRef tr = decode_tile(s, D, t);
        const uint32_t acc = tc % NA, aph = (tc / NA) & 1u;
        if (!mbar_wait(smem_u32(&acce[acc]), aph ^ 1u, abort, a.status)) break;
        tc_fence_after();
        const uint32_t dG = tmem + acc * 128u;
        const uint32_t dZ = tmem + NA * 128u + acc * static_cast<uint32_t>(NZ);
        for (int kc = 0; kc < s.nkc; kc += BPS) {
          const uint32_t st = consumed % S, ph = (consumed / S) & 1u;
          if (!mbar_wait(smem_u32(&full[st]), ph, abort, a.status)) { ok = false; break; }
          if (FUSED && tr.is_k) {
            if (!mbar_wait(smem_u32(&conv[st]), (kpar >> st) & 1u, abort, a.status)) { ok = false; break; }
            kpar ^= 1u << st;
          }
          tc_fence_after();
          const uint32_t sx = smem_u32(smem + st * SB);
          const int nb = min(BPS, s.nkc - kc);
#pragma unroll
          for (int b = 0; b < BPS; ++b) {
            if (b >= nb) break;
            const uint32_t bx = sx + b * kTileBytes;
            // K-major: +32 B per K16 step; MN-major (two 64-row atoms 8 KB apart): +2048 B
            const uint64_t ad = cols ? desc_mnmajor_sw128_2atoms(bx, kTileBytes / 2) : desc_kmajor_sw128(bx);
            const uint64_t astep = cols ? 128u : 2u;
            const uint64_t vd = desc_kmajor_sw128(sx + kVOff + b * Cfg::kVBytes);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint32_t accum = ((kc + b) | k) != 0 ? 1u : 0u;
              umma_bf16(dG, ad + astep * k, ad + astep * k, idG, accum);
              if (tr.is_k) umma_bf16(dZ, ad + astep * k, vd + 2u * k, idZ, accum);
            }
          }
          umma_commit(smem_u32(&empty[st]));
          ++consumed;
        }
        if (!ok) break;
        umma_commit(smem_u32(&accf[acc]));
        ++tc;
      }
      // Retire every MMA before tensor memory and shared memory go away.
      umma_commit(smem_u32(done));
      mbar_wait(smem_u32(done), 0u, &no_abort_flag, a.status);
    }
  } else if (warp < 2 + GramWarps<FUSED>::kEpiWarps) {
    // ---------------- epilogue: TMEM -> global ----------------
    const int q = warp & 3;  // tcgen05.ld: warp w may read TMEM lanes 32*(w%4) .. +31
    const int row = q * 32 + lane;
    const int half = (warp - 2) >> 2;  // fused: two threads per row, one per half of its columns
    constexpr int CW = 128 * 128 / NE;  // accumulator columns per thread when storing G
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const int gpt = 128 / s.dh;
    const unsigned epoch = FUSED ? __ldcg(a.epoch) : 0u;
    uint32_t tc = 0;
    for (int t = blockIdx.x; t < T; t += gridDim.x) {
      const TileRef tr = decode_tile(s, D, t);
      const uint32_t acc = tc % NA, aph = (tc / NA) & 1u;
      const bool got = mbar_wait(smem_u32(&accf[acc]), aph, abort, a.status);
      __syncwarp();  // tcgen05.ld is warp-collective: reconverge after the per-lane wait
      // One decision for all epilogue warps, so none of them can be left alone at a
      // named barrier further down when another gave up.
      if (!named_bar_and(4, NE, got)) break;
      tc_fence_after();
      if (FUSED && !tr.is_k) {  // (hands the accumulator back itself, right after reading G_Q)
        fused_iterate<DH>(a, tr.layer, tr.idx, tmem + lane_off + acc * 128u, q, half, warp - 2, lane, ep,
                          abort, smem_u32(&acce[acc]), epoch);
        ++tc;
        continue;
      }
      float* Gout = (tr.is_k ? a.gk : a.gq) +
                    (static_cast<size_t>(tr.layer) * (tr.is_k ? s.tiles_k : s.tiles_q) + tr.idx) * 16384u;
#pragma unroll 1
      for (int c0 = half * CW; c0 < half * CW + CW; c0 += 16) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_off + acc * 128u + c0, r);
        tmem_ld_wait();
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) Gout[(c0 + jj) * 128 + row] = __uint_as_float(r[jj]);
      }
      if (tr.is_k && half == 0) {
        const int gi = row / s.dh, i = row % s.dh;
        const int g = tr.idx * gpt + gi;
        const int twoG = 2 * s.G;
#pragma unroll 1
        for (int c0 = 0; c0 < NZ; c0 += 16) {
          uint32_t r[16];
          tmem_ld16(tmem + lane_off + NA * 128u + acc * static_cast<uint32_t>(NZ) + c0, r);
          tmem_ld_wait();
#pragma unroll
          for (int jj = 0; jj < 16; ++jj) {
            const int rel = c0 + jj - gi * twoG;
            if (g < s.nkv && rel >= 0 && rel < twoG) {
              const int half = rel >= s.G ? 1 : 0;
              const int head = g * s.G + rel - half * s.G;
              a.z0[((static_cast<size_t>(tr.layer) * s.nq + head) * 2 + half) * s.dh + i] =
                  __uint_as_float(r[jj]);
            }
          }
        }
      }
      if (FUSED && tr.is_k) {  // publish G_K and z0 of this key tile to the query tiles' epilogues
        __threadfence();
        named_bar_sync(3, NE);
        if (row == 0 && half == 0) st_release_u32(a.flags + tr.layer * s.tiles_k + tr.idx, epoch);
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&acce[acc]));
      ++tc;
    }
  } else if constexpr (FUSED) {
    // ---------------- converters: fp32 v rows -> bf16 / f16 hi + lo operand rows --------
    // Per key stage and chunk, thread ct takes 8 consecutive columns (one 16-byte unit of
    // the SW128 K-major operand) of head row r = u / 8 for u = ct, ct + 64, ...; it writes
    // the hi part to operand row gi*2G + j and the lo part to gi*2G + G + j (head j of
    // group gi of the tile) and sums the squares of its v entries.  The rows are not
    // normalised: the epilogue scales z0 by 1/||v|| from these sums.
    constexpr int NC = 32 * GramWarps<FUSED>::kConvWarps;
    constexpr int UMAX = (NZ / 2) * 8 / NC > 0 ? (NZ / 2) * 8 / NC : 1;
    const int ct = threadIdx.x - 32 * (2 + GramWarps<FUSED>::kEpiWarps);
    const int rt = (128 / DH) * s.G;  // head rows of a key tile (<= NZ / 2)
    const unsigned epoch = __ldcg(a.epoch);
    const uint32_t ns = static_cast<uint32_t>((s.nkc + BPS - 1) / BPS);  // stages per tile
    uint32_t cnt = 0, kpar = 0u;
    bool ok = true;
    for (int t = blockIdx.x; t < T && ok; t += gridDim.x) {
      const TileRef tr = decode_tile(s, D, t);
      if (!tr.is_k) {  // query tiles: no v operand, only the stage count moves on
        cnt += ns;
        continue;
      }
      float n2[UMAX];
#pragma unroll
      for (int i = 0; i < UMAX; ++i) n2[i] = 0.0f;
      for (int kc = 0; kc < s.nkc; kc += BPS) {
        const uint32_t st = cnt % S;
        if (!mbar_wait(smem_u32(&vfull[st]), (kpar >> st) & 1u, abort, a.status)) { ok = false; break; }
        const int nb = min(BPS, s.nkc - kc);
#pragma unroll
        for (int b = 0; b < BPS; ++b) {
          if (b >= nb) break;
          const uint8_t* F = smem + st * SB + kFOff + b * Cfg::kFBytes;
          uint8_t* V = smem + st * SB + kVOff + b * Cfg::kVBytes;
#pragma unroll
          for (int i = 0; i < UMAX; ++i) {
            const int u = ct + NC * i;
            const int r = u >> 3, c8 = u & 7;
            if (r < rt) {
              const float4 x0 = *reinterpret_cast<const float4*>(F + r * 256 + c8 * 32);
              const float4 x1 = *reinterpret_cast<const float4*>(F + r * 256 + c8 * 32 + 16);
              const float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
              uint32_t hb[8], lb[8];
#pragma unroll
              for (int e = 0; e < 8; ++e) {
                n2[i] = fmaf(xv[e], xv[e], n2[i]);
                split_hilo(xv[e], f16, hb[e], lb[e]);
              }
              const int gi = r / s.G, j = r - gi * s.G;
              const int rh = gi * 2 * s.G + j, rl = rh + s.G;
              *reinterpret_cast<uint4*>(V + rh * 128 + ((c8 ^ (rh & 7)) << 4)) =
                  make_uint4(hb[0] | (hb[1] << 16), hb[2] | (hb[3] << 16), hb[4] | (hb[5] << 16), hb[6] | (hb[7] << 16));
              *reinterpret_cast<uint4*>(V + rl * 128 + ((c8 ^ (rl & 7)) << 4)) =
                  make_uint4(lb[0] | (lb[1] << 16), lb[2] | (lb[3] << 16), lb[4] | (lb[5] << 16), lb[6] | (lb[7] << 16));
            }
          }
        }
        fence_proxy_async_smem();  // the tensor core reads what these generic stores wrote
        mbar_arrive(smem_u32(&conv[st]));
        kpar ^= 1u << st;
        ++cnt;
      }
      if (!ok) break;
      // ||v||^2 of every head of the tile, then this tile's v-norm flag
      const int head0 = tr.idx * (128 / DH) * s.G;
#pragma unroll
      for (int i = 0; i < UMAX; ++i) {
        float v2 = n2[i];
        v2 += __shfl_xor_sync(0xFFFFFFFFu, v2, 1);
        v2 += __shfl_xor_sync(0xFFFFFFFFu, v2, 2);
        v2 += __shfl_xor_sync(0xFFFFFFFFu, v2, 4);
        const int u = ct + NC * i;
        const int r = u >> 3;
        if ((u & 7) == 0 && r < rt && head0 + r < s.nq)
          a.vn2[static_cast<size_t>(tr.layer) * s.nq + head0 + r] = v2;
      }
      named_bar_sync(6, NC);
      if (ct == 0) {
        __threadfence();
        st_release_u32(a.vflags + tr.layer * s.tiles_k + tr.idx, epoch);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if (FUSED && threadIdx.x == 0) {
    // The last CTA to finish (every CTA gets here, also after giving up on a bounded
    // wait) clears the per-layer head counts and advances the flag epoch for the next
    // launch; every CTA of this cooperative launch read the epoch at its start, and a
    // replayed CUDA graph never takes this launch's flags for its own.
    __threadfence();
    if (atomicAdd(a.done_cnt, 1u) == gridDim.x - 1u) {
      for (int l = 0; l < s.L; ++l) a.layer_cnt[l] = 0u;
      *a.done_cnt = 0u;
      const unsigned n = __ldcg(a.epoch) + 1u;
      *a.epoch = n == 0u ? 1u : n;
      __threadfence();
    }
  }
}

// ---- k power iterations per head in R^{d_h} -------------------------------------------
// 256 threads hold G_Q and G_K in registers: warp w owns rows [w*DH/8, (w+1)*DH/8),
// lane l owns columns [l*DH/32, (l+1)*DH/32).  A matvec is 64 (d_h 128) FMAs per
// thread, a 16-shuffle transpose reduction per warp and one shared-memory exchange.
template <int DH>
__global__ void __launch_bounds__(256) iterate_kernel(const __grid_constant__ IterArgs a) {
  constexpr int RPW = DH / 8;
  constexpr int CPL = DH / 32;
  const Shape& s = a.s;
  const size_t hidx = blockIdx.x;
  const int l = static_cast<int>(hidx / s.nq), h = static_cast<int>(hidx % s.nq);
  const int g = h / s.G;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int oq = (h * DH) % 128, ok = (g * DH) % 128;
  const float* GQ = a.gq + (static_cast<size_t>(l) * s.tiles_q + (h * DH) / 128) * 16384u + oq * 128 + oq;
  const float* GK = a.gk + (static_cast<size_t>(l) * s.tiles_k + (g * DH) / 128) * 16384u + ok * 128 + ok;

  float gq[RPW][CPL], gk[RPW][CPL];
#pragma unroll
  for (int rr = 0; rr < RPW; ++rr) {
    const int r = warp * RPW + rr;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      gq[rr][c] = __ldg(GQ + r * 128 + lane * CPL + c);
      gk[rr][c] = __ldg(GK + r * 128 + lane * CPL + c);
    }
  }
  __shared__ float zs[DH], ts[DH], ws[DH];
  if (tid < DH) zs[tid] = a.z0[(hidx * 2 + 0) * DH + tid] + a.z0[(hidx * 2 + 1) * DH + tid];
  __syncthreads();
  float z[CPL], y[CPL];
#pragma unroll
  for (int c = 0; c < CPL; ++c) z[c] = zs[lane * CPL + c];
  // The loop normalises with rsqrt: z = c * B v with c = rsqrt(n^2) * sqrt(n^2) of the
  // previous iteration (1 for z0), so sigma = sqrt(z . t) / c and y / ||v'|| are formed
  // once, with IEEE operations, after the loop.
  float inv_n = 1.0f, n2_prev = 1.0f;         // this iteration's c = inv_n * sqrt(n2_prev)
  float s2_last = 0.0f, in_last = 1.0f, n2_c = 1.0f;
  for (int it = 0; it < a.iters; ++it) {
    // t = G_Q z  (= A u');  sigma^2 = z . t (= ||u'||^2);  y = t / sigma (= A u)
    float part[RPW];
#pragma unroll
    for (int rr = 0; rr < RPW; ++rr) {
      float acc = 0.0f;
#pragma unroll
      for (int c = 0; c < CPL; ++c) acc = fmaf(gq[rr][c], z[c], acc);
      part[rr] = acc;
    }
    int idx;
    float red = warp_transpose_reduce<RPW>(part, lane, idx);
    if (transpose_reduce_writer<RPW>(lane)) ts[warp * RPW + idx] = red;
    __syncthreads();
    float t[CPL], s2 = 0.0f;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      t[c] = ts[lane * CPL + c];
      s2 = fmaf(z[c], t[c], s2);
    }
    s2 = warp_sum(s2);
    s2 = s2 < 0.0f ? 0.0f : s2;  // rounding can dip below 0; NaN must survive
    s2_last = s2;
    in_last = inv_n;
    n2_c = n2_prev;
    const float inv_s = s2 == 0.0f ? 0.0f : rsqrtf(s2);  // zero guard that lets a NaN through
#pragma unroll
    for (int c = 0; c < CPL; ++c) y[c] = t[c] * inv_s;
    // w = G_K y  (= B v');  n^2 = y . w (= ||v'||^2);  z = w / n (= B v)
#pragma unroll
    for (int rr = 0; rr < RPW; ++rr) {
      float acc = 0.0f;
#pragma unroll
      for (int c = 0; c < CPL; ++c) acc = fmaf(gk[rr][c], y[c], acc);
      part[rr] = acc;
    }
    red = warp_transpose_reduce<RPW>(part, lane, idx);
    if (transpose_reduce_writer<RPW>(lane)) ws[warp * RPW + idx] = red;
    __syncthreads();
    float wv[CPL], n2 = 0.0f;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      wv[c] = ws[lane * CPL + c];
      n2 = fmaf(y[c], wv[c], n2);
    }
    n2 = warp_sum(n2);
    n2 = n2 < 0.0f ? 0.0f : n2;
    inv_n = n2 == 0.0f ? 0.0f : rsqrtf(n2);
    n2_prev = n2;
#pragma unroll
    for (int c = 0; c < CPL; ++c) z[c] = wv[c] * inv_n;
  }
  const float cz = in_last * sqrtf(n2_c);
  const float sigma = cz == 0.0f ? 0.0f : sqrtf(s2_last) / cz;
  const float ny = sqrtf(n2_prev);
  if (warp == 0) {
#pragma unroll
    for (int c = 0; c < CPL; ++c) a.ybuf[hidx * DH + lane * CPL + c] = ny == 0.0f ? 0.0f : y[c] / ny;
  }
  if (tid == 0) {
    a.sigma[hidx] = sigma;
    if (!isfinite(sigma)) set_status(a.status, GAS_DEV_NONFINITE_SIGMA);
    if (a.scale_out != nullptr) atomic_max_nonneg(&a.scale_out[l], a.scale_c * sigma);
  }
}

template <int NZ, int DH, bool FUSED, bool GENERIC>
cudaError_t launch_gram_cfg(const GramArgs& a, int num_sms, cudaStream_t st) {
  using Cfg = GramCfg<NZ, GramBps<NZ, GENERIC>::value, FUSED>;
  auto kern = gram_kernel<NZ, DH, FUSED, GENERIC>;
  static unsigned long long configured = 0;  // one bit per device: the attribute is per device
  cudaError_t e = set_smem_per_device(reinterpret_cast<const void*>(kern), static_cast<int>(Cfg::kSmem), configured);
  if (e != cudaSuccess) return e;
  const int T = a.s.L * (a.s.tiles_k + a.s.tiles_q);
  const int grid = T < num_sms ? T : num_sms;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(GramWarps<FUSED>::kThreads);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // all CTAs co-resident: key-tile flags cannot deadlock
  attr[0].val.cooperative = FUSED ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int NZ, int DH, bool FUSED>
cudaError_t launch_gram_variant(const GramArgs& a, int num_sms, cudaStream_t st) {
  return (a.s.cols || a.s.f16) ? launch_gram_cfg<NZ, DH, FUSED, true>(a, num_sms, st)
                               : launch_gram_cfg<NZ, DH, FUSED, false>(a, num_sms, st);
}

template <int NZ>
cudaError_t launch_gram_nz(const GramArgs& a, int num_sms, bool fused, cudaStream_t st) {
  if (a.s.dh == 128)
    return fused ? launch_gram_variant<NZ, 128, true>(a, num_sms, st) : launch_gram_variant<NZ, 128, false>(a, num_sms, st);
  if (a.s.dh == 64)
    return fused ? launch_gram_variant<NZ, 64, true>(a, num_sms, st) : launch_gram_variant<NZ, 64, false>(a, num_sms, st);
  return cudaErrorInvalidValue;
}

}  // namespace

template <int NZ>
size_t gram_smem_max() {
  const size_t a = GramCfg<NZ, GramBps<NZ, false>::value, false>::kSmem;
  const size_t b = GramCfg<NZ, GramBps<NZ, false>::value, true>::kSmem;
  const size_t c = GramCfg<NZ, GramBps<NZ, true>::value, false>::kSmem;
  const size_t d = GramCfg<NZ, GramBps<NZ, true>::value, true>::kSmem;
  const size_t ab = a > b ? a : b, cd = c > d ? c : d;
  return ab > cd ? ab : cd;
}

size_t gram_smem_bytes(int nz) {
  switch (nz) {
    case 16: return gram_smem_max<16>();
    case 32: return gram_smem_max<32>();
    case 64: return gram_smem_max<64>();
    case 128: return gram_smem_max<128>();
    default: return 0;
  }
}

cudaError_t launch_prep_v(const PrepArgs& a, cudaStream_t st) {
  prep_v_kernel<<<a.s.L * a.s.nq, 256, 0, st>>>(a);
  return cudaGetLastError();
}



cudaError_t launch_gram(const GramArgs& a, int num_sms, bool fused, cudaStream_t st) {
  switch (a.s.nz) {
    case 16: return launch_gram_nz<16>(a, num_sms, fused, st);
    case 32: return launch_gram_nz<32>(a, num_sms, fused, st);
    case 64: return launch_gram_nz<64>(a, num_sms, fused, st);
    case 128: return launch_gram_nz<128>(a, num_sms, fused, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_iterate(const IterArgs& a, cudaStream_t st) {
  if (a.s.dh == 128) iterate_kernel<128><<<a.s.L * a.s.nq, 256, 0, st>>>(a);
  else if (a.s.dh == 64) iterate_kernel<64><<<a.s.L * a.s.nq, 256, 0, st>>>(a);
  else return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace gas
