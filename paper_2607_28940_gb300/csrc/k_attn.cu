// Attention kernels of the decoder block.
//
// serving_attn: the serving-stream attention of App. B — a context row attends
// to the S context rows of its request, a candidate row to those S rows and to
// itself, never to another candidate.  At most S + 1 keys per row.
//
// cross_attn: the multi-query cross-attention of Sec. 4.1.2 — every candidate
// (and context) row of request r attends to the request's shared cached keys:
// in LOCAL_GLOBAL mode the min(L_local, L_r) most recent rows plus the pooled
// anchor (the sparse cross-attention equation), in FULL mode all L_r rows.
//
// Both: scale 1/sqrt(d_h), per-head online softmax in fp32.  A group of
// TPH = d_h / VEC threads (VEC = elements per 16-byte vector) owns one
// (row, head); dot products are reduced with warp shuffles inside the group.
#include <algorithm>

#include "txs_internal.cuh"

namespace txs {

namespace {

}  // namespace

namespace {

template <typename T, int DH>
struct Group {
  static constexpr int VEC = Vec16<T>::N;
  static constexpr int TPH = DH / VEC;
  static_assert(TPH >= 1 && TPH <= 32 && (TPH & (TPH - 1)) == 0, "threads per head");
  // Lanes of this thread's group: rows of one warp may differ (and so may
  // their key counts), so shuffles only synchronise the owning group.
  static __device__ __forceinline__ unsigned mask() {
    if (TPH == 32) return 0xffffffffu;
    const unsigned lane = threadIdx.x & 31;
    return ((1u << TPH) - 1u) << (lane & ~static_cast<unsigned>(TPH - 1));
  }
  static __device__ __forceinline__ float reduce(float x, unsigned m) {
#pragma unroll
    for (int o = TPH / 2; o > 0; o >>= 1) x += __shfl_xor_sync(m, x, o);
    return x;
  }
};

struct OnlineSoftmax {
  float m = -INFINITY, l = 0.f;
  // returns (scale for the old accumulator, weight of the new value)
  __device__ __forceinline__ void push(float s, float& corr, float& w) {
    const float mn = fmaxf(m, s);
    corr = expf(m - mn);
    w = expf(s - mn);
    l = l * corr + w;
    m = mn;
  }
};


// Online softmax over n_keys keys whose rows are `key_row(t)` (element
// pointers of width d in global memory; this thread's slice at `col`), one key
// per step (measured faster than batching keys: fewer registers, more warps).
template <typename T, typename G, typename KeyRow>
__device__ __forceinline__ void attend_rows(const float* q, int n_keys, int col, unsigned gmask, float scale,
                                            OnlineSoftmax& smx, float* acc, KeyRow key_row) {
  constexpr int VEC = G::VEC;
  for (int t = 0; t < n_keys; ++t) {
    const T* kr;
    const T* vr;
    key_row(t, kr, vr);
    float k[VEC], v[VEC];
    Vec16<T>::load(kr + col, k);
    Vec16<T>::load(vr + col, v);
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < VEC; ++i) dot = fmaf(q[i], k[i], dot);
    dot = G::reduce(dot, gmask) * scale;
    float corr, w;
    smx.push(dot, corr, w);
#pragma unroll
    for (int i = 0; i < VEC; ++i) acc[i] = acc[i] * corr + w * v[i];
  }
}

// Serving-stream attention: thread group per (row, head); a candidate row
// attends to the S context rows of its request and to itself, a context row to
// the S context rows.  The context rows' K/V are read by every row of the
// request and stay in L1.
template <typename T, int DH>
__global__ void __launch_bounds__(256) serving_attn_kernel(const T* __restrict__ qkv, T* __restrict__ out,
                                                           const int* __restrict__ row_req, int n_rows,
                                                           int n_cand_rows, int S, int H, int d, float scale) {
  pdl_launch_dependents();
  pdl_wait();
  using G = Group<T, DH>;
  constexpr int VEC = G::VEC;
  const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const long long pair = gid / G::TPH;
  const int sub = static_cast<int>(gid % G::TPH);
  if (pair >= static_cast<long long>(n_rows) * H) return;   // whole group
  const int row = static_cast<int>(pair / H);
  const int h = static_cast<int>(pair % H);
  const long long ld = 3LL * d;
  const int col = h * DH + sub * VEC;
  const unsigned gmask = G::mask();
  float q[VEC], acc[VEC];
  Vec16<T>::load(qkv + row * ld + col, q);
#pragma unroll
  for (int i = 0; i < VEC; ++i) acc[i] = 0.f;
  OnlineSoftmax smx;
  const int r = __ldg(row_req + row);
  const long long c0 = n_cand_rows + static_cast<long long>(r) * S;
  const int n_keys = S + (row < n_cand_rows ? 1 : 0);
  attend_rows<T, G>(q, n_keys, col, gmask, scale, smx, acc, [&](int t, const T*& kr, const T*& vr) {
    const long long krow = t < S ? c0 + t : row;
    kr = qkv + krow * ld + d;
    vr = qkv + krow * ld + 2 * d;
  });
  const float inv = 1.f / smx.l;
#pragma unroll
  for (int i = 0; i < VEC; ++i) acc[i] *= inv;
  Vec16<T>::store(out + static_cast<long long>(row) * d + col, acc);
}

struct CrossArgs {
  const int* row_req;
  int n_rows;
  const int* kv_off;    // [R+1] cache row offsets (capacity layout)
  const int* kv_len;    // [R]   current lengths
  const float* Kg;      // [R, dkv] anchor key of this layer (LOCAL_GLOBAL), fp32
  const float* Vg;
  int l_local;
  int mode;
  int H, d;
  int dkv, group;       // cached row width; query heads per K/V head
  float scale;
};

template <typename T, int DH>
__global__ void __launch_bounds__(256) cross_attn_kernel(const T* __restrict__ q_in, T* __restrict__ out,
                                                         const T* __restrict__ Kc, const T* __restrict__ Vc,
                                                         const CrossArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  using G = Group<T, DH>;
  constexpr int VEC = G::VEC;
  const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const long long pair = gid / G::TPH;
  const int sub = static_cast<int>(gid % G::TPH);
  if (pair >= static_cast<long long>(a.n_rows) * a.H) return;   // whole group
  const int row = static_cast<int>(pair / a.H);
  const int h = static_cast<int>(pair % a.H);
  const int col = h * DH + sub * VEC;                         // query / output columns
  const int ck = (h / a.group) * DH + sub * VEC;              // the same slice of its K/V head
  const int d = a.d, dkv = a.dkv;
  const unsigned gmask = G::mask();
  float q[VEC], acc[VEC];
  Vec16<T>::load(q_in + static_cast<long long>(row) * d + col, q);
#pragma unroll
  for (int i = 0; i < VEC; ++i) acc[i] = 0.f;
  OnlineSoftmax sm;
  const int r = __ldg(a.row_req + row);
  const int len = __ldg(a.kv_len + r);
  const long long base = __ldg(a.kv_off + r);
  const int lo = (a.mode == TXS_ATTN_LOCAL_GLOBAL) ? max(0, len - a.l_local) : 0;
  attend_rows<T, G>(q, len - lo, ck, gmask, a.scale, sm, acc, [&](int t, const T*& kr, const T*& vr) {
    kr = Kc + (base + lo + t) * dkv;
    vr = Vc + (base + lo + t) * dkv;
  });
  if (a.mode == TXS_ATTN_LOCAL_GLOBAL) {
    const float* kg = a.Kg + static_cast<long long>(r) * dkv + ck;
    const float* vg = a.Vg + static_cast<long long>(r) * dkv + ck;
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < VEC; ++i) dot = fmaf(q[i], __ldg(kg + i), dot);
    dot = G::reduce(dot, gmask) * a.scale;
    float corr, w;
    sm.push(dot, corr, w);
#pragma unroll
    for (int i = 0; i < VEC; ++i) acc[i] = acc[i] * corr + w * __ldg(vg + i);
  }
  const float inv = 1.f / sm.l;
#pragma unroll
  for (int i = 0; i < VEC; ++i) acc[i] *= inv;
  Vec16<T>::store(out + static_cast<long long>(row) * d + col, acc);
}

// LOCAL_GLOBAL cross-attention with the request's window staged in shared
// memory.  One CTA per (32 query rows, request): the window's key and value
// rows (at most kWin) and the anchor are copied once into shared memory; warp
// w takes heads w, w + 8, ..., and lane i the query row 32 c + i, so the 32
// lanes of a warp read the same key/value elements (shared-memory broadcast).
// Each thread computes all the row's scores for the head, the softmax and the
// weighted values in registers.
constexpr int kWin = 16;

struct CrossLgArgs {
  const int* cand_off;  // [R+1] candidate offsets (device)
  int n_cand, S;
  const int* kv_off;    // [R+1] cache row offsets
  const int* kv_len;    // [R]
  const float* Kg;      // [R, dkv] anchor key / value of this layer, fp32
  const float* Vg;
  int l_local, H, d;
  int dkv, group;       // cached row width; query heads per K/V head
  float scale_log2;     // log2(e) / sqrt(d_h)
};

template <typename T, int DH>
__global__ void __launch_bounds__(256) cross_lg_kernel(const T* __restrict__ q_in, T* __restrict__ out,
                                                       const T* __restrict__ Kc, const T* __restrict__ Vc,
                                                       const CrossLgArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  extern __shared__ __align__(16) uint8_t smem_lg[];
  const int d = a.d, dkv = a.dkv;
  float* sK = reinterpret_cast<float*>(smem_lg);              // [kWin][dkv], fp32
  float* sV = sK + kWin * dkv;                                // [kWin][dkv]
  float* sKg = sV + kWin * dkv;                               // [dkv]
  float* sVg = sKg + dkv;                                     // [dkv]
  const int r = blockIdx.y;
  const int c0 = __ldg(a.cand_off + r);
  const int M = __ldg(a.cand_off + r + 1) - c0;
  const int n_q = M + a.S;
  const int row0 = blockIdx.x * 32;
  if (row0 >= n_q) return;                                    // uniform
  const int len = __ldg(a.kv_len + r);
  const int lo = len > a.l_local ? len - a.l_local : 0;
  const int W = len - lo;                                     // <= kWin (checked on the host)
  const long long base = static_cast<long long>(__ldg(a.kv_off + r)) + lo;
  {
    constexpr int VE = Vec16<T>::N;                           // elements per 16 bytes
    const int per_row = dkv / VE;
    for (int i = threadIdx.x; i < W * per_row; i += blockDim.x) {
      const int t = i / per_row, c = (i - t * per_row) * VE;
      // converted once here: every lane (query row) reads every element
      float kf[VE], vf[VE];
      Vec16<T>::load(Kc + (base + t) * dkv + c, kf);
      Vec16<T>::load(Vc + (base + t) * dkv + c, vf);
#pragma unroll
      for (int e = 0; e < VE; e += 4) {
        *reinterpret_cast<float4*>(sK + t * dkv + c + e) = make_float4(kf[e], kf[e + 1], kf[e + 2], kf[e + 3]);
        *reinterpret_cast<float4*>(sV + t * dkv + c + e) = make_float4(vf[e], vf[e + 1], vf[e + 2], vf[e + 3]);
      }
    }
    for (int i = threadIdx.x; i < dkv; i += blockDim.x) {
      sKg[i] = __ldg(a.Kg + static_cast<long long>(r) * dkv + i);
      sVg[i] = __ldg(a.Vg + static_cast<long long>(r) * dkv + i);
    }
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = row0 + lane;                                  // query row within the request
  const bool valid = j < n_q;
  const long long grow = j < M ? static_cast<long long>(c0) + j
                               : a.n_cand + static_cast<long long>(r) * a.S + (j - M);
  for (int h = warp; h < a.H; h += (blockDim.x >> 5)) {
    const int col = h * DH;                                   // query / output columns
    const int ck = (h / a.group) * DH;                        // its K/V head
    float q[DH];
    if (valid) {
#pragma unroll
      for (int c = 0; c < DH; c += Vec16<T>::N) Vec16<T>::load(q_in + grow * d + col + c, q + c);
    } else {
#pragma unroll
      for (int c = 0; c < DH; ++c) q[c] = 0.f;
    }
#pragma unroll
    for (int c = 0; c < DH; ++c) q[c] *= a.scale_log2;
    // scores (log2 units): the window rows, then the anchor
    float sc[kWin + 1];
#pragma unroll
    for (int t = 0; t < kWin; ++t) {
      float dot = -INFINITY;
      if (t < W) {
        dot = 0.f;
#pragma unroll
        for (int c = 0; c < DH; c += 4) {
          const float4 k4 = *reinterpret_cast<const float4*>(sK + t * dkv + ck + c);
          dot = fmaf(q[c], k4.x, dot);
          dot = fmaf(q[c + 1], k4.y, dot);
          dot = fmaf(q[c + 2], k4.z, dot);
          dot = fmaf(q[c + 3], k4.w, dot);
        }
      }
      sc[t] = dot;
    }
    {
      float dot = 0.f;
#pragma unroll
      for (int c = 0; c < DH; c += 4) {
        const float4 k4 = *reinterpret_cast<const float4*>(sKg + ck + c);
        dot = fmaf(q[c], k4.x, dot);
        dot = fmaf(q[c + 1], k4.y, dot);
        dot = fmaf(q[c + 2], k4.z, dot);
        dot = fmaf(q[c + 3], k4.w, dot);
      }
      sc[kWin] = dot;
    }
    float mx = sc[kWin];
#pragma unroll
    for (int t = 0; t < kWin; ++t) mx = fmaxf(mx, sc[t]);
    float sum = 0.f;
#pragma unroll
    for (int t = 0; t <= kWin; ++t) {
      sc[t] = exp2f(sc[t] - mx);
      sum += sc[t];
    }
    // weighted values (q reused as the accumulator)
#pragma unroll
    for (int c = 0; c < DH; c += 4) {
      const float4 v4 = *reinterpret_cast<const float4*>(sVg + ck + c);
      q[c] = sc[kWin] * v4.x;
      q[c + 1] = sc[kWin] * v4.y;
      q[c + 2] = sc[kWin] * v4.z;
      q[c + 3] = sc[kWin] * v4.w;
    }
#pragma unroll
    for (int t = 0; t < kWin; ++t) {
      if (t < W) {
#pragma unroll
        for (int c = 0; c < DH; c += 4) {
          const float4 v4 = *reinterpret_cast<const float4*>(sV + t * dkv + ck + c);
          q[c] = fmaf(sc[t], v4.x, q[c]);
          q[c + 1] = fmaf(sc[t], v4.y, q[c + 1]);
          q[c + 2] = fmaf(sc[t], v4.z, q[c + 2]);
          q[c + 3] = fmaf(sc[t], v4.w, q[c + 3]);
        }
      }
    }
    if (valid) {
      const float inv = 1.f / sum;
#pragma unroll
      for (int c = 0; c < DH; ++c) q[c] *= inv;
#pragma unroll
      for (int c = 0; c < DH; c += Vec16<T>::N) Vec16<T>::store(out + grow * d + col + c, q + c);
    }
  }
}

template <typename T, int DH>
cudaError_t cross_launch(const T* q, T* out, const T* Kc, const T* Vc, CrossArgs a, cudaStream_t s) {
  const long long threads = static_cast<long long>(a.n_rows) * a.H * Group<T, DH>::TPH;
  const int blocks = static_cast<int>((threads + 255) / 256);
  a.scale = (1.0f / sqrtf(static_cast<float>(DH)));
  return launch_pdl(cross_attn_kernel<T, DH>, dim3(blocks), dim3(256), 0, s, q, out, Kc, Vc, a);
}

}  // namespace

template <typename T, int DH>
static cudaError_t serving_launch(const T* qkv, T* out, const int* row_req, int n_rows, int n_cand_rows, int S, int H,
                                  int d, cudaStream_t s) {
  const long long threads = static_cast<long long>(n_rows) * H * Group<T, DH>::TPH;
  const int blocks = static_cast<int>((threads + 255) / 256);
  return launch_pdl(serving_attn_kernel<T, DH>, dim3(blocks), dim3(256), 0, s, qkv, out, row_req, n_rows,
                    n_cand_rows, S, H, d, 1.0f / sqrtf(static_cast<float>(DH)));
}

template <typename T>
cudaError_t launch_serving_attn(const T* qkv, T* out, const int* row_req, int n_rows, int n_cand_rows, int S, int H,
                                int d, cudaStream_t s) {
  if (n_rows == 0) return cudaSuccess;
  prof_begin(KC_ATTN_SERVING, s);
  cudaError_t err;
  switch (d / H) {
    case 32: err = serving_launch<T, 32>(qkv, out, row_req, n_rows, n_cand_rows, S, H, d, s); break;
    case 64: err = serving_launch<T, 64>(qkv, out, row_req, n_rows, n_cand_rows, S, H, d, s); break;
    default: err = cudaErrorInvalidValue;
  }
  prof_end(KC_ATTN_SERVING, s);
  return err;
}

template <typename T>
cudaError_t launch_cross_attn(const T* q, T* out, const T* Kc, const T* Vc, const int* row_req, int n_rows,
                              const int* kv_off, const int* kv_len, const float* Kg, const float* Vg, int l_local,
                              int mode, int H, int Hkv, int d, cudaStream_t s) {
  if (n_rows == 0) return cudaSuccess;
  if (Hkv < 1 || H % Hkv) return cudaErrorInvalidValue;
  CrossArgs a{row_req, n_rows, kv_off, kv_len, Kg, Vg, l_local, mode, H, d, Hkv * (d / H), H / Hkv, 0.f};
  prof_begin(KC_ATTN_CROSS, s);
  cudaError_t err;
  switch (d / H) {
    case 32: err = cross_launch<T, 32>(q, out, Kc, Vc, a, s); break;
    case 64: err = cross_launch<T, 64>(q, out, Kc, Vc, a, s); break;
    default: err = cudaErrorInvalidValue;
  }
  prof_end(KC_ATTN_CROSS, s);
  return err;
}

template <typename T>
cudaError_t launch_cross_attn_lg(const T* q, T* out, const T* Kc, const T* Vc, const int* cand_off_dev,
                                 const int* cand_off_host, int n_req, int n_cand, int S, const int* kv_off,
                                 const int* kv_len, const float* Kg, const float* Vg, int l_local, int H, int Hkv,
                                 int d, cudaStream_t s) {
  const int dh = d / H;
  if (l_local > kWin || (dh != 32 && dh != 64) || d % 8 != 0) return cudaErrorNotSupported;
  if (Hkv < 1 || H % Hkv) return cudaErrorInvalidValue;
  const int dkv = Hkv * dh;
  int max_q = 0;
  for (int r = 0; r < n_req; ++r) max_q = std::max(max_q, cand_off_host[r + 1] - cand_off_host[r] + S);
  if (max_q == 0 || n_req == 0) return cudaSuccess;
  CrossLgArgs a{cand_off_dev, n_cand, S, kv_off, kv_len, Kg, Vg, l_local, H, d, dkv, H / Hkv,
                1.4426950408889634f / sqrtf(static_cast<float>(dh))};
  const size_t smem = static_cast<size_t>(2 * kWin * dkv) * sizeof(float) + 2 * dkv * sizeof(float);
  const dim3 grid((max_q + 31) / 32, n_req);
  prof_begin(KC_ATTN_CROSS, s);
  cudaError_t err;
  if (dh == 32) {
    if (smem > 48 * 1024) cudaFuncSetAttribute(cross_lg_kernel<T, 32>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    err = launch_pdl(cross_lg_kernel<T, 32>, grid, dim3(256), smem, s, q, out, Kc, Vc, a);
  } else {
    if (smem > 48 * 1024) cudaFuncSetAttribute(cross_lg_kernel<T, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    err = launch_pdl(cross_lg_kernel<T, 64>, grid, dim3(256), smem, s, q, out, Kc, Vc, a);
  }
  prof_end(KC_ATTN_CROSS, s);
  return err;
}

// LOCAL_GLOBAL cross-attention of the S context-token rows of every request
// (rows n_cand + r S + j of the packed layout), whose q the fused query
// projection left in `q`: one warp per (row, head).  Lane t < W scores the
// request's window row t, lane W its anchor (Sec. 4.1.2 sparse
// cross-attention equation, scale 1/sqrt(d_h)); the softmax runs across the
// lanes; lane c then sums the weighted values of output columns c, c + 32.
struct CtxAttnArgs {
  int n_req, n_cand, S, H, d, dkv, group, l_local;
  const int* kv_off;
  const int* kv_len;
  const float* Kg;
  const float* Vg;
  float scale_log2;
};

constexpr int kCtxKeys = 16;   // window rows (at most 15) + anchor

template <int DH>
__global__ void __launch_bounds__(256) ctx_attn_kernel(const __nv_bfloat16* __restrict__ q,
                                                       __nv_bfloat16* __restrict__ out,
                                                       const __nv_bfloat16* __restrict__ Kc,
                                                       const __nv_bfloat16* __restrict__ Vc, const CtxAttnArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (gw >= a.n_req * a.S * a.H) return;                     // uniform per warp
  const int i = gw / a.H, h = gw - i * a.H;
  const int r = i / a.S;
  const long long row = static_cast<long long>(a.n_cand) + i;
  const int kcol = (h / a.group) * DH;
  const int len = __ldg(a.kv_len + r);
  const int lo = len > a.l_local ? len - a.l_local : 0;
  const int W = len - lo;
  const long long base = static_cast<long long>(__ldg(a.kv_off + r)) + lo;
  // every load up front (one round of latency): q (all lanes), this lane's
  // key (window row `lane`, or the anchor for lane W), and this lane's value
  // columns (lane, lane + 32) of every key
  float qv[DH], kv[DH];
  float v0[kCtxKeys], v1[kCtxKeys];
#pragma unroll
  for (int c = 0; c < DH; c += 8) Vec16<__nv_bfloat16>::load(q + row * a.d + h * DH + c, qv + c);
  if (lane < W) {
#pragma unroll
    for (int c = 0; c < DH; c += 8) Vec16<__nv_bfloat16>::load(Kc + (base + lane) * a.dkv + kcol + c, kv + c);
  } else {
    const float* kg = a.Kg + static_cast<long long>(r) * a.dkv + kcol;
#pragma unroll
    for (int c = 0; c < DH; c += 4) {
      const float4 g4 = __ldg(reinterpret_cast<const float4*>(kg + c));
      kv[c] = g4.x; kv[c + 1] = g4.y; kv[c + 2] = g4.z; kv[c + 3] = g4.w;
    }
  }
  const float* vg = a.Vg + static_cast<long long>(r) * a.dkv + kcol;
#pragma unroll
  for (int t = 0; t < kCtxKeys; ++t) {
    v0[t] = v1[t] = 0.f;
    if (t < W) {
      const __nv_bfloat16* vr = Vc + (base + t) * a.dkv + kcol;
      v0[t] = __bfloat162float(vr[lane]);
      if (DH == 64) v1[t] = __bfloat162float(vr[lane + 32]);
    } else if (t == W) {
      v0[t] = __ldg(vg + lane);
      if (DH == 64) v1[t] = __ldg(vg + lane + 32);
    }
  }
  float s = -INFINITY;
  if (lane <= W) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c = 0; c < DH; ++c) acc[c & 3] = fmaf(qv[c], kv[c], acc[c & 3]);
    s = ((acc[0] + acc[1]) + (acc[2] + acc[3])) * a.scale_log2;
  }
  float mx = s;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  const float p = lane <= W ? exp2f(s - mx) : 0.f;
  float sum = p;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  // output columns lane, lane + 32 (DH = 64) of this head
  float o0 = 0.f, o1 = 0.f;
#pragma unroll
  for (int t = 0; t < kCtxKeys; ++t) {
    const float pt = __shfl_sync(0xffffffffu, p, t);   // 0 past the anchor
    o0 = fmaf(pt, v0[t], o0);
    if (DH == 64) o1 = fmaf(pt, v1[t], o1);
  }
  const float inv = 1.f / sum;
  __nv_bfloat16* dst = out + row * a.d + h * DH;
  dst[lane] = __float2bfloat16_rn(o0 * inv);
  if (DH == 64) dst[lane + 32] = __float2bfloat16_rn(o1 * inv);
}

cudaError_t launch_ctx_attn_lg(const __nv_bfloat16* q, __nv_bfloat16* out, const __nv_bfloat16* Kc,
                               const __nv_bfloat16* Vc, int n_req, int n_cand, int S, const int* kv_off,
                               const int* kv_len, const float* Kg, const float* Vg, int l_local, int H, int Hkv,
                               int d, cudaStream_t s) {
  const int dh = d / H;
  if ((dh != 32 && dh != 64) || l_local >= kCtxKeys || Hkv < 1 || H % Hkv) return cudaErrorInvalidValue;
  const long long warps = static_cast<long long>(n_req) * S * H;
  if (warps == 0) return cudaSuccess;
  CtxAttnArgs a{n_req, n_cand, S, H, d, Hkv * dh, H / Hkv, l_local, kv_off, kv_len, Kg, Vg,
                1.4426950408889634f / sqrtf(static_cast<float>(dh))};
  const dim3 grid(static_cast<unsigned>((warps + 7) / 8));
  prof_begin(KC_ATTN_CROSS, s);
  const cudaError_t err = dh == 64 ? launch_pdl(ctx_attn_kernel<64>, grid, dim3(256), 0, s, q, out, Kc, Vc, a)
                                   : launch_pdl(ctx_attn_kernel<32>, grid, dim3(256), 0, s, q, out, Kc, Vc, a);
  prof_end(KC_ATTN_CROSS, s);
  return err;
}

template cudaError_t launch_cross_attn_lg<float>(const float*, float*, const float*, const float*, const int*,
                                                 const int*, int, int, int, const int*, const int*, const float*,
                                                 const float*, int, int, int, int, cudaStream_t);
template cudaError_t launch_cross_attn_lg<__nv_bfloat16>(const __nv_bfloat16*, __nv_bfloat16*, const __nv_bfloat16*,
                                                         const __nv_bfloat16*, const int*, const int*, int, int, int,
                                                         const int*, const int*, const float*, const float*, int,
                                                         int, int, int, cudaStream_t);

template cudaError_t launch_serving_attn<float>(const float*, float*, const int*, int, int, int, int, int, cudaStream_t);
template cudaError_t launch_serving_attn<__nv_bfloat16>(const __nv_bfloat16*, __nv_bfloat16*, const int*, int, int,
                                                        int, int, int, cudaStream_t);
template cudaError_t launch_cross_attn<float>(const float*, float*, const float*, const float*, const int*, int,
                                              const int*, const int*, const float*, const float*, int, int, int, int,
                                              int, cudaStream_t);
template cudaError_t launch_cross_attn<__nv_bfloat16>(const __nv_bfloat16*, __nv_bfloat16*, const __nv_bfloat16*,
                                                      const __nv_bfloat16*, const int*, int, const int*, const int*,
                                                      const float*, const float*, int, int, int, int, int,
                                                      cudaStream_t);

}  // namespace txs
