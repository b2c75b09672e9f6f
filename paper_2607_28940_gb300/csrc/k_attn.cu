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
  const float* Kg;      // [R, d] anchor key of this layer (LOCAL_GLOBAL), fp32
  const float* Vg;
  int l_local;
  int mode;
  int H, d;
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
  const int col = h * DH + sub * VEC;
  const int d = a.d;
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
  attend_rows<T, G>(q, len - lo, col, gmask, a.scale, sm, acc, [&](int t, const T*& kr, const T*& vr) {
    kr = Kc + (base + lo + t) * d;
    vr = Vc + (base + lo + t) * d;
  });
  if (a.mode == TXS_ATTN_LOCAL_GLOBAL) {
    const float* kg = a.Kg + static_cast<long long>(r) * d + col;
    const float* vg = a.Vg + static_cast<long long>(r) * d + col;
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
                              int mode, int H, int d, cudaStream_t s) {
  if (n_rows == 0) return cudaSuccess;
  CrossArgs a{row_req, n_rows, kv_off, kv_len, Kg, Vg, l_local, mode, H, d, 0.f};
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

template cudaError_t launch_serving_attn<float>(const float*, float*, const int*, int, int, int, int, int, cudaStream_t);
template cudaError_t launch_serving_attn<__nv_bfloat16>(const __nv_bfloat16*, __nv_bfloat16*, const int*, int, int,
                                                        int, int, int, cudaStream_t);
template cudaError_t launch_cross_attn<float>(const float*, float*, const float*, const float*, const int*, int,
                                              const int*, const int*, const float*, const float*, int, int, int, int,
                                              cudaStream_t);
template cudaError_t launch_cross_attn<__nv_bfloat16>(const __nv_bfloat16*, __nv_bfloat16*, const __nv_bfloat16*,
                                                      const __nv_bfloat16*, const int*, int, const int*, const int*,
                                                      const float*, const float*, int, int, int, int, cudaStream_t);

}  // namespace txs
