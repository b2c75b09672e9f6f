// Cache-side kernels: attention pooling of the global anchor, its per-layer
// K/V projection, and the one-time weight preparation of txs_model_create.
//
// Attention pooling (Sec. 4.1.2, the global token of the local-global key set;
// Sec. 5.1, where pooling produces that token):
// alpha = softmax_i(phi_i . w_pool / sqrt(d)), g = sum_i alpha_i phi_i.  It is
// kept as an online-softmax state (m = max logit, s = sum exp(logit - m),
// acc = sum exp(logit - m) phi) so that an append (App. D incremental-encoding
// remark) merges new rows without revisiting old ones.  Rows are processed in
// chunks of kPoolChunk (one CTA each); chunk states are merged per request.
#include <algorithm>

#include "tc_ptx.cuh"

namespace txs {

constexpr int kPoolChunkV = 64;
extern const int kPoolChunk = kPoolChunkV;

namespace {

constexpr int kPoolWarps = 8;
constexpr int kPoolRowsPerWarp = kPoolChunkV / kPoolWarps;

// The last chunk CTA of request r to finish merges the request's nch_r chunk
// states part_r[c] = (m, s, acc[d]) (and, for an append, the stored state)
// into the pooling state and writes g = acc / s.  Called by every thread of
// a 256-thread CTA once its own chunk state is in part_r.
__device__ __forceinline__ void pool_merge_if_last(const float* pr, int nch_r, int d, int r, int merge_existing,
                                                   float* st_m, float* st_s, float* st_acc, float* g, int* counter) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  __shared__ int is_last;
  __threadfence();
  __syncthreads();
  if (tid == 0) is_last = atomicAdd(counter + r, 1) == nch_r - 1;
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  // chunk maxima and weighted sums as block reductions (thread t takes
  // chunks t, t + 256, ...), then each column's sum over the chunks with its
  // loads issued ahead of the multiply-adds; the order is fixed, so the
  // result is deterministic
  __shared__ float ch_scale[512];
  __shared__ float red[kPoolWarps];
  const float old_m = merge_existing ? st_m[r] : -INFINITY;
  const float old_s = merge_existing ? st_s[r] : 0.f;
  float mloc = -INFINITY;
  for (int ch = tid; ch < nch_r; ch += 256) mloc = fmaxf(mloc, __ldcg(pr + static_cast<long long>(ch) * (d + 2)));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
  if (lane == 0) red[warp] = mloc;
  __syncthreads();
  float Mr = old_m;
#pragma unroll
  for (int w8 = 0; w8 < kPoolWarps; ++w8) Mr = fmaxf(Mr, red[w8]);
  const float w_old = merge_existing ? expf(old_m - Mr) : 0.f;
  __syncthreads();                                  // red is reused below
  float sloc = 0.f;
  for (int ch = tid; ch < nch_r; ch += 256) {
    const float* pc = pr + static_cast<long long>(ch) * (d + 2);
    const float sc = expf(__ldcg(pc) - Mr);
    if (ch < 512) ch_scale[ch] = sc;
    sloc = fmaf(__ldcg(pc + 1), sc, sloc);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sloc += __shfl_xor_sync(0xffffffffu, sloc, o);
  if (lane == 0) red[warp] = sloc;
  __syncthreads();
  float Sr = __fmul_rn(old_s, w_old);
#pragma unroll
  for (int w8 = 0; w8 < kPoolWarps; ++w8) Sr = __fadd_rn(Sr, red[w8]);
  for (int k = tid; k < d; k += 256) {
    float a = merge_existing ? __fmul_rn(st_acc[static_cast<long long>(r) * d + k], w_old) : 0.f;
    int ch = 0;
    for (; ch + 8 <= nch_r && ch + 8 <= 512; ch += 8) {
      float pv[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) pv[u] = __ldcg(pr + static_cast<long long>(ch + u) * (d + 2) + 2 + k);
#pragma unroll
      for (int u = 0; u < 8; ++u) a = fmaf(pv[u], ch_scale[ch + u], a);
    }
    for (; ch < nch_r; ++ch) {
      const float* pc = pr + static_cast<long long>(ch) * (d + 2);
      const float sc = ch < 512 ? ch_scale[ch] : expf(__ldcg(pc) - Mr);
      a = fmaf(__ldcg(pc + 2 + k), sc, a);
    }
    st_acc[static_cast<long long>(r) * d + k] = a;
    g[static_cast<long long>(r) * d + k] = a / Sr;
  }
  __syncthreads();
  if (tid == 0) {
    st_m[r] = Mr;
    st_s[r] = Sr;
    counter[r] = 0;   // ready for the next call
  }
}

// One CTA per (chunk of kPoolChunk rows, request).  Each warp loads its rows
// (all loads issued before any arithmetic), computes the pooling logits with a
// warp reduction and folds the rows into an online-softmax state; the CTA then
// merges its warps' states.  One coalesced read of the behavior rows.
// MERGE = false (prefix pooling of a stream): only the chunk states are
// written; seg_off is then null and the rows are [0, n_fixed).
template <typename T, int MAXC, bool MERGE = true>
__global__ void __launch_bounds__(256) pool_partial_kernel(const T* __restrict__ phi, const int* __restrict__ seg_off,
                                                           const float* __restrict__ w_pool, int d, float inv_sqrt_d,
                                                           int max_chunks, float* __restrict__ part,
                                                           int merge_existing, float* st_m, float* st_s,
                                                           float* st_acc, float* __restrict__ g, int* counter,
                                                           int n_fixed) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = Vec16<T>::N;               // MAXC: 16-byte chunks per lane, ceil(d / (32 VEC))
  __shared__ float sm_m[kPoolWarps], sm_s[kPoolWarps];
  __shared__ float sm_acc[kPoolWarps][512];
  const int r = blockIdx.y, c = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int seg_beg = MERGE ? seg_off[r] : 0, seg_end = MERGE ? seg_off[r + 1] : n_fixed;
  const int beg = seg_beg + c * kPoolChunkV;
  const int nrows = min(seg_end - beg, kPoolChunkV);
  float* out = part + (static_cast<long long>(r) * max_chunks + c) * (d + 2);
  if (nrows <= 0) {
    for (int i = tid; i < d; i += 256) out[2 + i] = 0.f;
    if (tid == 0) {
      out[0] = -INFINITY;
      out[1] = 0.f;
    }
    return;
  }
  constexpr int nch = MAXC;
  float w[MAXC][VEC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int col = (j * 32 + lane) * VEC;
#pragma unroll
    for (int i = 0; i < VEC; ++i) w[j][i] = (j < nch && col + i < d) ? __ldg(w_pool + col + i) : 0.f;
  }
  // this warp's rows: beg + warp + 8 t, loaded RB at a time (all loads of a
  // batch issued before its arithmetic)
  constexpr int RB = MAXC >= 4 ? 2 : (MAXC == 2 ? 4 : kPoolRowsPerWarp);
  float m = -INFINITY, s = 0.f;
  float acc[MAXC][VEC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j)
#pragma unroll
    for (int q = 0; q < VEC; ++q) acc[j][q] = 0.f;
#pragma unroll
  for (int t0 = 0; t0 < kPoolRowsPerWarp; t0 += RB) {
    float v[RB][MAXC][VEC];
#pragma unroll
    for (int t = 0; t < RB; ++t) {
      const int i = warp + kPoolWarps * (t0 + t);
#pragma unroll
      for (int j = 0; j < MAXC; ++j) {
        const int col = (j * 32 + lane) * VEC;
        if (i < nrows && col < d) Vec16<T>::load(phi + static_cast<long long>(beg + i) * d + col, v[t][j]);
        else {
#pragma unroll
          for (int q = 0; q < VEC; ++q) v[t][j][q] = 0.f;
        }
      }
    }
    // the batch's logits first (independent reductions), then one rescale
    float z[RB];
#pragma unroll
    for (int t = 0; t < RB; ++t) {
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < MAXC; ++j)
#pragma unroll
        for (int q = 0; q < VEC; ++q) dot = fmaf(v[t][j][q], w[j][q], dot);
      z[t] = dot;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int t = 0; t < RB; ++t) z[t] += __shfl_xor_sync(0xffffffffu, z[t], o);
    float mb = m;
#pragma unroll
    for (int t = 0; t < RB; ++t) {
      z[t] *= inv_sqrt_d;
      if (warp + kPoolWarps * (t0 + t) < nrows) mb = fmaxf(mb, z[t]);
    }
    const float corr = mb == -INFINITY ? 1.f : expf(m - mb);   // no valid row yet: nothing to rescale
    s *= corr;
#pragma unroll
    for (int j = 0; j < MAXC; ++j)
#pragma unroll
      for (int q = 0; q < VEC; ++q) acc[j][q] *= corr;
#pragma unroll
    for (int t = 0; t < RB; ++t) {
      if (warp + kPoolWarps * (t0 + t) < nrows) {
        const float e = expf(z[t] - mb);
        s += e;
#pragma unroll
        for (int j = 0; j < MAXC; ++j)
#pragma unroll
          for (int q = 0; q < VEC; ++q) acc[j][q] = fmaf(e, v[t][j][q], acc[j][q]);
      }
    }
    m = mb;
  }
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int col = (j * 32 + lane) * VEC;
#pragma unroll
    for (int q = 0; q < VEC; ++q)
      if (j < nch && col + q < d) sm_acc[warp][col + q] = acc[j][q];
  }
  if (lane == 0) {
    sm_m[warp] = m;
    sm_s[warp] = s;
  }
  __syncthreads();
  float M = -INFINITY;
#pragma unroll
  for (int w8 = 0; w8 < kPoolWarps; ++w8) M = fmaxf(M, sm_m[w8]);
  float scale[kPoolWarps];
  float S = 0.f;
#pragma unroll
  for (int w8 = 0; w8 < kPoolWarps; ++w8) {
    scale[w8] = sm_s[w8] > 0.f ? expf(sm_m[w8] - M) : 0.f;
    S += sm_s[w8] * scale[w8];
  }
  // one chunk per request (every request's rows fit one chunk, as in an
  // append of up to kPoolChunkV rows): merge with the stored state right
  // here, with the arithmetic of the general merge below
  const bool single = MERGE && gridDim.x == 1;
  float a_k[2];                                      // this thread's columns tid, tid + 256 (d <= 512)
#pragma unroll
  for (int kk = 0; kk < 2; ++kk) {
    const int k = tid + 256 * kk;
    float a = 0.f;
    if (k < d) {
#pragma unroll
      for (int w8 = 0; w8 < kPoolWarps; ++w8) a = fmaf(sm_acc[w8][k], scale[w8], a);
      if (!single) out[2 + k] = a;
    }
    a_k[kk] = a;
  }
  if (single) {
    const float old_m = merge_existing ? st_m[r] : -INFINITY;
    const float old_s = merge_existing ? st_s[r] : 0.f;
    const float Mr = fmaxf(old_m, M);
    const float w_old = merge_existing ? expf(old_m - Mr) : 0.f;
    const float sc = expf(M - Mr);
    const float Sr = __fadd_rn(__fmul_rn(old_s, w_old), fmaf(S, sc, 0.f));
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const int k = tid + 256 * kk;
      if (k < d) {
        const float a0 = merge_existing ? __fmul_rn(st_acc[static_cast<long long>(r) * d + k], w_old) : 0.f;
        const float a = fmaf(a_k[kk], sc, a0);
        st_acc[static_cast<long long>(r) * d + k] = a;
        g[static_cast<long long>(r) * d + k] = a / Sr;
      }
    }
    __syncthreads();                                 // every thread has read st_m / st_s
    if (tid == 0) {
      st_m[r] = Mr;
      st_s[r] = Sr;
    }
    return;
  }
  if (tid == 0) {
    out[0] = M;
    out[1] = S;
  }
  if constexpr (!MERGE) return;
  pool_merge_if_last(part + static_cast<long long>(r) * max_chunks * (d + 2),
                     (seg_end - seg_beg + kPoolChunkV - 1) / kPoolChunkV, d, r, merge_existing, st_m, st_s, st_acc,
                     g, counter);
}

constexpr int kPoolStages = 4;
constexpr int kPoolStageBytes = 16384;
constexpr int kPoolStreamCtasPerSm = 3;   // 64 KB ring each

// Rebuild pooling of long histories.  One CTA per (chunk of chunk_rows rows,
// request).  A request's rows are contiguous, so a stage of SR = 8 RW rows is
// one untiled bulk copy; thread 0 keeps kPoolStages of them in flight
// through a shared-memory ring (64 KB per CTA in flight, independent of the
// register count), and each warp folds RW rows of every stage into its
// online-softmax state.  The CTA's chunk state goes to part and the last
// CTA of the request merges (pool_merge_if_last).
template <typename T, int MAXC, int RW>
__global__ void __launch_bounds__(256) pool_stream_kernel(const T* __restrict__ phi, const int* __restrict__ seg_off,
                                                          const float* __restrict__ w_pool, int d, float inv_sqrt_d,
                                                          int chunk_rows, int max_chunks, float* __restrict__ part,
                                                          int merge_existing, float* st_m, float* st_s, float* st_acc,
                                                          float* __restrict__ g, int* counter, int* status) {
  constexpr int VEC = Vec16<T>::N;
  constexpr int SR = kPoolWarps * RW;
  extern __shared__ __align__(128) uint8_t pool_ring[];
  __shared__ __align__(8) uint64_t full[kPoolStages];
  __shared__ float sm_m[kPoolWarps], sm_s[kPoolWarps];
  __shared__ int abort_flag;
  const int r = blockIdx.y, c = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
#pragma unroll
    for (int i = 0; i < kPoolStages; ++i) tc::mbar_init(&full[i], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    abort_flag = 0;
  }
  pdl_launch_dependents();
  pdl_wait();
  const int seg_beg = seg_off[r], seg_end = seg_off[r + 1];
  const int beg = seg_beg + c * chunk_rows;
  const int nrows = min(seg_end - beg, chunk_rows);
  if (nrows <= 0) return;                           // past the request's rows (uniform over the CTA)
  const int n_st = (nrows + SR - 1) / SR;
  const uint32_t row_bytes = static_cast<uint32_t>(d) * sizeof(T);
  const T* src0 = phi + static_cast<long long>(beg) * d;
  __syncthreads();                                  // barriers initialised
  if (tid == 0) {
    for (int j = 0; j < min(n_st, kPoolStages); ++j) {
      const uint32_t bytes = static_cast<uint32_t>(min(SR, nrows - j * SR)) * row_bytes;
      tc::mbar_expect_tx(&full[j], bytes);
      tc::bulk_load(pool_ring + j * kPoolStageBytes, src0 + static_cast<long long>(j) * SR * d, bytes, &full[j]);
    }
  }
  float w[MAXC][VEC], acc[MAXC][VEC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int col = (j * 32 + lane) * VEC;
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
      w[j][i] = col + i < d ? __ldg(w_pool + col + i) : 0.f;
      acc[j][i] = 0.f;
    }
  }
  float m = -INFINITY, ssum = 0.f;
  int j = 0;
  for (; j < n_st; ++j) {
    const int slot = j % kPoolStages;
    if (!tc::mbar_wait_plain(&full[slot], (j / kPoolStages) & 1)) abort_flag = 1;
    const T* st = reinterpret_cast<const T*>(pool_ring + slot * kPoolStageBytes);
    const int nr = min(SR, nrows - j * SR);
    float v[RW][MAXC][VEC];
#pragma unroll
    for (int t = 0; t < RW; ++t) {
      const int i = warp + kPoolWarps * t;
#pragma unroll
      for (int q = 0; q < MAXC; ++q) {
        const int col = (q * 32 + lane) * VEC;
        if (i < nr && col < d) Vec16<T>::load(st + i * d + col, v[t][q]);
        else {
#pragma unroll
          for (int e = 0; e < VEC; ++e) v[t][q][e] = 0.f;
        }
      }
    }
    float z[RW];
#pragma unroll
    for (int t = 0; t < RW; ++t) {
      float dot = 0.f;
#pragma unroll
      for (int q = 0; q < MAXC; ++q)
#pragma unroll
        for (int e = 0; e < VEC; ++e) dot = fmaf(v[t][q][e], w[q][e], dot);
      z[t] = dot;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int t = 0; t < RW; ++t) z[t] += __shfl_xor_sync(0xffffffffu, z[t], o);
    float mb = m;
#pragma unroll
    for (int t = 0; t < RW; ++t) {
      z[t] *= inv_sqrt_d;
      if (warp + kPoolWarps * t < nr) mb = fmaxf(mb, z[t]);
    }
    const float corr = mb == -INFINITY ? 1.f : expf(m - mb);
    ssum *= corr;
#pragma unroll
    for (int q = 0; q < MAXC; ++q)
#pragma unroll
      for (int e = 0; e < VEC; ++e) acc[q][e] *= corr;
#pragma unroll
    for (int t = 0; t < RW; ++t) {
      if (warp + kPoolWarps * t < nr) {
        const float e = expf(z[t] - mb);
        ssum += e;
#pragma unroll
        for (int q = 0; q < MAXC; ++q)
#pragma unroll
          for (int u = 0; u < VEC; ++u) acc[q][u] = fmaf(e, v[t][q][u], acc[q][u]);
      }
    }
    m = mb;
    __syncthreads();                                // every warp is done with this slot
    if (abort_flag) break;
    if (tid == 0 && j + kPoolStages < n_st) {
      const int jn = j + kPoolStages;
      const uint32_t bytes = static_cast<uint32_t>(min(SR, nrows - jn * SR)) * row_bytes;
      tc::mbar_expect_tx(&full[slot], bytes);
      tc::bulk_load(pool_ring + slot * kPoolStageBytes, src0 + static_cast<long long>(jn) * SR * d, bytes,
                    &full[slot]);
    }
  }
  if (abort_flag) {
    // let the copies still in flight land (bounded) before the CTA exits
    if (tid == 0) {
      latch_status(status, TXS_ERR_DEVICE_TIMEOUT);
      for (int jj = j; jj < min(n_st, j + kPoolStages); ++jj)
        tc::mbar_wait_plain(&full[jj % kPoolStages], (jj / kPoolStages) & 1);
    }
    return;
  }
  // combine the warps' states; the ring is free now and holds acc[8][512]
  float* sm_acc = reinterpret_cast<float*>(pool_ring);
#pragma unroll
  for (int q = 0; q < MAXC; ++q) {
    const int col = (q * 32 + lane) * VEC;
#pragma unroll
    for (int e = 0; e < VEC; ++e)
      if (col + e < d) sm_acc[warp * 512 + col + e] = acc[q][e];
  }
  if (lane == 0) {
    sm_m[warp] = m;
    sm_s[warp] = ssum;
  }
  __syncthreads();
  float M = -INFINITY;
#pragma unroll
  for (int w8 = 0; w8 < kPoolWarps; ++w8) M = fmaxf(M, sm_m[w8]);
  float scale[kPoolWarps];
  float S = 0.f;
#pragma unroll
  for (int w8 = 0; w8 < kPoolWarps; ++w8) {
    scale[w8] = sm_s[w8] > 0.f ? expf(sm_m[w8] - M) : 0.f;
    S += sm_s[w8] * scale[w8];
  }
  float* out = part + (static_cast<long long>(r) * max_chunks + c) * (d + 2);
  for (int k = tid; k < d; k += 256) {
    float a = 0.f;
#pragma unroll
    for (int w8 = 0; w8 < kPoolWarps; ++w8) a = fmaf(sm_acc[w8 * 512 + k], scale[w8], a);
    out[2 + k] = a;
  }
  if (tid == 0) {
    out[0] = M;
    out[1] = S;
  }
  pool_merge_if_last(part + static_cast<long long>(r) * max_chunks * (d + 2),
                     (seg_end - seg_beg + chunk_rows - 1) / chunk_rows, d, r, merge_existing, st_m, st_s, st_acc, g,
                     counter);
}

constexpr int kAnchorReq = 16;        // anchors staged per CTA (grid.y covers the rest)
constexpr int kAnchorRowsPerWarp = 4;  // weight rows per warp (each staged anchor value read once for all four)

// Anchor projections gkv[blk][r][c] = g_r . Wt[n] + b[n] for the 2 nL dkv
// rows n of the transposed K/V weights (n = blk dkv + c).  One CTA per
// (8 kAnchorRowsPerWarp weight rows, 16 requests): the 16 fp32 anchors are
// staged in shared memory once, each warp reads its weight rows once
// (16-byte vectors) and dots them with all 16 anchors.
template <typename T, int NCH>
__global__ void __launch_bounds__(256) anchor_proj_kernel(const float* __restrict__ g, const T* __restrict__ Wt,
                                                          const float* __restrict__ b, float* __restrict__ gkv,
                                                          int R, int d, int dkv, int n_total) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = Vec16<T>::N;
  extern __shared__ float sg[];                    // [kAnchorReq][d]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r0 = blockIdx.y * kAnchorReq;
  const int nr = min(kAnchorReq, R - r0);
  // all weight loads of this warp's rows, then the anchors (every load issued
  // before the first use)
  float w[kAnchorRowsPerWarp][NCH][VEC];
  const int nw0 = (blockIdx.x * 8 + warp) * kAnchorRowsPerWarp;
#pragma unroll
  for (int k = 0; k < kAnchorRowsPerWarp; ++k)
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const int col = (j * 32 + lane) * VEC;
      if (nw0 + k < n_total && col < d) Vec16<T>::load(Wt + static_cast<long long>(nw0 + k) * d + col, w[k][j]);
      else {
#pragma unroll
        for (int q = 0; q < VEC; ++q) w[k][j][q] = 0.f;
      }
    }
  constexpr int kStage = kAnchorReq * 512 / 4 / 256;   // float4 per thread (d <= 512)
  float4 st[kStage];
  const float4* gsrc = reinterpret_cast<const float4*>(g + static_cast<long long>(r0) * d);
#pragma unroll
  for (int u = 0; u < kStage; ++u) {
    const int i = threadIdx.x + u * 256;
    if (i * 4 < nr * d) st[u] = __ldg(gsrc + i);
  }
#pragma unroll
  for (int u = 0; u < kStage; ++u) {
    const int i = threadIdx.x + u * 256;
    if (i * 4 < nr * d) reinterpret_cast<float4*>(sg)[i] = st[u];
  }
  __syncthreads();
  // dot[k][t] = Wt[nw0 + k] . g[r0 + t]: each anchor value from shared
  // memory serves the warp's kAnchorRowsPerWarp weight rows
  float dot[kAnchorRowsPerWarp][kAnchorReq];
#pragma unroll
  for (int k = 0; k < kAnchorRowsPerWarp; ++k)
#pragma unroll
    for (int t = 0; t < kAnchorReq; ++t) dot[k][t] = 0.f;
#pragma unroll
  for (int t = 0; t < kAnchorReq; ++t) {
    if (t < nr) {
#pragma unroll
      for (int j = 0; j < NCH; ++j) {
        const int col = (j * 32 + lane) * VEC;
        if (col < d) {
          const float4* gp = reinterpret_cast<const float4*>(sg + t * d + col);
#pragma unroll
          for (int q4 = 0; q4 < VEC / 4; ++q4) {
            const float4 x = gp[q4];
#pragma unroll
            for (int k = 0; k < kAnchorRowsPerWarp; ++k) {
              dot[k][t] = fmaf(w[k][j][4 * q4], x.x, dot[k][t]);
              dot[k][t] = fmaf(w[k][j][4 * q4 + 1], x.y, dot[k][t]);
              dot[k][t] = fmaf(w[k][j][4 * q4 + 2], x.z, dot[k][t]);
              dot[k][t] = fmaf(w[k][j][4 * q4 + 3], x.w, dot[k][t]);
            }
          }
        }
      }
    }
  }
#pragma unroll
  for (int k = 0; k < kAnchorRowsPerWarp; ++k) {
    const int n = nw0 + k;
    if (n >= n_total) break;
#pragma unroll
    for (int t = 0; t < kAnchorReq; ++t)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) dot[k][t] += __shfl_xor_sync(0xffffffffu, dot[k][t], o);
    if (lane < nr) {
      float v = 0.f;
#pragma unroll
      for (int t = 0; t < kAnchorReq; ++t)
        if (t == lane) v = dot[k][t];
      const int blk = n / dkv, c = n - blk * dkv;
      gkv[(static_cast<long long>(blk) * R + r0 + lane) * dkv + c] = v + __ldg(b + n);
    }
  }
}

// Wt[c, r] = W[r, c] for W [rows, cols]; Wt has leading dimension rows.
template <typename T>
__global__ void transpose_kernel(const T* __restrict__ W, T* __restrict__ Wt, int rows, int cols) {
  __shared__ T tile[32][33];
  const int bx = blockIdx.x * 32, by = blockIdx.y * 32;
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int r = by + j, c = bx + threadIdx.x;
    if (r < rows && c < cols) tile[j][threadIdx.x] = W[static_cast<long long>(r) * cols + c];
  }
  __syncthreads();
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int c = bx + j, r = by + threadIdx.x;
    if (r < rows && c < cols) Wt[static_cast<long long>(c) * rows + r] = tile[threadIdx.x][j];
  }
}

template <typename T>
__global__ void to_f32_kernel(const T* __restrict__ src, float* __restrict__ dst, long long n) {
  for (long long i = blockIdx.x * 256LL + threadIdx.x; i < n; i += static_cast<long long>(gridDim.x) * 256)
    dst[i] = Elem<T>::load(src + i);
}

// Head fold (weights only): weff[j, a] = W_dec[j] . Q_dec[a] for j < 2d, and
// cdec[a] = b_dec . Q_dec[a], so logits = [z, x] weff + cdec (Sec. 4.1.3 with a
// linear f_dec).
template <typename T>
__global__ void fold_head_kernel(const T* __restrict__ W_dec, const T* __restrict__ b_dec,
                                 const T* __restrict__ Q_dec, float* __restrict__ weff, float* __restrict__ cdec,
                                 int d, int k) {
  const int t = blockIdx.x * 256 + threadIdx.x;
  if (t >= (2 * d + 1) * k) return;
  const int j = t / k, a = t - j * k;
  const T* w = j < 2 * d ? W_dec + static_cast<long long>(j) * d : b_dec;
  const T* q = Q_dec + static_cast<long long>(a) * d;
  float s = 0.f;
  for (int c = 0; c < d; ++c) s = fmaf(Elem<T>::load(w + c), Elem<T>::load(q + c), s);
  if (j < 2 * d) weff[static_cast<long long>(j) * k + a] = s;
  else cdec[a] = s;
}

// Deep & Wide head fold (weights only; App. B f_dec = [x_wide W_w + b_w,
// FFN([z, x_deep])] with the FFN's last layer W_d2, b_d2).  With Q_w, Q_d the
// columns of Q_dec against the wide and deep parts of k_dec:
//   weff_x[j, a] = W_w[j] . Q_w[a] for j < dw_in, 0 for the deep features;
//   cdec[a]      = b_w . Q_w[a] + b_d2 . Q_d[a];
//   w2q[f, a]    = W_d2[f] . Q_d[a],
// so logits = x weff_x + cdec + GELU([z, x_deep] W_d1 + b_d1) w2q.
template <typename T>
__global__ void fold_dw_kernel(const T* __restrict__ W_w, const T* __restrict__ b_w, const T* __restrict__ W_d2,
                               const T* __restrict__ b_d2, const T* __restrict__ Q_dec, float* __restrict__ weff_x,
                               float* __restrict__ cdec, float* __restrict__ w2q, int d, int dw_in, int dw_out,
                               int Fh, int k) {
  const int t = blockIdx.x * 256 + threadIdx.x;
  if (t >= (d + 1 + Fh) * k) return;
  const int j = t / k, a = t - j * k;
  const T* q = Q_dec + static_cast<long long>(a) * d;
  const int dd = d - dw_out;
  float s = 0.f;
  if (j < d) {
    if (j < dw_in)
      for (int c = 0; c < dw_out; ++c)
        s = fmaf(Elem<T>::load(W_w + static_cast<long long>(j) * dw_out + c), Elem<T>::load(q + c), s);
    weff_x[static_cast<long long>(j) * k + a] = s;
  } else if (j == d) {
    for (int c = 0; c < dw_out; ++c) s = fmaf(Elem<T>::load(b_w + c), Elem<T>::load(q + c), s);
    for (int c = 0; c < dd; ++c) s = fmaf(Elem<T>::load(b_d2 + c), Elem<T>::load(q + dw_out + c), s);
    cdec[a] = s;
  } else {
    const int f = j - d - 1;
    for (int c = 0; c < dd; ++c)
      s = fmaf(Elem<T>::load(W_d2 + static_cast<long long>(f) * dd + c), Elem<T>::load(q + dw_out + c), s);
    w2q[static_cast<long long>(f) * k + a] = s;
  }
}

// Order-independent 64-bit content hash: sum over 32-bit words of a
// splitmix64-style finaliser of (word, index, salt).
__global__ void hash_kernel(const uint32_t* __restrict__ p, long long n_words, uint64_t salt,
                            unsigned long long* out) {
  uint64_t acc = 0;
  for (long long i = blockIdx.x * 256LL + threadIdx.x; i < n_words; i += static_cast<long long>(gridDim.x) * 256) {
    uint64_t z = (static_cast<uint64_t>(p[i]) << 32 ^ static_cast<uint64_t>(i)) + salt * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    acc += z ^ (z >> 31);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) atomicAdd(out, static_cast<unsigned long long>(acc));
}

}  // namespace

template <typename T, int MAXC, int RW>
cudaError_t launch_pool_stream(const T* phi, const int* seg_off, int R, int chunks, int chunk_rows, const float* w_pool,
                               int d, float isd, int max_chunks, float* part, int merge_existing, float* st_m,
                               float* st_s, float* st_acc, float* g, int* counter, int* status, cudaStream_t s) {
  constexpr int kSmem = kPoolStages * kPoolStageBytes;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(pool_stream_kernel<T, MAXC, RW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  return launch_pdl(pool_stream_kernel<T, MAXC, RW>, dim3(chunks, R), dim3(256), kSmem, s, phi, seg_off, w_pool, d,
                    isd, chunk_rows, max_chunks, part, merge_existing, st_m, st_s, st_acc, g, counter, status);
}

template <typename T, int RW>
cudaError_t launch_pool_stream_c(int nch, const T* phi, const int* seg_off, int R, int chunks, int chunk_rows,
                                 const float* w_pool, int d, float isd, int max_chunks, float* part, int merge_existing,
                                 float* st_m, float* st_s, float* st_acc, float* g, int* counter, int* status,
                                 cudaStream_t s) {
  if (nch == 1)
    return launch_pool_stream<T, 1, RW>(phi, seg_off, R, chunks, chunk_rows, w_pool, d, isd, max_chunks, part,
                                        merge_existing, st_m, st_s, st_acc, g, counter, status, s);
  if (nch == 2)
    return launch_pool_stream<T, 2, RW>(phi, seg_off, R, chunks, chunk_rows, w_pool, d, isd, max_chunks, part,
                                        merge_existing, st_m, st_s, st_acc, g, counter, status, s);
  return launch_pool_stream<T, 4, RW>(phi, seg_off, R, chunks, chunk_rows, w_pool, d, isd, max_chunks, part,
                                      merge_existing, st_m, st_s, st_acc, g, counter, status, s);
}

// Chunks of more than kPoolChunkV rows go through the streaming kernel (rows
// 16-byte aligned); an append of at most kPoolChunkV rows per request keeps
// the one-chunk kernel, which merges in the CTA.
template <typename T>
cudaError_t launch_pool(const T* phi, const int* seg_off, int R, int max_rows, const float* w_pool, int d,
                        int max_chunks, float* part, int merge_existing, float* st_m, float* st_s, float* st_acc,
                        float* g, int* counter, int* status, cudaStream_t s) {
  const int chunks = (max_rows + kPoolChunkV - 1) / kPoolChunkV;
  if (chunks > max_chunks) return cudaErrorInvalidValue;
  if (chunks == 0) return cudaSuccess;   // no new rows: the stored state and g stay as they are
  constexpr int VEC = Vec16<T>::N;
  const int nch = (d + 32 * VEC - 1) / (32 * VEC);
  if (nch > 4 || d > 512) return cudaErrorInvalidValue;
  const float isd = 1.0f / sqrtf(static_cast<float>(d));
  const int row_bytes = d * static_cast<int>(sizeof(T));
  const bool stream = max_rows > kPoolChunkV && row_bytes % 16 == 0 && reinterpret_cast<uintptr_t>(phi) % 16 == 0;
  cudaError_t err0 = cudaSuccess;
  prof_begin(KC_POOL, s);
  if (stream) {
    // the longest chunk that still gives every SM its resident CTAs twice over
    int chunk_rows = 256;
    while (chunk_rows > kPoolChunkV &&
           static_cast<long long>(R) * ((max_rows + chunk_rows - 1) / chunk_rows) <
               2LL * kPoolStreamCtasPerSm * tc::num_sms())
      chunk_rows /= 2;
    const int n_chunks = (max_rows + chunk_rows - 1) / chunk_rows;
    const int rw = kPoolStageBytes / (kPoolWarps * row_bytes);   // rows per warp and stage
    if (rw >= 4)
      err0 = launch_pool_stream_c<T, 4>(nch, phi, seg_off, R, n_chunks, chunk_rows, w_pool, d, isd, max_chunks, part,
                                        merge_existing, st_m, st_s, st_acc, g, counter, status, s);
    else if (rw >= 2)
      err0 = launch_pool_stream_c<T, 2>(nch, phi, seg_off, R, n_chunks, chunk_rows, w_pool, d, isd, max_chunks, part,
                                        merge_existing, st_m, st_s, st_acc, g, counter, status, s);
    else
      err0 = launch_pool_stream_c<T, 1>(nch, phi, seg_off, R, n_chunks, chunk_rows, w_pool, d, isd, max_chunks, part,
                                        merge_existing, st_m, st_s, st_acc, g, counter, status, s);
  } else {
    const dim3 grid(chunks, R);
    if (nch == 1)
      err0 = launch_pdl(pool_partial_kernel<T, 1>, grid, dim3(256), 0, s, phi, seg_off, w_pool, d, isd, max_chunks,
                        part, merge_existing, st_m, st_s, st_acc, g, counter, 0);
    else if (nch == 2)
      err0 = launch_pdl(pool_partial_kernel<T, 2>, grid, dim3(256), 0, s, phi, seg_off, w_pool, d, isd, max_chunks,
                        part, merge_existing, st_m, st_s, st_acc, g, counter, 0);
    else
      err0 = launch_pdl(pool_partial_kernel<T, 4>, grid, dim3(256), 0, s, phi, seg_off, w_pool, d, isd, max_chunks,
                        part, merge_existing, st_m, st_s, st_acc, g, counter, 0);
  }
  cudaError_t err = err0 != cudaSuccess ? err0 : cudaGetLastError();
  prof_end(KC_POOL, s);
  return err;
}

template <typename T>
cudaError_t launch_anchor_proj(const float* g, const T* Wt_kv, const float* b_kv, float* gkv, int R, int d, int dkv,
                               int n_layers, cudaStream_t s) {
  constexpr int VEC = Vec16<T>::N;
  const int nch = (d + 32 * VEC - 1) / (32 * VEC);
  if (R <= 0) return cudaSuccess;
  if (d % 4 || d > 512) return cudaErrorInvalidValue;
  const int n_total = 2 * n_layers * dkv;
  const dim3 grid((n_total + 8 * kAnchorRowsPerWarp - 1) / (8 * kAnchorRowsPerWarp),
                  (R + kAnchorReq - 1) / kAnchorReq);
  const size_t smem = sizeof(float) * kAnchorReq * d;   // <= 32 KB for d <= 512
  prof_begin(KC_GLOBAL_KV, s);
  cudaError_t err;
  if (nch == 1) err = launch_pdl(anchor_proj_kernel<T, 1>, grid, dim3(256), smem, s, g, Wt_kv, b_kv, gkv, R, d, dkv, n_total);
  else if (nch == 2) err = launch_pdl(anchor_proj_kernel<T, 2>, grid, dim3(256), smem, s, g, Wt_kv, b_kv, gkv, R, d, dkv, n_total);
  else if (nch <= 4) err = launch_pdl(anchor_proj_kernel<T, 4>, grid, dim3(256), smem, s, g, Wt_kv, b_kv, gkv, R, d, dkv, n_total);
  else return cudaErrorInvalidValue;
  prof_end(KC_GLOBAL_KV, s);
  return err;
}

template <typename T>
cudaError_t launch_transpose(const T* W, T* Wt, int rows, int cols, cudaStream_t s) {
  dim3 grid((cols + 31) / 32, (rows + 31) / 32);
  transpose_kernel<T><<<grid, dim3(32, 8), 0, s>>>(W, Wt, rows, cols);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_to_f32(const T* src, float* dst, long long n, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const long long blocks = (n + 255) / 256;
  to_f32_kernel<T><<<static_cast<int>(blocks < 4096 ? blocks : 4096), 256, 0, s>>>(src, dst, n);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_fold_head(const T* W_dec, const T* b_dec, const T* Q_dec, float* weff, float* cdec, int d, int k,
                             cudaStream_t s) {
  const int n = (2 * d + 1) * k;
  fold_head_kernel<T><<<(n + 255) / 256, 256, 0, s>>>(W_dec, b_dec, Q_dec, weff, cdec, d, k);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_fold_dw(const T* W_w, const T* b_w, const T* W_d2, const T* b_d2, const T* Q_dec, float* weff_x,
                           float* cdec, float* w2q, int d, int dw_in, int dw_out, int Fh, int k, cudaStream_t s) {
  const int n = (d + 1 + Fh) * k;
  fold_dw_kernel<T><<<(n + 255) / 256, 256, 0, s>>>(W_w, b_w, W_d2, b_d2, Q_dec, weff_x, cdec, w2q, d, dw_in, dw_out,
                                                     Fh, k);
  return cudaGetLastError();
}

cudaError_t launch_hash(const void* p, long long bytes, uint64_t salt, unsigned long long* out, cudaStream_t s) {
  const long long words = bytes / 4;
  if (words == 0) return cudaSuccess;
  const long long blocks = (words + 255) / 256;
  hash_kernel<<<static_cast<int>(blocks < 1024 ? blocks : 1024), 256, 0, s>>>(static_cast<const uint32_t*>(p), words,
                                                                              salt, out);
  return cudaGetLastError();
}

// Self-test of the bounded waits every pipeline of this library uses: one
// thread waits (tc::mbar_wait, kSpinCycles) on an mbarrier nothing arrives
// at; when the wait gives up the kernel latches TXS_ERR_DEVICE_TIMEOUT into
// the status word and returns, leaving the context usable.
__global__ void wait_timeout_probe_kernel(int* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    abort_flag = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0 && !tc::mbar_wait(&bar, 0, &abort_flag)) latch_status(status, TXS_ERR_DEVICE_TIMEOUT);
}

cudaError_t launch_wait_timeout_probe(int* status, cudaStream_t s) {
  wait_timeout_probe_kernel<<<1, 32, 0, s>>>(status);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ prefix pooling

// Streaming events (Sec. 4.2 prefix reuse; Sec. 5.1 a global token for each
// event timestamp): event t's anchor is the attention pooling of the first
// ends[t] behavior rows of the user.  The stream is pooled once in chunks of
// kPoolChunkV rows (pool_partial_kernel, no merge); then one CTA per event
// merges the states of the chunks wholly inside its prefix with the rows of
// the last, partial chunk (online-softmax merge: every term rescaled to the
// common maximum).  The CTA also writes the event's cache view: first row
// off_user, length ends[t].
constexpr int kEvMax = 4096;

struct PrefixPoolArgs {
  int n_ev;
  int off_user;
  int ends[kEvMax];
};

template <typename T, int MAXC>
__global__ void __launch_bounds__(256) prefix_finish_kernel(const T* __restrict__ phi,
                                                            const float* __restrict__ w_pool, int d,
                                                            float inv_sqrt_d, const float* __restrict__ part,
                                                            float* __restrict__ g, int* __restrict__ ev_off,
                                                            int* __restrict__ ev_len,
                                                            const __grid_constant__ PrefixPoolArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = Vec16<T>::N;
  constexpr int W = 8;
  __shared__ float sm_m[W], sm_s[W];
  extern __shared__ float sm_acc[];                      // [W][d]
  const int t = blockIdx.x;
  const int end = a.ends[t];
  const int nfull = end / kPoolChunkV;                   // chunks wholly inside the prefix
  const int beg = nfull * kPoolChunkV;                   // rows [beg, end) pooled here
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    ev_off[t] = a.off_user;
    ev_len[t] = end;
  }
  const int nch = (d + 32 * VEC - 1) / (32 * VEC);      // 16-byte vectors per lane
  float w[MAXC][VEC], acc[MAXC][VEC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j)
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
      const int col = (j * 32 + lane) * VEC + i;
      w[j][i] = (j < nch && col < d) ? __ldg(w_pool + col) : 0.f;
      acc[j][i] = 0.f;
    }
  float m = -INFINITY, ssum = 0.f;
  for (int row = beg + warp; row < end; row += W) {
    const T* pr = phi + static_cast<long long>(row) * d;
    float x[MAXC][VEC];
    float dot = 0.f;
#pragma unroll
    for (int j = 0; j < MAXC; ++j) {
      const int col = (j * 32 + lane) * VEC;
      if (j < nch && col < d) {
        Vec16<T>::load(pr + col, x[j]);
      } else {
#pragma unroll
        for (int i = 0; i < VEC; ++i) x[j][i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < VEC; ++i) dot = fmaf(x[j][i], w[j][i], dot);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    const float lg = dot * inv_sqrt_d;
    const float mn = fmaxf(m, lg);
    const float corr = expf(m - mn);                     // 0 on the first row
    const float p = expf(lg - mn);
    ssum = ssum * corr + p;
#pragma unroll
    for (int j = 0; j < MAXC; ++j)
#pragma unroll
      for (int i = 0; i < VEC; ++i) acc[j][i] = fmaf(acc[j][i], corr, p * x[j][i]);
    m = mn;
  }
  if (lane == 0) {
    sm_m[warp] = m;
    sm_s[warp] = ssum;
  }
#pragma unroll
  for (int j = 0; j < MAXC; ++j)
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
      const int col = (j * 32 + lane) * VEC + i;
      if (j < nch && col < d) sm_acc[warp * d + col] = acc[j][i];
    }
  __syncthreads();
  // common maximum over the full chunks and the warps' partial states
  float M = -INFINITY;
  for (int c = 0; c < nfull; ++c) M = fmaxf(M, __ldg(part + static_cast<long long>(c) * (d + 2)));
#pragma unroll
  for (int k = 0; k < W; ++k) M = fmaxf(M, sm_m[k]);
  float S = 0.f;
  for (int c = 0; c < nfull; ++c) {
    const float* pc = part + static_cast<long long>(c) * (d + 2);
    S = fmaf(__ldg(pc + 1), expf(__ldg(pc) - M), S);
  }
  float scale[W];
#pragma unroll
  for (int k = 0; k < W; ++k) {
    scale[k] = sm_s[k] > 0.f ? expf(sm_m[k] - M) : 0.f;  // a warp with no rows contributes nothing
    S = fmaf(sm_s[k], scale[k], S);
  }
  const float inv = 1.f / S;
  for (int col = threadIdx.x; col < d; col += blockDim.x) {
    float v = 0.f;
#pragma unroll
    for (int k = 0; k < W; ++k) v = fmaf(sm_acc[k * d + col], scale[k], v);
    for (int c = 0; c < nfull; ++c) {
      const float* pc = part + static_cast<long long>(c) * (d + 2);
      v = fmaf(__ldg(pc + 2 + col), expf(__ldg(pc) - M), v);
    }
    g[static_cast<long long>(t) * d + col] = v * inv;
  }
}

size_t prefix_pool_scratch_floats(int max_end, int d) {
  return static_cast<size_t>((max_end + kPoolChunkV - 1) / kPoolChunkV) * (d + 2);
}

template <typename T>
cudaError_t launch_prefix_pool(const T* phi, const int* ends, int n_ev, int off_user, const float* w_pool, int d,
                               float* part, float* g, int* ev_off, int* ev_len, cudaStream_t s) {
  if (n_ev <= 0) return cudaSuccess;
  if (n_ev > kEvMax) return cudaErrorInvalidValue;
  PrefixPoolArgs a;
  a.n_ev = n_ev;
  a.off_user = off_user;
  int max_end = 0;
  for (int t = 0; t < n_ev; ++t) {
    a.ends[t] = ends[t];
    max_end = std::max(max_end, ends[t]);
  }
  constexpr int VEC = Vec16<T>::N;
  const int nch = (d + 32 * VEC - 1) / (32 * VEC);
  if (nch > 4 || d > 512) return cudaErrorInvalidValue;
  const float isd = 1.0f / sqrtf(static_cast<float>(d));
  const size_t smem = static_cast<size_t>(8) * d * sizeof(float);
  const int n_chunks = max_end / kPoolChunkV;           // only whole chunks are pooled ahead
  prof_begin(KC_POOL, s);
  cudaError_t err = cudaSuccess;
  if (n_chunks > 0) {
    const dim3 grid(n_chunks, 1);
    if (nch <= 1)
      err = launch_pdl(pool_partial_kernel<T, 1, false>, grid, dim3(256), 0, s, phi, nullptr, w_pool, d, isd, n_chunks,
                       part, 0, nullptr, nullptr, nullptr, nullptr, nullptr, max_end);
    else if (nch <= 2)
      err = launch_pdl(pool_partial_kernel<T, 2, false>, grid, dim3(256), 0, s, phi, nullptr, w_pool, d, isd, n_chunks,
                       part, 0, nullptr, nullptr, nullptr, nullptr, nullptr, max_end);
    else
      err = launch_pdl(pool_partial_kernel<T, 4, false>, grid, dim3(256), 0, s, phi, nullptr, w_pool, d, isd, n_chunks,
                       part, 0, nullptr, nullptr, nullptr, nullptr, nullptr, max_end);
  }
  if (err == cudaSuccess) {
    if (nch <= 1)
      err = launch_pdl(prefix_finish_kernel<T, 1>, dim3(n_ev), dim3(256), smem, s, phi, w_pool, d, isd, part, g,
                       ev_off, ev_len, a);
    else if (nch <= 2)
      err = launch_pdl(prefix_finish_kernel<T, 2>, dim3(n_ev), dim3(256), smem, s, phi, w_pool, d, isd, part, g,
                       ev_off, ev_len, a);
    else
      err = launch_pdl(prefix_finish_kernel<T, 4>, dim3(n_ev), dim3(256), smem, s, phi, w_pool, d, isd, part, g,
                       ev_off, ev_len, a);
  }
  prof_end(KC_POOL, s);
  return err;
}

#define TXS_INST(T)                                                                                                 \
  template cudaError_t launch_pool<T>(const T*, const int*, int, int, const float*, int, int, float*, int, float*, \
                                      float*, float*, float*, int*, int*, cudaStream_t);                            \
  template cudaError_t launch_prefix_pool<T>(const T*, const int*, int, int, const float*, int, float*, float*,     \
                                             int*, int*, cudaStream_t);                                             \
  template cudaError_t launch_anchor_proj<T>(const float*, const T*, const float*, float*, int, int, int, int,     \
                                             cudaStream_t);                                                         \
  template cudaError_t launch_transpose<T>(const T*, T*, int, int, cudaStream_t);                                  \
  template cudaError_t launch_to_f32<T>(const T*, float*, long long, cudaStream_t);                                \
  template cudaError_t launch_fold_head<T>(const T*, const T*, const T*, float*, float*, int, int, cudaStream_t); \
  template cudaError_t launch_fold_dw<T>(const T*, const T*, const T*, const T*, const T*, float*, float*, float*,   \
                                         int, int, int, int, int, cudaStream_t);
TXS_INST(float)
TXS_INST(__nv_bfloat16)
#undef TXS_INST

}  // namespace txs
