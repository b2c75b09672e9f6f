// Tensor-core GEMM for sm_103a with fused epilogues: C = A B^T (+ epilogue).
//
// A [M, K] bf16 row-major (activations or behavior rows), B [N, K] bf16
// row-major (a transposed weight, K-major), fp32 accumulation in TMEM.
// Used by every dense projection of the path: the cache build K/V projection
// (Sec. 4.1.2, K = Phi_b W_K, V = Phi_b W_V), the serving-attention QKV, the
// cross-attention query, the output projections with residual + LayerNorm
// (Sec. 4.1.2 crossAttend equation) and the FFN with GELU.
//
// Persistent kernel, one CTA per SM, 128 x BN output tiles: warp 0 streams A/B
// tiles with TMA into a STAGES-deep ring of 128-byte-swizzled shared-memory
// buffers, warp 1 issues tcgen05.mma (M=128, N<=256 per instruction, K=16)
// into one of two TMEM accumulators, warps 2-9 read the accumulator back with
// tcgen05.ld (one row per thread, two warps per row block, each half of the
// columns) and run the epilogue while the next tile accumulates into the other
// buffer.  All waits are bounded; a timeout latches TXS_ERR_DEVICE_TIMEOUT.
#include <cstdio>

#include <type_traits>

#include "tc_ptx.cuh"

namespace txs {
namespace tc {

// ------------------------------------------------------------------ epilogues


// Same, from a generic pointer (shared or global memory).
__device__ __forceinline__ void load_f32x32_gen(const float* p, float* b) {
  const float4* q = reinterpret_cast<const float4*>(p);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    float4 t = q[j];
    b[4 * j] = t.x; b[4 * j + 1] = t.y; b[4 * j + 2] = t.z; b[4 * j + 3] = t.w;
  }
}

// largest r with off[r] <= row, off[0..n] non-decreasing (generic pointer)
__device__ __forceinline__ int find_seg_gen(const int* off, int n, int row) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= row) lo = mid; else hi = mid - 1;
  }
  return lo;
}

constexpr int kStageN = 4096;     // bias entries staged in shared memory
constexpr int kStageNRes = 1024;  // the same with a resident B slice (less room)
constexpr int kStageSeg = 1024;   // request offsets staged in shared memory (cache-row remap)




constexpr int kEpiWarps = 8;                  // two warps per TMEM lane quarter
constexpr int NUM_THREADS = 64 + 32 * kEpiWarps;
constexpr int kRedStride = 17;                // per-row exchange slots: sum + 16 logits

// Epilogue of one 128 x BN tile for one warp: TMEM lanes `tlane` (32 rows of
// the tile), columns [c0, c0 + BN/2) of the accumulator.  The two warps that
// share a lane quarter exchange row sums (and head logits) through `red`.
template <int BN, int EPI, int NAP>
__device__ __forceinline__ void epilogue(const EpiArgs& e, uint32_t tacc, int row, int n0, int c0, int q, int h,
                                         float* red, const float* s_weff, const float* bias,
                                         const int* seg_off, const int* dst_row0, const CUtensorMap* tmO,
                                         uint8_t* stage, int& kchunk) {
  constexpr int HALF = BN / 2;
  const bool valid = row < e.M;
  const int lane = threadIdx.x & 31;
  float v[32];
  if constexpr (EPI == EPI_BIAS || EPI == EPI_BIAS_GELU || EPI == EPI_KV) {
    // bulk-store coordinates of this warp's 32 rows: plain outputs are a
    // [M, N] tensor (rows past M are dropped by the store); the cache is a
    // [blocks * cap_total, col_blk] tensor (column blocks of width col_blk,
    // at least 32, may be narrower than the tile) and takes the bulk path
    // only when all 32 rows are valid and belong to one request (consecutive
    // cache rows)
    bool tma_ok = true;
    long long orow = row;
    long long orow0 = row - lane;                // the warp's first row
    if constexpr (EPI == EPI_KV) {
      int r = 0;
      if (valid) {
        r = find_seg_gen(seg_off, e.n_seg, row);
        orow = static_cast<long long>(dst_row0[r]) + (row - seg_off[r]);
      }
      // lane 0 holds the warp's first row: if it is invalid, so are all
      const int r_first = __shfl_sync(0xffffffffu, r, 0);
      orow0 = __shfl_sync(0xffffffffu, orow, 0);
      tma_ok = valid && r == r_first;
    }
    tma_ok = __all_sync(0xffffffffu, tma_ok);
    // stores the 32 columns starting at output column n of this warp's rows
    auto put = [&](const float* vals, int n) {
      __nv_bfloat16* out = nullptr;
      int tx = n, ty = static_cast<int>(orow0);
      if constexpr (EPI == EPI_KV) {
        const int blk = n / e.col_blk, xin = n - blk * e.col_blk;
        if (valid) out = static_cast<__nv_bfloat16*>(e.out) + orow * e.ldo + blk * e.col_blk_stride + xin;
        tx = xin;
        ty = static_cast<int>(static_cast<long long>(blk) * (e.col_blk_stride / e.col_blk) + orow0);
      } else {
        if (valid) out = static_cast<__nv_bfloat16*>(e.out) + orow * e.ldo + n;
      }
      store_chunk(vals, out, valid, tma_ok, tmO, tx, ty, stage, kchunk++, lane);
    };
    if constexpr (HALF % 64 == 0) {
      // 64 columns per TMEM load (one wait), two bulk-stored chunks
#pragma unroll 1
      for (int c = 0; c < HALF; c += 64) {
        float w[64];
        tmem_ld64(tacc + c0 + c, w);
#pragma unroll
        for (int hh = 0; hh < 64; hh += 32) {
          float b[32];
          load_f32x32_gen(bias + n0 + c0 + c + hh, b);
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            float2 x = fadd2(make_float2(w[hh + i], w[hh + i + 1]), make_float2(b[i], b[i + 1]));
            if constexpr (EPI == EPI_BIAS_GELU) x = gelu_erf_as2(x);
            w[hh + i] = x.x;
            w[hh + i + 1] = x.y;
          }
          put(w + hh, n0 + c0 + c + hh);
        }
      }
    } else {
#pragma unroll 1
      for (int c = 0; c < HALF; c += 32) {
        tmem_ld32(tacc + c0 + c, v);
        float b[32];
        load_f32x32_gen(bias + n0 + c0 + c, b);
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          float2 x = fadd2(make_float2(v[i], v[i + 1]), make_float2(b[i], b[i + 1]));
          if constexpr (EPI == EPI_BIAS_GELU) x = gelu_erf_as2(x);
          v[i] = x.x;
          v[i + 1] = x.y;
        }
        put(v, n0 + c0 + c);
      }
    }
  } else {
    // Row LayerNorm over the full row (BN == N): two passes over TMEM, the
    // pre-norm values written back in place; halves combined through `red`.
    const int trow = q * 32 + lane;              // row within the tile
    float* my = red + (h * 128 + trow) * kRedStride;
    const float* other = red + ((1 - h) * 128 + trow) * kRedStride;
    const __nv_bfloat16* res = valid ? static_cast<const __nv_bfloat16*>(e.res) + row * e.ldr : nullptr;
    float sum = 0.f;
#pragma unroll 1
    for (int c = 0; c < HALF; c += 32) {
      tmem_ld32(tacc + c0 + c, v);
      float b[32], r[32];
      load_f32x32(e.bias + c0 + c, b);
      if (valid) load_bf16x32(res + c0 + c, r);
      else {
#pragma unroll
        for (int i = 0; i < 32; ++i) r[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        v[i] += b[i] + r[i];
        sum += v[i];
      }
      tmem_st32(tacc + c0 + c, v);
    }
    my[0] = sum;
    named_bar(1 + q, 64);
    const float mean = (sum + other[0]) / static_cast<float>(BN);
    named_bar(1 + q, 64);                        // both read before the slot is reused
    float sq = 0.f;
#pragma unroll 1
    for (int c = 0; c < HALF; c += 32) {
      tmem_ld32(tacc + c0 + c, v);
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float t = v[i] - mean;
        sq += t * t;
      }
    }
    my[0] = sq;
    named_bar(1 + q, 64);
    const float rstd = rsqrtf((sq + other[0]) / static_cast<float>(BN) + e.ln_eps);
    float lg[NAP];
#pragma unroll
    for (int a = 0; a < NAP; ++a) lg[a] = 0.f;
    __nv_bfloat16* out = nullptr;
    if constexpr (EPI == EPI_LN) {
      if (valid) out = static_cast<__nv_bfloat16*>(e.out) + row * e.ldo + c0;
    }
    const int ty = row - lane;
#pragma unroll 1
    for (int c = 0; c < HALF; c += 32) {
      tmem_ld32(tacc + c0 + c, v);
      float g[32], bt[32];
      load_f32x32(e.gamma + c0 + c, g);
      load_f32x32(e.beta + c0 + c, bt);
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = (v[i] - mean) * rstd * g[i] + bt[i];
      if constexpr (EPI == EPI_LN) {
        store_chunk(v, out + c, valid, true, tmO, c0 + c, ty, stage, kchunk++, lane);
      } else {
        // head: z . W_eff_z, weights zero-padded to NAP actions in shared memory
        const float4* w4 = reinterpret_cast<const float4*>(s_weff + (c0 + c) * NAP);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
#pragma unroll
          for (int a4 = 0; a4 < NAP / 4; ++a4) {
            const float4 w = w4[i * (NAP / 4) + a4];
            lg[4 * a4] = fmaf(v[i], w.x, lg[4 * a4]);
            lg[4 * a4 + 1] = fmaf(v[i], w.y, lg[4 * a4 + 1]);
            lg[4 * a4 + 2] = fmaf(v[i], w.z, lg[4 * a4 + 2]);
            lg[4 * a4 + 3] = fmaf(v[i], w.w, lg[4 * a4 + 3]);
          }
        }
      }
    }
    if constexpr (EPI == EPI_LN_HEAD) {
      const int na = e.n_act;
      named_bar(1 + q, 64);                      // partner has read `sq`
#pragma unroll
      for (int a = 0; a < NAP; ++a) my[1 + a] = lg[a];
      named_bar(1 + q, 64);
      if (h == 0 && valid && row < e.n_cand_rows) {
        float mx = -INFINITY;
#pragma unroll
        for (int a = 0; a < NAP; ++a)
          if (a < na) {
            lg[a] += other[1 + a] + __ldg(e.xlog + static_cast<long long>(row) * na + a);
            mx = fmaxf(mx, lg[a]);
          }
        float s = 0.f, p[NAP];
#pragma unroll
        for (int a = 0; a < NAP; ++a) {
          p[a] = a < na ? expf(lg[a] - mx) : 0.f;
          s += p[a];
        }
        const float inv = 1.f / s;
#pragma unroll
        for (int a = 0; a < NAP; ++a)
          if (a < na) {
            e.logits[static_cast<long long>(row) * na + a] = lg[a];
            if (e.probs) e.probs[static_cast<long long>(row) * na + a] = p[a] * inv;
          }
      }
    }
    named_bar(1 + q, 64);                        // `red` free for the next tile
  }
}

// ------------------------------------------------------------------ kernel

// BRES: the CTA's whole B slice (BN x K, K <= KRES) stays resident in shared
// memory and only A streams through the ring.
template <int BN, int EPI, int NAP = 4, bool BRES = false>
struct Shape {
  static constexpr int BN_MMA = BN < 256 ? BN : 256;     // N of one tcgen05.mma
  static constexpr int B_BOX = BN_MMA;                    // rows of one TMA box of B
  static constexpr int KRES = 256;
  static constexpr int BRES_BYTES = BRES ? BN * KRES * 2 : 0;
  static constexpr int B_STAGE_BYTES = BRES ? 0 : BN * BK * 2;
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr bool LN = EPI == EPI_LN || EPI == EPI_LN_HEAD;
  static constexpr int RED_BYTES = LN ? 2 * 128 * kRedStride * 4 : 0;
  static constexpr int WEFF_BYTES = EPI == EPI_LN_HEAD ? BN * NAP * 4 : 0;
  // bias [kStageN] floats ([kStageNRes] with BRES), then (cache-row remap) offsets and
  // first rows; rounded to 1 KB so that the staging buffers after it start on
  // a swizzle-atom boundary
  static constexpr int AUX_BYTES =
      LN ? 0
         : (((BRES ? kStageNRes * 4 : kStageN * 4) + (EPI == EPI_KV ? (2 * kStageSeg + 1) * 4 : 0) + 1023) / 1024) * 1024;
  // bulk-store staging: two 2 KB buffers per epilogue warp (bf16 outputs)
  static constexpr int STG_BYTES = EPI == EPI_LN_HEAD ? 0 : kEpiWarps * 2 * 2048;
  static constexpr int EXTRA = BRES_BYTES + RED_BYTES + WEFF_BYTES + AUX_BYTES + STG_BYTES + 1024 + 256;
  static constexpr int STAGES_FIT = (227 * 1024 - EXTRA) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
  static constexpr int ACC_BUFS = BN <= 256 ? 2 : 1;      // TMEM double buffer
  static constexpr int TMEM_COLS = BN * ACC_BUFS < 32 ? 32 : BN * ACC_BUFS;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EXTRA;
  static_assert(STAGES >= 2, "pipeline depth");
  static_assert(!(BRES && LN), "resident B only for the plain epilogues");
  static_assert((RED_BYTES + WEFF_BYTES + AUX_BYTES) % 1024 == 0 || STG_BYTES == 0,
                "staging buffers need 512-byte alignment (64-byte swizzle atoms)");
  static_assert((RED_BYTES + WEFF_BYTES + AUX_BYTES + STG_BYTES) % 16 == 0, "mbarriers must stay 8-byte aligned");
  static_assert(SMEM_BYTES <= 232448, "shared memory");
  static_assert((TMEM_COLS & (TMEM_COLS - 1)) == 0 && TMEM_COLS <= 512, "TMEM columns");
};

// Persistent: CTA b processes tiles b, b + gridDim.x, ... (tile t -> n tile
// t % n_tiles, m tile t / n_tiles).  With BRES, CTA b instead takes the
// contiguous range [b T / G, (b + 1) T / G) of the T tiles in n-major order
// (tile t -> n tile t / m_tiles, m tile t % m_tiles), so it loads one B slice,
// rarely two; the CTAs of different n slices walk the m tiles in step and
// share each A tile through L2.  Warp 0: TMA producer over all tiles and K
// blocks; warp 1: MMA issuer, accumulating tile i into TMEM buffer i % 2;
// warps 2..9: epilogue, releasing the buffer as soon as its last TMEM read is
// done so the next tile's MMAs overlap this tile's stores.
// Request offsets of a cache projection carried by value (EPI_KV only):
// [in_off (n+1) | dst0 (n) | lengths (n)]; n_seg < 0: not carried.
struct KvParams {
  int n_seg;
  int v[3 * kKvParamReq + 1];
};
struct NoParams {
  int n_seg;
};
template <int EPI>
using ParamsFor = typename std::conditional<EPI == EPI_KV, KvParams, NoParams>::type;

template <int BN, int EPI, int NAP, bool BRES>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmO, const EpiArgs e,
                   const __grid_constant__ ParamsFor<EPI> kp) {
  using S = Shape<BN, EPI, NAP, BRES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S::STAGES * A_STAGE_BYTES;
  uint8_t* sBres = sB + S::STAGES * S::B_STAGE_BYTES;
  float* red = reinterpret_cast<float*>(sBres + S::BRES_BYTES);
  float* s_weff = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(red) + S::RED_BYTES);
  float* s_bias = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(s_weff) + S::WEFF_BYTES);
  int* s_seg = reinterpret_cast<int*>(s_bias + (BRES ? kStageNRes : kStageN));
  int* s_dst = s_seg + kStageSeg + 1;
  uint8_t* s_stage = reinterpret_cast<uint8_t*>(s_bias) + S::AUX_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(s_stage + S::STG_BYTES);
  uint64_t* empty = full + S::STAGES;
  uint64_t* acc_full = empty + S::STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* b_full = acc_empty + 2;     // resident B slice loaded
  uint64_t* b_empty = b_full + 1;       // last MMA reading the resident B slice done
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(b_empty + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tiles = e.N / BN;
  const int num_tiles = ((e.M + BM - 1) / BM) * n_tiles;
  const int num_kb = e.K / BK;
  const int m_tiles = (e.M + BM - 1) / BM;
  // this CTA's tiles: t_lo, t_lo + t_step, ... < t_hi
  int t_lo = blockIdx.x, t_hi = num_tiles, t_step = gridDim.x;
  if constexpr (BRES) {
    t_lo = static_cast<int>(static_cast<long long>(blockIdx.x) * num_tiles / gridDim.x);
    t_hi = static_cast<int>(static_cast<long long>(blockIdx.x + 1) * num_tiles / gridDim.x);
    t_step = 1;
  }
  auto tile_n = [&](int t) { return BRES ? t / m_tiles : t % n_tiles; };
  auto tile_m = [&](int t) { return BRES ? t % m_tiles : t / n_tiles; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full + b, 1);
      mbar_init(acc_empty + b, kEpiWarps);
    }
    mbar_init(b_full, 1);
    mbar_init(b_empty, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_holder, S::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  // the set-up above overlaps the previous kernel's tail; its outputs are read below
  pdl_launch_dependents();
  // The weights are not written by the kernels before this one: the
  // producer issues the weight part of its first k-blocks (or the resident
  // weight slice) before waiting, so that fetch overlaps the predecessor's
  // tail.  The activations (A) are loaded only after the wait.
  int n_pre = 0;                      // leading k-blocks whose weights are in flight
  if (warp == 0 && lane == 0 && t_lo < t_hi) {
    const int n0 = tile_n(t_lo) * BN;
    if constexpr (BRES) {
      mbar_expect_tx(b_full, BN * e.K * 2);
      for (int kb = 0; kb < num_kb; ++kb)
#pragma unroll
        for (int j = 0; j < BN; j += S::B_BOX)
          tma_load_2d(sBres + kb * (BN * BK * 2) + j * (BK * 2), &tmB, b_full, kb * BK, n0 + j);
    } else {
      n_pre = num_kb < S::STAGES ? num_kb : S::STAGES;
      for (int kb = 0; kb < n_pre; ++kb) {   // fresh ring: these stages are free
        mbar_expect_tx(full + kb, S::STAGE_BYTES);
#pragma unroll
        for (int j = 0; j < BN; j += S::B_BOX)
          tma_load_2d(sB + kb * S::B_STAGE_BYTES + j * (BK * 2), &tmB, full + kb, kb * BK, n0 + j);
      }
    }
  }
  pdl_wait();
  if constexpr (EPI == EPI_LN_HEAD) {
    for (int i = threadIdx.x; i < e.N * NAP; i += NUM_THREADS) {
      const int c = i / NAP, a = i - c * NAP;
      s_weff[i] = a < e.n_act ? e.weff_z[c * e.n_act + a] : 0.f;
    }
    __syncthreads();
  }
  // epilogue operands read by every tile: bias (and the cache-row remap) in
  // shared memory when they fit
  const float* bias = e.bias;
  const int* seg_off = e.seg_off;
  const int* dst_row0 = e.dst_row0;
  if constexpr (!S::LN) {
    if (e.N <= (BRES ? kStageNRes : kStageN)) {
      for (int i = threadIdx.x; i < e.N; i += NUM_THREADS) s_bias[i] = e.bias[i];
      bias = s_bias;
    }
    if constexpr (EPI == EPI_KV) {
      if (kp.n_seg >= 0) {
        // offsets carried by value: stage them, and CTA 0 publishes them
        // (with the new lengths) for the kernels that follow
        const int n = kp.n_seg;
        for (int i = threadIdx.x; i <= n; i += NUM_THREADS) s_seg[i] = kp.v[i];
        for (int i = threadIdx.x; i < n; i += NUM_THREADS) s_dst[i] = kp.v[n + 1 + i];
        if (blockIdx.x == 0) {
          for (int i = threadIdx.x; i < 2 * n + 1; i += NUM_THREADS) e.kv_dev_up[i] = kp.v[i];
          for (int i = threadIdx.x; i < n; i += NUM_THREADS) e.kv_dev_len[i] = kp.v[2 * n + 1 + i];
        }
        seg_off = s_seg;
        dst_row0 = s_dst;
      } else if (e.n_seg <= kStageSeg) {
        for (int i = threadIdx.x; i <= e.n_seg; i += NUM_THREADS) s_seg[i] = e.seg_off[i];
        for (int i = threadIdx.x; i < e.n_seg; i += NUM_THREADS) s_dst[i] = e.dst_row0[i];
        seg_off = s_seg;
        dst_row0 = s_dst;
      }
    }
    __syncthreads();
  }

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
      int it = 0;  // global k-block counter (ring position)
      int nb = 0, cur_n = -1;   // resident B slices loaded, current slice
      if (BRES && t_lo < t_hi) {   // the first slice was issued before the wait
        nb = 1;
        cur_n = tile_n(t_lo) * BN;
      }
      bool ok = true;
      for (int t = t_lo; t < t_hi && ok; t += t_step) {
        const int m0 = tile_m(t) * BM, n0 = tile_n(t) * BN;
        if constexpr (BRES) {
          if (n0 != cur_n) {
            if (nb > 0 && !mbar_wait(b_empty, (nb - 1) & 1, abort_flag)) break;
            mbar_expect_tx(b_full, BN * e.K * 2);
            for (int kb = 0; kb < num_kb; ++kb)
#pragma unroll
              for (int j = 0; j < BN; j += S::B_BOX)
                tma_load_2d(sBres + kb * (BN * BK * 2) + j * (BK * 2), &tmB, b_full, kb * BK, n0 + j);
            ++nb;
            cur_n = n0;
          }
        }
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % S::STAGES;
          const uint32_t ph = (it / S::STAGES) & 1;
          if (it < n_pre) {       // weights already in flight, bytes already expected
            tma_load_2d(sA + s * A_STAGE_BYTES, &tmA, full + s, kb * BK, m0);
            continue;
          }
          if (!mbar_wait(empty + s, ph ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          mbar_expect_tx(full + s, S::STAGE_BYTES);
          tma_load_2d(sA + s * A_STAGE_BYTES, &tmA, full + s, kb * BK, m0);
          if constexpr (!BRES) {
#pragma unroll
            for (int j = 0; j < BN; j += S::B_BOX)
              tma_load_2d(sB + s * S::B_STAGE_BYTES + j * (BK * 2), &tmB, full + s, kb * BK, n0 + j);
          }
        }
      }
      if (*abort_flag) {
        // let the copies already in flight land before shared memory is released
        for (int k = it > S::STAGES ? it - S::STAGES : 0; k < it; ++k)
          mbar_wait_plain(full + k % S::STAGES, (k / S::STAGES) & 1);
        if (BRES && nb > 0) mbar_wait_plain(b_full, (nb - 1) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, S::BN_MMA);
      int it = 0, i = 0;
      int nb = 0, cur_n = -1;
      bool ok = true;
      for (int t = t_lo; t < t_hi && ok; t += t_step, ++i) {
        const int nt = tile_n(t);
        if constexpr (BRES) {
          if (nt != cur_n) {
            if (!mbar_wait(b_full, nb & 1, abort_flag)) break;
            ++nb;
            cur_n = nt;
          }
        }
        const int buf = i % S::ACC_BUFS;
        const uint32_t use = i / S::ACC_BUFS;
        if (!mbar_wait(acc_empty + buf, (use & 1) ^ 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t dacc = tmem + buf * BN;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % S::STAGES;
          const uint32_t ph = (it / S::STAGES) & 1;
          if (!mbar_wait(full + s, ph, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t adesc = sdesc_sw128(smem_u32(sA + s * A_STAGE_BYTES));
          const uint64_t bdesc = BRES ? sdesc_sw128(smem_u32(sBres + kb * (BN * BK * 2)))
                                      : sdesc_sw128(smem_u32(sB + s * S::B_STAGE_BYTES));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
#pragma unroll
            for (int j = 0; j < BN / S::BN_MMA; ++j) {
              // 32 bytes along K per step inside the swizzle row; N halves are
              // S::BN_MMA rows (x 128 bytes) apart
              const uint64_t boff = static_cast<uint64_t>((j * S::BN_MMA * BK * 2) >> 4);
              mma_bf16(dacc + j * S::BN_MMA, adesc + 2 * k, bdesc + boff + 2 * k, idesc,
                       (kb > 0 || k > 0) ? 1u : 0u);
            }
          }
          mma_commit(empty + s);
        }
        mma_commit(acc_full + buf);   // also on abort: the epilogue waits on every issued MMA
        if constexpr (BRES) {
          // the resident slice is free once this tile's MMAs are done
          if (t + 1 >= t_hi || tile_n(t + 1) != nt) mma_commit(b_empty);
        }
      }
    }
  } else {
    const int ew = warp - 2;
    const int q = warp & 3;           // TMEM lane quarter this warp may access
    const int h = ew / 4;             // column half
    uint8_t* stage = s_stage + ew * 4096;
    int kchunk = 0;
    int i = 0;
    for (int t = t_lo; t < t_hi; t += t_step, ++i) {
      const int buf = i % S::ACC_BUFS;
      const uint32_t use = i / S::ACC_BUFS;
      // Go on exactly when the accumulator is complete: both warps of a lane
      // quarter see the same barrier phase, so they agree (they meet at named
      // barriers inside the LayerNorm epilogues).  Warp-uniform because
      // tcgen05.ld is .sync.aligned.
      bool go = mbar_wait(acc_full + buf, use & 1, abort_flag);
      go = __shfl_sync(0xffffffffu, go ? 1 : 0, 0) != 0;
      if (!go) break;
      tc_fence_after();
      const int m0 = tile_m(t) * BM, n0 = tile_n(t) * BN;
      epilogue<BN, EPI, NAP>(e, tmem + buf * BN + (static_cast<uint32_t>(q * 32) << 16), m0 + q * 32 + lane, n0,
                             h * (BN / 2), q, h, red, s_weff, bias, seg_off, dst_row0, &tmO, stage, kchunk);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty + buf);
    }
    if (lane == 0) bulk_wait_all();   // this warp's bulk stores are complete before exit
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, S::TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) latch_status(e.status, TXS_ERR_DEVICE_TIMEOUT);
}

// ------------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 tensor map over a row-major [rows, cols] matrix with leading
// dimension ld (elements), box {64 columns, box_rows rows}, 128-byte swizzle.
bool make_tmap(CUtensorMap* tm, const void* base, long long rows, long long cols, long long ld, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Output map for bulk stores: bf16 [rows, cols] with leading dimension ld,
// box {32 columns, 32 rows}, 64-byte swizzle.
bool make_tmap_out(CUtensorMap* tm, const void* base, long long rows, long long cols, long long ld) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(base) & 15) || (ld * 2) % 16) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Element-wise GELU of the epilogues, for tests: variant 0 is the bf16
// tensor-core epilogue's (gelu_erf_as2, on pairs), 1 the fp32 path's
// (gelu_erf).
__global__ void __launch_bounds__(256) gelu_eval_kernel(const float* __restrict__ x, float* __restrict__ y, long long n,
                                                        int variant) {
  for (long long i = (static_cast<long long>(blockIdx.x) * 256 + threadIdx.x) * 2; i < n;
       i += static_cast<long long>(gridDim.x) * 512) {
    const bool two = i + 1 < n;
    if (variant == 0) {
      const float2 r = gelu_erf_as2(make_float2(x[i], two ? x[i + 1] : 0.f));
      y[i] = r.x;
      if (two) y[i + 1] = r.y;
    } else {
      y[i] = gelu_erf(x[i]);
      if (two) y[i + 1] = gelu_erf(x[i + 1]);
    }
  }
}

cudaError_t launch_gelu_eval(const float* x, float* y, long long n, int variant, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const long long blocks = std::min<long long>((n + 511) / 512, 4096);
  gelu_eval_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(x, y, n, variant);
  return cudaGetLastError();
}

int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  }
  return n;
}

template <int BN, int EPI, int NAP = 4, bool BRES = false>
static cudaError_t launch_bn(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                             cudaStream_t s, int cls) {
  using Sh = Shape<BN, EPI, NAP, BRES>;
  if (BRES && e.K > Sh::KRES) return cudaErrorInvalidValue;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t err = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI, NAP, BRES>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, Sh::SMEM_BYTES);
    if (err != cudaSuccess) return err;
    attr_set = true;
  }
  CUtensorMap ta, tb, to;
  if (!make_tmap(&ta, A, e.M, e.K, lda, BM)) return cudaErrorInvalidValue;
  if (!make_tmap(&tb, B, e.N, e.K, e.K, Sh::B_BOX)) return cudaErrorInvalidValue;
  if (EPI == EPI_LN_HEAD) {
    to = ta;   // unused
  } else if (EPI == EPI_KV) {
    // the cache viewed as [(N / col_blk) * cap_total rows, col_blk] bf16
    const long long rows = static_cast<long long>(e.N / e.col_blk) * (e.col_blk_stride / e.col_blk);
    if (!make_tmap_out(&to, e.out, rows, e.col_blk, e.ldo)) return cudaErrorInvalidValue;
  } else {
    if (!make_tmap_out(&to, e.out, e.M, e.N, e.ldo)) return cudaErrorInvalidValue;
  }
  const long long tiles = static_cast<long long>((e.M + BM - 1) / BM) * (e.N / BN);
  const int grid = static_cast<int>(tiles < num_sms() ? tiles : num_sms());
  ParamsFor<EPI> kp;
  kp.n_seg = -1;
  if constexpr (EPI == EPI_KV) {
    if (e.kv_host_up && e.kv_host_len && e.n_seg <= kKvParamReq && e.n_seg <= kStageSeg) {
      const int n = e.n_seg;
      kp.n_seg = n;
      for (int i = 0; i < 2 * n + 1; ++i) kp.v[i] = e.kv_host_up[i];
      for (int i = 0; i < n; ++i) kp.v[2 * n + 1 + i] = e.kv_host_len[i];
    }
  }
  prof_begin(cls, s);
  cudaError_t err = launch_pdl(gemm_tc_kernel<BN, EPI, NAP, BRES>, dim3(grid), dim3(NUM_THREADS), Sh::SMEM_BYTES,
                               s, ta, tb, to, e, kp);
  prof_end(cls, s);
  return err;
}

bool tc_gemm_supported(int N, int K, int epi) {
  if (K <= 0 || K % BK != 0 || N <= 0) return false;
  if (epi == EPI_LN || epi == EPI_LN_HEAD) return N == 64 || N == 128 || N == 256 || N == 512;
  return N % 64 == 0;
}

template <int EPI>
static cudaError_t launch_plain(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                                cudaStream_t s, int cls) {
  // the widest tile that divides N (and the cache's column blocks) while there
  // are still at least as many tiles as SMs; narrower tiles otherwise
  const long long m_tiles = (e.M + BM - 1) / BM;
  auto fits = [&](int bn) {
    if (e.N % bn) return false;
    // cache column blocks: a tile covers whole blocks or lies inside one
    if (EPI == EPI_KV && e.col_blk % bn != 0 && (e.col_blk % 32 != 0 || bn % e.col_blk != 0)) return false;
    return true;
  };
  // short K and at least two tiles per SM: keep each CTA's B slice resident
  if (fits(256) && e.K <= Shape<256, EPI, 4, true>::KRES && m_tiles * (e.N / 256) >= 2 * num_sms())
    return launch_bn<256, EPI, 4, true>(A, lda, B, e, s, cls);
  if (fits(256) && m_tiles * (e.N / 256) >= num_sms()) return launch_bn<256, EPI>(A, lda, B, e, s, cls);
  if (fits(128)) return launch_bn<128, EPI>(A, lda, B, e, s, cls);
  if (fits(64)) return launch_bn<64, EPI>(A, lda, B, e, s, cls);
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_tc(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                           cudaStream_t s, int cls) {
  if (e.M == 0) return cudaSuccess;
  if (!tc_gemm_supported(e.N, e.K, e.epi)) return cudaErrorInvalidValue;
  if ((reinterpret_cast<uintptr_t>(A) & 15) || (reinterpret_cast<uintptr_t>(B) & 15) || (lda % 8))
    return cudaErrorInvalidValue;
  if (e.epi == EPI_LN_HEAD && (e.n_act < 1 || e.n_act > 16)) return cudaErrorInvalidValue;
  // rows of 256 or 512 columns: one 128-column slice per CTA of a cluster
  if (e.epi == EPI_LN || e.epi == EPI_LN_HEAD) {
    const cudaError_t r = launch_gemm_ln_cluster(A, lda, B, e, s, cls);
    if (r != cudaErrorNotSupported) return r;
  }
  switch (e.epi) {
    case EPI_LN:
      switch (e.N) {
        case 64: return launch_bn<64, EPI_LN>(A, lda, B, e, s, cls);
        case 128: return launch_bn<128, EPI_LN>(A, lda, B, e, s, cls);
        case 256: return launch_bn<256, EPI_LN>(A, lda, B, e, s, cls);
        default: return launch_bn<512, EPI_LN>(A, lda, B, e, s, cls);
      }
    case EPI_LN_HEAD:
      if (e.n_act <= 4) {
        switch (e.N) {
          case 64: return launch_bn<64, EPI_LN_HEAD, 4>(A, lda, B, e, s, cls);
          case 128: return launch_bn<128, EPI_LN_HEAD, 4>(A, lda, B, e, s, cls);
          case 256: return launch_bn<256, EPI_LN_HEAD, 4>(A, lda, B, e, s, cls);
          default: return launch_bn<512, EPI_LN_HEAD, 4>(A, lda, B, e, s, cls);
        }
      }
      switch (e.N) {
        case 64: return launch_bn<64, EPI_LN_HEAD, 16>(A, lda, B, e, s, cls);
        case 128: return launch_bn<128, EPI_LN_HEAD, 16>(A, lda, B, e, s, cls);
        case 256: return launch_bn<256, EPI_LN_HEAD, 16>(A, lda, B, e, s, cls);
        default: return launch_bn<512, EPI_LN_HEAD, 16>(A, lda, B, e, s, cls);
      }
    case EPI_BIAS: return launch_plain<EPI_BIAS>(A, lda, B, e, s, cls);
    case EPI_BIAS_GELU: return launch_plain<EPI_BIAS_GELU>(A, lda, B, e, s, cls);
    case EPI_KV: return launch_plain<EPI_KV>(A, lda, B, e, s, cls);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace tc

cudaError_t launch_gemm_tc(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                           cudaStream_t s, int cls) {
  return tc::launch_gemm_tc(A, lda, B, e, s, cls);
}
bool tc_gemm_supported(int N, int K, int epi) { return tc::tc_gemm_supported(N, K, epi); }
cudaError_t launch_gelu_eval(const float* x, float* y, long long n, int variant, cudaStream_t s) {
  return tc::launch_gelu_eval(x, y, n, variant, s);
}

}  // namespace txs
